"""The C-ABI library loads without a GPU and exports every symbol that
include/ace.h declares; argument checks that need no device run too."""
import ctypes
import os
import re

import pytest

from paper_2609_05228_gb300 import ace, build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "ace.h")


@pytest.fixture(scope="module")
def libace():
    if not os.path.exists(ace.LIBPATH):
        build.build()
    return ctypes.CDLL(ace.LIBPATH)


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ace_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ["ace_layer_create", "ace_moe_forward", "ace_last_skip_mask", "ace_layer_destroy",
                     "ace_route_logits", "ace_moe_forward_host", "ace_last_permutation",
                     "ace_last_router_logits", "ace_status_string", "ace_last_error_message"]:
        assert required in names


def test_library_exports_every_declared_symbol(libace):
    missing = [n for n in declared_functions() if not hasattr(libace, n)]
    assert not missing, missing


def test_host_side_argument_checks(libace):
    ace._lib = None
    L = ace.lib()
    assert L.ace_status_string(0) == b"ACE_OK"
    assert L.ace_status_string(5) == b"ACE_ERR_TIMEOUT"
    # NULL descriptor / bad sizes are rejected before any device call
    out = ctypes.c_void_p()
    st = L.ace_layer_create(None, None, None, None, None, None, None, None, None, None, ctypes.byref(out))
    assert st == 1
    d = ace.ace_layer_desc(64, 8, 9, 64, 16, ace.ACE_BF16, 1e-6, 1e-6, 1.0, 1, 0)   # k > N
    st = L.ace_layer_create(ctypes.byref(d), 1, None, 1, 1, 1, 1, 1, 1, None, ctypes.byref(out))
    assert st == 1 and b"top_k" in L.ace_last_error_message()
    d = ace.ace_layer_desc(100, 8, 2, 64, 16, ace.ACE_BF16, 1e-6, 1e-6, 1.0, 1, 0)  # d % 64
    st = L.ace_layer_create(ctypes.byref(d), 1, None, 1, 1, 1, 1, 1, 1, None, ctypes.byref(out))
    assert st == 2
    assert L.ace_moe_forward(None, None, None, 1, ace.ace_skip_ctl(0, 0.1), None) == 1
    assert L.ace_last_skip_mask(None, None, None, None, None, None) == 1


def test_struct_layouts_match_header(tmp_path):
    """The binding's ctypes structs have the sizes and field offsets that a C
    compiler gives the header's structs."""
    src = tmp_path / "layout.c"
    src.write_text(
        '#include <stdio.h>\n#include <stddef.h>\n#include "ace.h"\n'
        "int main(void) {\n"
        '  printf("%zu %zu %zu %zu\\n", sizeof(ace_skip_ctl), offsetof(ace_skip_ctl, value),'
        " offsetof(ace_skip_ctl, fusion), sizeof(ace_layer_desc));\n"
        '  printf("%zu %zu\\n", offsetof(ace_layer_desc, eps), offsetof(ace_layer_desc, add_residual));\n'
        "  return 0;\n}\n")
    exe = tmp_path / "layout"
    import subprocess
    subprocess.run(["gcc", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()
    got = [int(v) for v in out]
    want = [ctypes.sizeof(ace.ace_skip_ctl), ace.ace_skip_ctl.value.offset, ace.ace_skip_ctl.fusion.offset,
            ctypes.sizeof(ace.ace_layer_desc), ace.ace_layer_desc.eps.offset, ace.ace_layer_desc.add_residual.offset]
    assert got == want


def test_unknown_fusion_rejected_on_host(libace):
    ace._lib = None
    L = ace.lib()
    bad = ace.ace_skip_ctl(ace.ACE_SKIP_RATIO, 0.5, 6)
    fake = ctypes.c_void_p(16)
    st = L.ace_route_decide_noalloc(fake, 4, 8, 2, fake, fake, ctypes.c_float(1e-6), 1, bad, fake, fake, fake,
                                    fake, None)
    assert st == 1 and b"fusion" in L.ace_last_error_message()
    with pytest.raises(ValueError):
        ace._ctl("ratio", 0.5, "median")
    assert ace._ctl("ratio", 0.5, "score").fusion == ace.ACE_FUSION_SCORE


def test_stack_argument_checks_on_host(libace):
    ace._lib = None
    L = ace.lib()
    out = ctypes.c_void_p(7)
    assert L.ace_stack_create(None, 2, ctypes.byref(out)) == 1 and out.value is None
    arr = (ctypes.c_void_p * 1)(None)
    assert L.ace_stack_create(arr, 1, ctypes.byref(out)) == 1
    assert L.ace_stack_forward(None, None, None, 1, ace.ace_skip_ctl(0, 0.1, 0), None) == 1
    L.ace_stack_destroy(None)


def test_debug_library_exports_the_same_boundary():
    """libace_debug.so (index guards, canary words) exports every declared
    symbol too; the two builds report which one they are, and the canary hook
    rejects a NULL layer before touching a device."""
    if not os.path.exists(build.DEBUG_LIBPATH):
        build.build()
    dbg = ctypes.CDLL(build.DEBUG_LIBPATH)
    rel = ctypes.CDLL(ace.LIBPATH)
    missing = [n for n in declared_functions() if not hasattr(dbg, n)]
    assert not missing, missing
    assert dbg.ace_debug_checks_enabled() == 1
    assert rel.ace_debug_checks_enabled() == 0
    dbg.ace_debug_poke_canary.argtypes = [ctypes.c_void_p, ctypes.c_int]
    assert dbg.ace_debug_poke_canary(None, 0) == 1          # ACE_ERR_INVALID_ARG
