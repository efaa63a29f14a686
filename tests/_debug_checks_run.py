"""Child process of tests/test_gpu_debug_checks.py: loads libace_debug.so
(ACE_LIB_VARIANT=debug) and runs small layers through it. Every forward must
leave a clean error word and intact canary words (ace_layer_sync) and still
pass replay parity; then a canary byte planted from the host must be
reported, naming the array."""
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path[:0] = [HERE, os.path.dirname(HERE)]

import numpy as np  # noqa: E402
import torch  # noqa: E402

import _replay as RP  # noqa: E402
import oracle as O  # noqa: E402
from paper_2609_05228_gb300 import ace, offline, synth  # noqa: E402


def dev(a, bf):
    a = np.ascontiguousarray(a)
    if bf:
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(a).cuda()


def host(t):
    if t.dtype == torch.bfloat16:
        return (t.view(torch.int16).cpu().numpy().view(np.uint16).astype(np.uint32) << 16).view(np.float32).astype(
            np.float64)
    return t.cpu().numpy().astype(np.float64)


def main():
    assert ace.LIBNAME == "libace_debug.so" and ace.ace_debug_checks_enabled(), "debug library not loaded"
    # the last spec (hidden 512, 24 experts) adds a second tensor-core shape at decode batch sizes
    specs = [synth.LayerSpec(256, 20, 4, 128, dtype="bf16"), synth.LayerSpec(256, 100, 8, 128, dtype="bf16"),
             synth.LayerSpec(256, 20, 4, 128, dtype="f32"), synth.LayerSpec(512, 24, 4, 256, dtype="bf16")]
    runs = 0
    for si, spec in enumerate(specs):
        w = synth.make_layer(spec, seed=11 + si)
        a_gsp, a_rcr = offline.tables(w)
        layer = ace.AceLayer(w, a_gsp, a_rcr, max_tokens=300)
        bf = spec.dtype == "bf16"
        for T in ((1, 3, 8, 9, 129) if spec.hidden == 512 else (1, 3, 17, 129, 300)):
            x = synth.make_tokens(spec, T, seed=T)
            xd = dev(x, bf)
            out = torch.empty_like(xd)
            for mode, val in (("ratio", 0.5), ("threshold", 0.3)):
                layer.forward(xd, out, T, mode, val)
                ace.ace_layer_sync(layer.handle)        # error word clean, canaries intact
                dec, z = RP.replay_decision(layer.handle, spec, a_gsp, a_rcr, T, mode, val)
                y_ref = O.moe_forward(x, w, decision=dec)
                RP.compare(host(out), y_ref, f32=not bf)
                runs += 1
        if si == 0:
            # a byte past one array's end, planted from the host, is caught and named
            ace.ace_debug_poke_canary(layer.handle, 3)
            try:
                ace.ace_layer_sync(layer.handle)
                raise AssertionError("overwritten canary not reported")
            except ace.AceError as e:
                assert e.status == 4 and "past the end of" in str(e), str(e)
        layer.close()
    print(f"debug checks clean: {runs} forwards")


if __name__ == "__main__":
    main()
