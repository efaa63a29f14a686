"""The product's offline GSP/RCR tool (Gram route) against the oracle's
direct products of Algorithms 2 and 3."""
import numpy as np

import oracle as O
from paper_2609_05228_gb300 import offline, synth


def _layer(seed, d=48, n=7, m=20):
    g = np.random.Generator(np.random.PCG64(seed))
    spec = synth.LayerSpec(d, n, 2, m, dtype="f32")
    return synth.LayerWeights(spec, (g.standard_normal((n, d)) * 0.3).astype(np.float32), np.zeros(n, np.float32),
                              (g.standard_normal((n, m, d)) * 0.3).astype(np.float32),
                              (g.standard_normal((n, m, d)) * 0.3).astype(np.float32),
                              (g.standard_normal((n, d, m)) * 0.3).astype(np.float32),
                              (1 + g.uniform(-0.2, 0.2, d)).astype(np.float32))


def test_offline_tables_match_oracle():
    for seed in range(3):
        w = _layer(seed)
        a, r = offline.tables(w)
        a_ref = O.gsp_table(w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6)
        r_ref = O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6)
        np.testing.assert_allclose(a, a_ref, rtol=2e-6)
        np.testing.assert_allclose(r, r_ref, rtol=2e-6)
        _, r2 = offline.tables(w, apply_gamma=True)
        r2_ref = O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6, apply_gamma=True)
        np.testing.assert_allclose(r2, r2_ref, rtol=2e-6)


def test_offline_tables_bf16_layer():
    w = synth.make_layer(synth.LayerSpec(128, 6, 2, 64, dtype="bf16"), seed=3)
    a, r = offline.tables(w)
    np.testing.assert_allclose(a, O.gsp_table(w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6), rtol=2e-6)
    np.testing.assert_allclose(r, O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6), rtol=2e-6)


def test_offline_tables_thread_count_does_not_change_bits():
    w = _layer(11, d=64, n=9, m=24)
    a1, r1 = offline.ace_offline_tables(w.gamma, w.router_w, w.w_gate, w.w_up, w.w_down, 1e-6, n_threads=1)
    a4, r4 = offline.ace_offline_tables(w.gamma, w.router_w, w.w_gate, w.w_up, w.w_down, 1e-6, n_threads=4)
    assert a1.tobytes() == a4.tobytes() and r1.tobytes() == r4.tobytes()


def test_offline_library_boundary():
    """libace_offline.so exports what include/ace_offline.h declares and
    rejects bad arguments without writing."""
    import ctypes
    import os
    import re
    hdr = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "ace_offline.h")
    text = re.sub(r"/\*.*?\*/", "", open(hdr).read(), flags=re.S)
    names = sorted(set(re.findall(r"\b(ace_[a-z0-9_]+)\s*\(", text)))
    L = offline.lib()
    assert names == ["ace_offline_tables"] and all(hasattr(L, n) for n in names)
    out = np.full(4, 7.0, np.float32)
    z = np.zeros(16, np.float32)
    st = L.ace_offline_tables(0, 4, 4, 1, z.ctypes.data, z.ctypes.data, z.ctypes.data, z.ctypes.data,
                              z.ctypes.data, ctypes.c_double(1e-6), 0, 1, out.ctypes.data, out.ctypes.data)
    assert st == 1 and (out == 7.0).all()
    st = L.ace_offline_tables(4, 4, 4, 1, None, z.ctypes.data, z.ctypes.data, z.ctypes.data,
                              z.ctypes.data, ctypes.c_double(1e-6), 0, 1, out.ctypes.data, out.ctypes.data)
    assert st == 1 and (out == 7.0).all()
