"""GPU offline tables (ace_offline_tables_device) against the oracle's direct
fp64 products of Algorithms 2 and 3, and against the host library on a
full-size layer.

The small layers are built so that a mistake in any one factor moves the
normalised tables: per-expert, per-column and per-K-index weight scales, a
strongly non-uniform gamma (so Gamma applied as gamma instead of gamma^2, or
to the wrong index, changes the experts' ratios) and a large offset shared by
all router rows (so a missing centring changes the RCR prototypes)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle as O
from paper_2609_05228_gb300 import ace, offline, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def _hetero_layer(seed, d=256, n=16, m=128):
    g = np.random.Generator(np.random.PCG64(seed))

    def logu(lo, hi, shape):
        return np.exp(g.uniform(np.log(lo), np.log(hi), shape))

    w_gate = g.standard_normal((n, m, d)) * 0.02 * logu(0.25, 4, (n, 1, d))
    w_up = g.standard_normal((n, m, d)) * 0.02 * logu(0.25, 4, (n, 1, d))
    w_down = g.standard_normal((n, d, m)) * 0.02 * logu(0.5, 2, (n, 1, 1)) * logu(0.25, 4, (n, 1, m))
    router = g.standard_normal((n, d)) * 0.02 * logu(0.5, 2, (n, 1)) + 0.05 * g.standard_normal(d)[None, :]
    gamma = logu(0.2, 5, d)
    spec = synth.LayerSpec(d, n, 2, m, dtype="bf16")
    b = synth.bf16_bits
    return synth.LayerWeights(spec, b(router), np.zeros(n, np.float32), b(w_gate), b(w_up), b(w_down), b(gamma),
                              seed)


@pytest.mark.parametrize("seed", [0, 1])
def test_tables_device_match_oracle(seed):
    w = _hetero_layer(seed)
    a_ref = O.gsp_table(w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6)
    assert a_ref.max() / a_ref.min() > 2.0          # the experts really differ
    for apply_gamma in (False, True):
        a, r = offline.tables_device(w, 1e-6, apply_gamma)
        r_ref = O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, 1e-6, apply_gamma=apply_gamma)
        np.testing.assert_allclose(a, a_ref, rtol=2e-5)
        np.testing.assert_allclose(r, r_ref, rtol=2e-5)


def test_tables_device_chunking_and_repeatability():
    """Experts processed in chunks (ragged last chunk, one expert at a time)
    give the same bits as one chunk, and repeated calls give the same bits."""
    w = _hetero_layer(5, d=256, n=16, m=192)
    per_expert = 3 * 256 * 192 * 2
    ref = offline.tables_device(w)
    for budget in (per_expert * 3, per_expert * 5 + 7, 1):
        out = offline.tables_device(w, tile_budget=budget)
        assert out[0].tobytes() == ref[0].tobytes() and out[1].tobytes() == ref[1].tobytes(), budget
    again = offline.tables_device(w)
    assert again[0].tobytes() == ref[0].tobytes() and again[1].tobytes() == ref[1].tobytes()


def test_tables_device_match_host_library_full_size():
    """The d=2048, N=128, m=768 layer of the decode and prefill benchmarks:
    GPU tables against the host library's fp64 Gram route."""
    w = synth.make_layer(synth.spec_qwen(), 0)
    a_h, r_h = offline.tables(w)
    a_g, r_g = offline.tables_device(w)
    np.testing.assert_allclose(a_g, a_h, rtol=3e-5)
    np.testing.assert_allclose(r_g, r_h, rtol=3e-5)


def test_tables_device_argument_errors():
    z = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ace.AceError) as ei:
        ace.ace_offline_tables_device(100, 4, 64, z, z, z, z, z)      # d not a multiple of 256
    assert ei.value.status == 2
    with pytest.raises(ace.AceError) as ei:
        ace.ace_offline_tables_device(256, 4, 64, z, None, z, z, z)
    assert ei.value.status == 1
