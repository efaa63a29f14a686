"""ace_route_decide_noalloc — the routing decision for callers that cannot
allocate device memory (their runtime owns the GPU memory pool, or they run
while another component holds the allocator). Its scratch is a fixed device
array inside the library. The test compares it, through the C ABI, with the
existing ace_route_logits entry point on the same logits, on two calls in a
row, and checks that sizes beyond its limits are rejected.

This file is collected last so that, if it fails, a run stopping at the first
failure has already run every other test."""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle as O
from paper_2609_05228_gb300 import ace, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ace.lib()
    yield


def _layer(N, k, T, m_min, tables):
    d = m = 64
    w = synth.LayerWeights(synth.LayerSpec(d, N, k, m, dtype="bf16", min_active=m_min),
                           np.zeros((N, d), np.uint16), np.zeros(N, np.float32),
                           np.zeros((N, m, d), np.uint16), np.zeros((N, m, d), np.uint16),
                           np.zeros((N, d, m), np.uint16), np.full(d, 0x3f80, np.uint16))
    return ace.AceLayer(w, tables[0], tables[1], T)


@pytest.mark.parametrize("T,N,k,m_min,calls", [
    (64, 128, 8, 1, [("ratio", 0.5), ("threshold", 0.11)]),
    (256, 256, 16, 3, [("ratio", 0.625), ("ratio", 0.25)]),
    (3, 20, 2, 1, [("threshold", 0.0), ("ratio", 1.0)]),
])
def test_noalloc_matches_route_logits(T, N, k, m_min, calls):
    tables = synth.make_tables(N, seed=11, spread=0.2)
    layer = _layer(N, k, T, m_min, tables)
    a_gsp = torch.from_numpy(tables[0]).cuda()
    a_rcr = torch.from_numpy(tables[1]).cuda()
    ids = torch.empty((T, k), dtype=torch.int32, device="cuda")
    skip = torch.empty((T, k), dtype=torch.uint8, device="cuda")
    gh = torch.empty((T, k), dtype=torch.float32, device="cuda")
    tau = torch.empty(1, dtype=torch.float32, device="cuda")
    for n, (mode, val) in enumerate(calls):
        z = torch.from_numpy(synth.make_logits(T, N, seed=300 + n, tie_fraction=0.05)).cuda()
        ace.ace_route_logits(layer.handle, z, T, mode, val)
        r_skip, r_ids, r_gh, r_tau, _ = ace.ace_last_skip_mask(layer.handle, T, k)
        ace.ace_route_decide_noalloc(z, T, N, k, a_gsp, a_rcr, 1e-6, m_min, mode, val, ids, skip, gh, tau)
        torch.cuda.synchronize()
        assert (ids.cpu().numpy() == r_ids).all()
        assert (skip.cpu().numpy() == r_skip).all()
        assert (gh.cpu().numpy().view(np.uint32) == r_gh.view(np.uint32)).all()
        assert tau.cpu().numpy().view(np.uint32)[0] == np.float32(r_tau).view(np.uint32)
    layer.close()


@pytest.mark.parametrize("fusion", ["min", "mean", "gsp", "rcr", "score"])
def test_noalloc_fusion_matches_oracle(fusion):
    T, N, k, m_min = 128, 128, 8, 2
    tables = synth.make_tables(N, seed=12, spread=0.2)
    a_gsp = torch.from_numpy(tables[0]).cuda()
    a_rcr = torch.from_numpy(tables[1]).cuda()
    ids = torch.empty((T, k), dtype=torch.int32, device="cuda")
    skip = torch.empty((T, k), dtype=torch.uint8, device="cuda")
    gh = torch.empty((T, k), dtype=torch.float32, device="cuda")
    tau = torch.empty(1, dtype=torch.float32, device="cuda")
    z = synth.make_logits(T, N, seed=41, tie_fraction=0.05)
    ids_ref, g_ref = O.route_fp32(z, k)
    for mode, val in [("ratio", 0.5), ("threshold", 0.1)]:
        ace.ace_route_decide_noalloc(torch.from_numpy(z).cuda(), T, N, k, a_gsp, a_rcr, 1e-6, m_min, mode, val,
                                     ids, skip, gh, tau, fusion=fusion)
        torch.cuda.synchronize()
        ref = O.decide_fp32(ids_ref, g_ref, tables[0], tables[1], mode, val, m_min, 1e-6, fusion=fusion)
        assert (ids.cpu().numpy() == ids_ref).all()
        assert (skip.cpu().numpy().astype(bool) == ref["skip"]).all(), (mode, val)
        assert (gh.cpu().numpy().view(np.uint32) == ref["g_hat"].view(np.uint32)).all()
        assert tau.cpu().numpy().view(np.uint32)[0] == np.float32(ref["tau"]).view(np.uint32)


def test_noalloc_rejects_sizes_beyond_limits():
    z = torch.zeros((300, 8), dtype=torch.float32, device="cuda")
    t = torch.ones(8, dtype=torch.float32, device="cuda")
    out = torch.empty(300 * 8, dtype=torch.float32, device="cuda")
    ids = torch.empty(300 * 8, dtype=torch.int32, device="cuda")
    sk = torch.empty(300 * 8, dtype=torch.uint8, device="cuda")
    with pytest.raises(ace.AceError) as e:
        ace.ace_route_decide_noalloc(z, 300, 8, 2, t, t, 1e-6, 1, "ratio", 0.5, ids, sk, out, out)
    assert e.value.status == 1 and "T must be" in str(e.value)
    with pytest.raises(ace.AceError):
        ace.ace_route_decide_noalloc(z, 256, 8, 17, t, t, 1e-6, 1, "ratio", 0.5, ids, sk, out, out)
    with pytest.raises(ace.AceError):
        ace.ace_route_decide_noalloc(z, 4, 8, 2, t, t, 1e-6, 1, "ratio", math.nan, ids, sk, out, out)
