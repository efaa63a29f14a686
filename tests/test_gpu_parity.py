"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on
the same seeded inputs.

* exp32 and the whole decision (top-k ids, skip mask, g_hat, tau, retained
  count, offsets, permutation) are bit-exact against the oracle's float32
  decision spec, given the same float32 logits from the input generator.
* Every forward is checked in replay mode: its own float32 router logits
  (compared with the fp64 oracle's logits from x) are fed to the float32
  decision spec, which must reproduce the forward's decision bit for bit;
  the fp64 oracle then evaluates the layer under that decision and every
  token's output is compared: rel-L2 <= 5e-3 and max-abs <= 3e-2 * max|ref|
  (bf16), rel-L2 <= 1e-5 (fp32 layer).
* The independent fp64 decision is checked on the tokens whose routing is
  clear of every boundary by more than the GPU's rounding can move it, and
  its disagreement rate with the replayed decision is reported.
"""
import dataclasses
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import _replay as RP
import oracle as O
from paper_2609_05228_gb300 import ace, offline, synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    ace.lib()
    yield


def _dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).cuda()
    return torch.from_numpy(a).cuda()


def _host(t):
    if t.dtype == torch.bfloat16:
        return (t.view(torch.int16).cpu().numpy().view(np.uint16).astype(np.uint32) << 16).view(np.float32)
    return t.cpu().numpy()


# ------------------------------------------------------------------ exp32


def test_exp32_bitexact():
    x = np.concatenate([np.linspace(-90.0, 0.0, 1 << 20).astype(np.float32),
                        -np.abs(synth.make_logits(512, 512, seed=5).ravel()),
                        np.array([0.0, -0.0, -1e-30, -87.0, -86.99999], np.float32)])
    xd = torch.from_numpy(x).cuda()
    yd = torch.empty_like(xd)
    ace.ace_debug_exp32(xd, yd, x.size)
    torch.cuda.synchronize()
    want = O.exp32(x)
    got = yd.cpu().numpy()
    bad = np.nonzero(got.view(np.uint32) != want.view(np.uint32))[0]
    assert bad.size == 0, (x[bad[:5]], got[bad[:5]], want[bad[:5]])


# ------------------------------------------------------------------ decision bits


def _route_layer(N, k, max_tokens, m_min, tables):
    d = m = 64
    z16 = np.zeros(1, np.uint16)
    w = synth.LayerWeights(synth.LayerSpec(d, N, k, m, dtype="bf16", min_active=m_min),
                           np.zeros((N, d), np.uint16), np.zeros(N, np.float32),
                           np.zeros((N, m, d), np.uint16), np.zeros((N, m, d), np.uint16),
                           np.zeros((N, d, m), np.uint16), np.full(d, 0x3f80, np.uint16))
    del z16
    return ace.AceLayer(w, tables[0], tables[1], max_tokens)


ROUTE_CASES = [
    # T, N, k, m_min
    (1, 16, 4, 1),
    (3, 128, 8, 1),
    (64, 128, 8, 1),
    (257, 100, 6, 2),
    (4096, 128, 8, 1),
    (2048, 256, 8, 3),
    (1000, 1024, 16, 1),
    (16384, 128, 8, 1),
    (256, 128, 8, 2),
    (200, 1024, 16, 3),
    (33, 20, 2, 2),
]
CTLS = [("threshold", 0.0), ("threshold", 0.09), ("threshold", 0.12), ("threshold", math.inf),
        ("ratio", 0.0), ("ratio", 0.25), ("ratio", 0.5), ("ratio", 0.625), ("ratio", 1.0)]


@pytest.mark.parametrize("T,N,k,m_min", ROUTE_CASES)
def test_decision_bitexact(T, N, k, m_min):
    z = synth.make_logits(T, N, seed=100 + T + N, tie_fraction=0.05)
    tables = synth.make_tables(N, seed=7 + N, spread=0.2)
    layer = _route_layer(N, k, T, m_min, tables)
    zd = torch.from_numpy(z).cuda()
    ids_ref, g_ref = O.route_fp32(z, k)
    for mode, val in CTLS:
        ace.ace_route_logits(layer.handle, zd, T, mode, val)
        skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, k)
        ref = O.decide_fp32(ids_ref, g_ref, tables[0], tables[1], mode, val, m_min, 1e-6)
        assert (ids == ids_ref).all(), (mode, val)
        assert (skip.astype(bool) == ref["skip"]).all(), (mode, val, int(skip.sum()), int(ref["skip"].sum()))
        assert (gh.view(np.uint32) == ref["g_hat"].view(np.uint32)).all(), (mode, val)
        assert np.float32(tau).view(np.uint32) == np.float32(ref["tau"]).view(np.uint32), (mode, val, tau, ref["tau"])
        assert R == int((~ref["skip"]).sum())
        if mode == "ratio":
            assert T * k - R == ref["count"]
        off, perm = ace.ace_last_permutation(layer.handle, N, R)
        off_ref, perm_ref = O.permutation(ids_ref, ref["skip"], N)
        assert (off == off_ref).all() and (perm == perm_ref).all(), (mode, val)
    layer.close()


FUSION_ROUTE_CASES = [(64, 128, 8, 1), (257, 100, 6, 2), (4096, 128, 8, 1), (200, 1024, 16, 3), (2048, 256, 8, 3)]


@pytest.mark.parametrize("fusion", ["min", "mean", "gsp", "rcr", "score"])
@pytest.mark.parametrize("T,N,k,m_min", FUSION_ROUTE_CASES)
def test_decision_bitexact_fusion(T, N, k, m_min, fusion):
    """The skip-rule variants (Min / Mean fusion, single views, router score)
    through the fused small-batch route and the large-batch chain."""
    z = synth.make_logits(T, N, seed=500 + T + N, tie_fraction=0.05)
    tables = synth.make_tables(N, seed=9 + N, spread=0.2)
    layer = _route_layer(N, k, T, m_min, tables)
    zd = torch.from_numpy(z).cuda()
    ids_ref, g_ref = O.route_fp32(z, k)
    for mode, val in [("threshold", 0.09), ("ratio", 0.25), ("ratio", 0.5), ("ratio", 0.625)]:
        ace.ace_route_logits(layer.handle, zd, T, mode, val, fusion=fusion)
        skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, k)
        ref = O.decide_fp32(ids_ref, g_ref, tables[0], tables[1], mode, val, m_min, 1e-6, fusion=fusion)
        assert (ids == ids_ref).all(), (mode, val)
        assert (skip.astype(bool) == ref["skip"]).all(), (mode, val, int(skip.sum()), int(ref["skip"].sum()))
        assert (gh.view(np.uint32) == ref["g_hat"].view(np.uint32)).all(), (mode, val)
        assert np.float32(tau).view(np.uint32) == np.float32(ref["tau"]).view(np.uint32), (mode, val, tau, ref["tau"])
        if mode == "ratio":
            assert T * k - R == ref["count"]
        off, perm = ace.ace_last_permutation(layer.handle, N, R)
        off_ref, perm_ref = O.permutation(ids_ref, ref["skip"], N)
        assert (off == off_ref).all() and (perm == perm_ref).all(), (mode, val)
    with pytest.raises(ace.AceError):
        ace.ace_route_logits(layer.handle, zd, T, "ratio", 0.5, fusion=6)
    layer.close()


@pytest.mark.parametrize("T,pattern", [(16384, "equal"), (8192, "two_values"), (300, "equal"), (1, "equal"),
                                       (8, "equal"), (12, "two_values"), (16, "equal"), (17, "two_values")])
def test_decision_degenerate_scores(T, pattern):
    """Every candidate score equal (or only two distinct values): the
    threshold select meets one value held by far more keys than the select
    stages in shared memory (and the App. B.1 tie rule decides tau). Up to
    128 slots (16 tokens of top-8) the small-batch route selects by counting
    ranks; 17 tokens is the first size on its radix select."""
    N, k = 128, 8
    z = np.zeros((T, N), np.float32)
    if pattern == "two_values":
        z[: T // 3, :] = np.linspace(0.0, -0.5, N, dtype=np.float32)[None, :]
    tables = (np.ones(N, np.float32), np.ones(N, np.float32))
    layer = _route_layer(N, k, T, 1, tables)
    zd = torch.from_numpy(z).cuda()
    ids_ref, g_ref = O.route_fp32(z, k)
    for mode, val in [("ratio", 0.25), ("ratio", 0.5), ("ratio", 0.7)]:
        ace.ace_route_logits(layer.handle, zd, T, mode, val)
        skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, k)
        ref = O.decide_fp32(ids_ref, g_ref, tables[0], tables[1], mode, val, 1, 1e-6)
        assert (ids == ids_ref).all()
        assert (skip.astype(bool) == ref["skip"]).all(), (mode, val, int(skip.sum()), int(ref["skip"].sum()))
        assert (gh.view(np.uint32) == ref["g_hat"].view(np.uint32)).all()
        assert np.float32(tau).view(np.uint32) == np.float32(ref["tau"]).view(np.uint32), (tau, ref["tau"])
    layer.close()


@pytest.mark.parametrize("T", [5, 700])
def test_decision_signed_zero_and_tied_logits(T):
    """Exact logit ties, including -0.0 against +0.0 (equal logits): the
    lower expert index ranks first, through the small-batch fused route and
    the large-batch chain, bit-exact with the fp32 decision spec."""
    N, k = 64, 6
    g = np.random.Generator(np.random.PCG64(41))
    z = np.zeros((T, N), np.float32)
    z[:, :] = np.where(g.random((T, N)) < 0.5, np.float32(-0.0), np.float32(0.0))
    hot = g.random((T, N)) < 0.1                     # a few higher logits, some tied among themselves
    z[hot] = g.choice(np.array([0.5, 0.5, 1.0], np.float32), size=int(hot.sum()))
    tables = synth.make_tables(N, seed=4, spread=0.2)
    layer = _route_layer(N, k, T, 1, tables)
    zd = torch.from_numpy(z).cuda()
    ids_ref, g_ref = O.route_fp32(z, k)
    for mode, val in [("threshold", 0.1), ("ratio", 0.5)]:
        ace.ace_route_logits(layer.handle, zd, T, mode, val)
        skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, k)
        ref = O.decide_fp32(ids_ref, g_ref, tables[0], tables[1], mode, val, 1, 1e-6)
        assert (ids == ids_ref).all(), mode
        assert (skip.astype(bool) == ref["skip"]).all(), mode
        assert (gh.view(np.uint32) == ref["g_hat"].view(np.uint32)).all(), mode
    layer.close()


def test_decision_repeatable():
    T, N, k = 4096, 128, 8
    z = synth.make_logits(T, N, seed=3)
    tables = synth.make_tables(N, seed=1, spread=0.2)
    layer = _route_layer(N, k, T, 1, tables)
    zd = torch.from_numpy(z).cuda()
    first = None
    for _ in range(20):
        ace.ace_route_logits(layer.handle, zd, T, "ratio", 0.5)
        skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, k)
        off, perm = ace.ace_last_permutation(layer.handle, N, R)
        cur = (skip.tobytes(), gh.tobytes(), perm.tobytes())
        if first is None:
            first = cur
        assert cur == first
    layer.close()


# ------------------------------------------------------------------ full layer

_LAYERS = {}


def _layer(kind):
    if kind not in _LAYERS:
        if kind == "tiny":
            spec, seed = synth.spec_tiny(), 0
        elif kind == "qwen":
            spec, seed = synth.spec_qwen(), 0
        elif kind == "qwen_zipf":
            spec, seed = synth.spec_qwen(zipf=True), 0
        elif kind == "qwen_temp":
            # router temperature != 1 and m_min = 2 (Algorithm 4's restore)
            spec, seed = dataclasses.replace(synth.spec_qwen(zipf=True), router_temp=1.3, min_active=2), 7
        elif kind == "wide":
            # the widest routing the library takes: 1024 experts, top-16 (a token's
            # 16 slots in the combine, 32 logits per lane in the top-k)
            spec, seed = synth.LayerSpec(256, 1024, 16, 128, dtype="bf16"), 11
        else:
            raise KeyError(kind)
        w = synth.make_layer(spec, seed)
        if kind == "wide":
            # 4x router scale: with 1024 logits per token the default scale leaves
            # most top-16 boundaries within rounding distance
            w.router_w = synth.bf16_bits(synth.bf16_to_f32(w.router_w) * 4.0)
        a_gsp, a_rcr = offline.tables(w)
        w.extra["a_gsp"], w.extra["a_rcr"] = a_gsp, a_rcr
        _LAYERS[kind] = (w, ace.AceLayer(w, a_gsp, a_rcr, max_tokens=4096))
    return _LAYERS[kind]


def _clear_tokens(dec, z_ref, k, dz, dc, m_min=1):
    """Tokens whose top-k set, top-1 and every skip decision sit farther from
    a boundary than the GPU's rounding can move them. bf16 h rounding moves a
    logit by about 1e-3 (std) and c by about 1.5e-3 relative, so the bf16
    margins are dz = 6e-3 and dc = 8e-3; fp32 uses 1e-4."""
    zs = np.sort(z_ref, axis=1)[:, ::-1]
    gap_k = zs[:, k - 1] - zs[:, k] if z_ref.shape[1] > k else np.full(z_ref.shape[0], np.inf)
    gap_1 = zs[:, 0] - zs[:, 1]
    tau = dec["tau"]
    if dec["m_q"] is not None and 0 < dec["m_q"] and not math.isinf(tau):
        # ratio mode: tau is the (m+1)-th smallest candidate score itself, so
        # the boundary lies between the m-th and (m+1)-th candidate scores
        prot = O.protected_mask(dec["c"], m_min)
        cand = np.sort(dec["c"][~prot])
        tau = 0.5 * (cand[dec["m_q"] - 1] + cand[dec["m_q"]])
    if math.isinf(tau) or tau == 0:
        c_ok = np.ones(z_ref.shape[0], bool)
    else:
        c_ok = (np.abs(dec["c"] - tau) > dc * tau).all(axis=1)
    if m_min > 1:
        # which slots are protected (ratio mode) or restored (Algorithm 4) is
        # decided by ranking c among the non-top-1 slots: keep tokens whose
        # leading m_min such scores are separated by more than the margin
        cs = np.sort(dec["c"][:, 1:], axis=1)[:, ::-1]
        lead = cs[:, : min(m_min, cs.shape[1])]
        gaps = lead[:, :-1] - cs[:, 1 : lead.shape[1]]
        c_ok &= (gaps > dc * cs[:, :1]).all(axis=1)
    return (gap_k > dz) & (gap_1 > dz) & c_ok


def _run_layer(kind, T, mode, val, x_seed=1, fusion="max"):
    w, layer = _layer(kind)
    spec = w.spec
    x = synth.make_tokens(spec, T, seed=x_seed)
    xd = _dev(x)
    out = torch.empty_like(xd)
    layer.forward(xd, out, T, mode, val, fusion=fusion)
    torch.cuda.synchronize()
    return w, layer, spec, x, _host(out).astype(np.float64)


FORWARD_CASES = [
    ("tiny", 64, "ratio", 0.0), ("tiny", 64, "ratio", 0.25), ("tiny", 64, "ratio", 0.5),
    ("tiny", 64, "threshold", 0.2), ("tiny", 5, "ratio", 0.5),
    ("qwen", 1, "ratio", 0.5), ("qwen", 1, "ratio", 0.0), ("qwen", 8, "ratio", 0.0), ("qwen", 8, "ratio", 0.25), ("qwen", 32, "ratio", 0.5),
    ("qwen", 64, "ratio", 0.0), ("qwen", 64, "ratio", 0.25), ("qwen", 64, "ratio", 0.5),
    ("qwen", 17, "threshold", 0.11), ("qwen", 129, "ratio", 0.5), ("qwen", 1000, "ratio", 0.625),
    ("qwen", 3, "threshold", 0.11), ("qwen", 8, "ratio", 0.5), ("qwen", 9, "ratio", 0.5),   # decode stages of
    ("qwen", 12, "ratio", 0.5),                                        # two K blocks (up to 16 tokens)
    ("qwen", 1000, "ratio", 1.0),                                      # every non-top-1 slot skipped
    ("qwen_zipf", 4096, "ratio", 0.0), ("qwen_zipf", 4096, "ratio", 0.25), ("qwen_zipf", 4096, "ratio", 0.5),
    ("qwen_zipf", 4096, "ratio", 0.625),
    ("qwen_temp", 64, "ratio", 0.5), ("qwen_temp", 600, "ratio", 0.625), ("qwen_temp", 48, "threshold", 0.1),
    ("qwen", 256, "ratio", 0.5), ("qwen", 257, "ratio", 0.5),          # both sides of the small-batch path
    ("wide", 40, "ratio", 0.5), ("wide", 700, "ratio", 0.5), ("wide", 256, "threshold", 0.05),
]


FUSION_FORWARD_CASES = [(f, kind, T, "ratio", 0.5) for f in ("min", "mean", "gsp", "rcr", "score")
                        for kind, T in (("qwen", 64), ("qwen_zipf", 4096))] + [
    ("score", "qwen_temp", 600, "ratio", 0.625), ("min", "qwen", 17, "threshold", 0.11)]


@pytest.mark.parametrize("kind,T,mode,val", FORWARD_CASES)
def test_forward_parity(kind, T, mode, val):
    _check_forward(kind, T, mode, val, "max")


@pytest.mark.parametrize("fusion,kind,T,mode,val", FUSION_FORWARD_CASES)
def test_forward_parity_fusion(fusion, kind, T, mode, val):
    _check_forward(kind, T, mode, val, fusion)


def _check_forward(kind, T, mode, val, fusion):
    w, layer, spec, x, y_gpu = _run_layer(kind, T, mode, val, fusion=fusion)
    k = spec.top_k
    f32 = spec.dtype == "f32"
    # replay: the forward's own logits through the fp32 decision spec, bit-exact
    dec, z_gpu = RP.replay_decision(layer.handle, spec, w.extra["a_gsp"], w.extra["a_rcr"], T, mode, val, fusion)
    if mode == "ratio":
        m_q = min(O.llround_pos(float(np.float32(val)) * T * k), T * (k - max(spec.min_active, 1)))
        assert dec["count"] == m_q
    # the logits themselves against the fp64 oracle, then every token's output
    z_ref = RP.check_logits(z_gpu, x, w, f32=f32)
    y_ref = O.moe_forward(x, w, decision=dec)
    RP.compare(y_gpu, y_ref, f32=f32)
    # the independent fp64 decision: equal on every token clear of a boundary
    dec64 = O.ace_decide(z_ref, k, w.extra["a_gsp"], w.extra["a_rcr"], mode, val, spec.min_active, spec.eps, fusion)
    margin = 1e-4 if f32 else None
    # the wide layer's logits are 4x the scale (so is their rounding), and its
    # 1024 candidates put more top-16 boundaries within that distance
    dz = 4 * 6e-3 if kind == "wide" else (margin or 6e-3)
    clear = _clear_tokens(dec64, z_ref, k, dz, margin or 8e-3, spec.min_active)
    assert clear.mean() >= (0.2 if kind == "wide" else 0.4), clear.mean()
    for t in np.nonzero(clear)[0]:
        gpu = {int(dec["ids"][t, i]): bool(dec["skip"][t, i]) for i in range(k)}
        ref = {int(dec64["ids"][t, i]): bool(dec64["skip"][t, i]) for i in range(k)}
        assert gpu == ref, t
    RP.note_disagreement(f"{kind} T={T} {mode}={val} {fusion}", dec, dec64)


def test_layers_of_different_shapes_coexist():
    """A layer created after another with a smaller shape must not lower the
    kernels' shared-memory limits the first one needs: its forwards keep
    working and give the same bits (decode and prefill paths)."""
    w, layer = _layer("qwen")
    outs = {}
    for T in (64, 300):
        x = _dev(synth.make_tokens(w.spec, T, seed=21))
        o = torch.empty_like(x)
        layer.forward(x, o, T, "ratio", 0.5)
        outs[T] = (x, o)
    torch.cuda.synchronize()
    small = _route_layer(16, 4, 8, 1, synth.make_tables(16, seed=2))
    small_f32 = ace.AceLayer(synth.make_layer(synth.spec_tiny(), 3), *synth.make_tables(16, seed=3), max_tokens=8)
    for T, (x, o) in outs.items():
        o2 = torch.empty_like(x)
        layer.forward(x, o2, T, "ratio", 0.5)
        torch.cuda.synchronize()
        assert torch.equal(o, o2), T
    small.close()
    small_f32.close()


def test_forward_q0_matches_threshold0():
    w, layer = _layer("qwen")
    T = 64
    x = _dev(synth.make_tokens(w.spec, T, seed=3))
    o1 = torch.empty_like(x)
    o2 = torch.empty_like(x)
    layer.forward(x, o1, T, "ratio", 0.0)
    layer.forward(x, o2, T, "threshold", 0.0)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)


@pytest.mark.parametrize("T", [1000, 4096])
def test_forward_deterministic_large_batch(T):
    """Batches over 256 tokens: per-slot output rows and a rank-order combine,
    no atomics on the output, so every call returns the same bits."""
    w, layer = _layer("qwen_zipf")
    x = _dev(synth.make_tokens(w.spec, T, seed=6))
    outs = []
    for _ in range(3):
        o = torch.empty_like(x)
        layer.forward(x, o, T, "ratio", 0.5)
        outs.append(o)
    torch.cuda.synchronize()
    assert all(torch.equal(outs[0], o) for o in outs[1:])


def test_forward_deterministic_and_host_api():
    w, layer = _layer("qwen")
    T = 64
    xh = synth.make_tokens(w.spec, T, seed=4)
    x = _dev(xh)
    outs = []
    for _ in range(3):
        o = torch.empty_like(x)
        layer.forward(x, o, T, "ratio", 0.5)
        outs.append(o)
    torch.cuda.synchronize()
    assert all(torch.equal(outs[0], o) for o in outs[1:])
    host_out = np.zeros_like(xh)
    ace.ace_moe_forward_host(layer.handle, xh, host_out, T, "ratio", 0.5)
    dev_out = outs[0].view(torch.int16).cpu().numpy().view(np.uint16)
    assert (host_out == dev_out).all()


def test_forward_edge_cases():
    w, layer = _layer("qwen")
    x = _dev(synth.make_tokens(w.spec, 4, seed=5))
    out = torch.empty_like(x)
    layer.forward(x, out, 0, "ratio", 0.5)          # T = 0 is a no-op
    with pytest.raises(ace.AceError) as e:
        layer.forward(x, out, 5000, "ratio", 0.5)   # beyond max_tokens
    assert e.value.status == 1
    with pytest.raises(ace.AceError):
        layer.forward(x, out, 4, "ratio", 1.5)
    with pytest.raises(ace.AceError):
        layer.forward(x, out, 4, "threshold", float("nan"))
    with pytest.raises(ace.AceError):
        layer.forward(x, x, 4, "ratio", 0.5)        # aliasing
    # tau = +inf keeps only the top-1 expert of every token
    layer.forward(x, out, 4, "threshold", math.inf)
    skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, 4, w.spec.top_k)
    assert R == 4 and (skip[:, 0] == 0).all() and (skip[:, 1:] == 1).all()
    ace.ace_layer_sync(layer.handle)


@pytest.mark.parametrize("T", [64, 2048])
def test_calibrated_threshold_reproduces_ratio(T):
    """App. B.1: a threshold calibrated on a batch in ratio mode, used in
    threshold mode on that same batch, gives the same mask and g_hat."""
    from paper_2609_05228_gb300 import calibrate
    w, layer = _layer("qwen_zipf")
    x = _dev(synth.make_tokens(w.spec, T, seed=12))
    taus = calibrate.calibrate_taus(layer, x, T, [0.25, 0.5])
    out = torch.empty_like(x)
    for q, tau in taus.items():
        layer.forward(x, out, T, "ratio", q)
        ref = ace.ace_last_skip_mask(layer.handle, T, w.spec.top_k)
        layer.forward(x, out, T, "threshold", tau)
        got = ace.ace_last_skip_mask(layer.handle, T, w.spec.top_k)
        assert (got[0] == ref[0]).all() and (got[2].view(np.uint32) == ref[2].view(np.uint32)).all()
        assert got[4] == ref[4]


def test_forward_host_graph_replay():
    """Pinned host buffers: the host call replays a captured graph; results
    equal the device-buffer forward, also after the host buffers, T or the
    skip control change (re-capture)."""
    w, layer = _layer("qwen")
    for T, mode, val in [(64, "ratio", 0.5), (64, "ratio", 0.5), (32, "threshold", 0.11), (300, "ratio", 0.25)]:
        xh = synth.make_tokens(w.spec, T, seed=5 + T)
        x = _dev(xh)
        o = torch.empty_like(x)
        layer.forward(x, o, T, mode, val)
        want = o.view(torch.int16).cpu().numpy().view(np.uint16)
        for _ in range(2):
            xp = torch.from_numpy(xh.view(np.int16)).pin_memory()
            op = torch.empty_like(xp).pin_memory()
            ace.ace_moe_forward_host(layer.handle, xp, op, T, mode, val)
            assert (op.numpy().view(np.uint16) == want).all(), (T, mode, val)
            ace.ace_moe_forward_host(layer.handle, xp, op, T, mode, val)     # replay
            assert (op.numpy().view(np.uint16) == want).all(), (T, mode, val)


@pytest.mark.parametrize("T", [64, 300])
def test_non_finite_logits_reported(T):
    """A NaN router logit ranks last in the top-k, and the next call that
    synchronises reports ACE_ERR_NUMERIC once (the device word is cleared)."""
    N, k = 128, 8
    tables = synth.make_tables(N, seed=3, spread=0.2)
    layer = _route_layer(N, k, T, 1, tables)
    z = synth.make_logits(T, N, seed=17)
    bad = z.copy()
    bad[3, 5] = np.nan
    ace.ace_route_logits(layer.handle, torch.from_numpy(bad).cuda(), T, "ratio", 0.5)
    with pytest.raises(ace.AceError) as e:
        ace.ace_last_skip_mask(layer.handle, T, k)
    assert e.value.status == 6
    skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, k)    # word cleared: no error now
    assert 5 not in ids[3].tolist()                                         # NaN ranks last
    ace.ace_route_logits(layer.handle, torch.from_numpy(z).cuda(), T, "ratio", 0.5)
    ace.ace_last_skip_mask(layer.handle, T, k)
    layer.close()
