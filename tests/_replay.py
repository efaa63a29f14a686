"""Replay-mode parity helpers (the oracle's mode (ii)).

After a GPU forward, the layer's own float32 router logits are read back and
handed to the oracle's float32 decision spec (top-k with ties to the lower
expert index, Algorithm 4, the App. B.1 threshold, the permutation). That
decision must equal the GPU's bit for bit. The oracle then evaluates the
experts in fp64 under that same decision, so every token's output can be
compared with the bf16 tolerance: no token is left out for sitting near a
decision boundary.

Replaying the GPU's logits would hide a wrong router, so the logits are also
compared with the fp64 oracle's own (from x), with the output tolerance.
The independent fp64 decision (mode (i)) is only counted: its disagreement
rate with the replayed decision is collected in DISAGREEMENT and printed at
the end of the session (tests/conftest.py).
"""
import numpy as np

import oracle as O
from paper_2609_05228_gb300 import ace

# Layer outputs, bf16 weights and activations: relative L2 and max-abs
# (relative to max |ref|), the stated tolerance of the method's outputs.
RTOL_L2 = 5e-3
RTOL_MAX = 3e-2
# fp32 layers: inputs, weights and every intermediate in float32, fp32
# accumulation over d = 256 and m = 128 terms.
RTOL_L2_F32 = 1e-5

DISAGREEMENT = []


def replay_decision(handle, spec, a_gsp, a_rcr, T, mode, val, fusion="max"):
    """Assert the GPU decision of the last forward on `handle` equals the
    oracle's float32 decision spec on the forward's own logits, bit for bit:
    ids, skip mask, g_hat, tau, the realised count and the permutation.
    Returns (decision dict of the oracle, the GPU logits)."""
    N, k = spec.n_experts, spec.top_k
    z = ace.ace_last_router_logits(handle, T, N)
    skip, ids, gh, tau, R = ace.ace_last_skip_mask(handle, T, k)
    ids_ref, g_ref = O.route_fp32(z, k)
    ref = O.decide_fp32(ids_ref, g_ref, a_gsp, a_rcr, mode, val, spec.min_active, spec.eps, fusion=fusion)
    assert (ids == ids_ref).all(), "top-k ids"
    bad = np.nonzero(skip.astype(bool) != ref["skip"])
    assert bad[0].size == 0, ("skip mask", bad[0][:5], bad[1][:5])
    assert (gh.view(np.uint32) == ref["g_hat"].view(np.uint32)).all(), "g_hat bits"
    assert np.float32(tau).view(np.uint32) == np.float32(ref["tau"]).view(np.uint32), (tau, ref["tau"])
    assert R == int((~ref["skip"]).sum())
    if mode == "ratio":
        assert T * k - R == ref["count"]
    off, perm = ace.ace_last_permutation(handle, N, R)
    off_ref, perm_ref = O.permutation(ids_ref, ref["skip"], N)
    assert (off == off_ref).all() and (perm == perm_ref).all(), "permutation"
    return ref, z


def check_logits(z_gpu, x, w, f32=False, tokens=None):
    """The forward's router logits against the fp64 oracle's, from x."""
    spec = w.spec
    xs = x if tokens is None else x[tokens]
    zg = z_gpu if tokens is None else z_gpu[tokens]
    h = O.rmsnorm(xs, w.gamma, spec.rms_eps)
    z_ref = O.router_logits(h, w.router_w, w.router_b, spec.router_temp)
    compare(zg.astype(np.float64), z_ref, f32=f32, what="router logits")
    return z_ref


def compare(y_gpu, y_ref, f32=False, what="output"):
    """Every row, element by element: rel-L2 and max-abs against the oracle."""
    y_gpu = np.asarray(y_gpu, np.float64)
    y_ref = np.asarray(y_ref, np.float64)
    assert y_gpu.shape == y_ref.shape
    assert np.isfinite(y_gpu).all(), what
    nr = max(np.linalg.norm(y_ref), 1e-30)
    rel = np.linalg.norm(y_gpu - y_ref) / nr
    mx = np.abs(y_gpu - y_ref).max() / max(np.abs(y_ref).max(), 1e-30)
    if f32:
        assert rel <= RTOL_L2_F32, (what, rel)
    else:
        assert rel <= RTOL_L2, (what, rel)
        assert mx <= RTOL_MAX, (what, mx)
    return rel, mx


def bf16_half_ulp(v):
    """Half the spacing of bf16 values at |v| (the bound of one rounding)."""
    a = np.abs(np.asarray(v, np.float64))
    e = np.floor(np.log2(np.maximum(a, 2.0 ** -126)))
    return 0.5 * 2.0 ** (e - 7)


def compare_residual(out_gpu, x_in, y_ref, what="layer output"):
    """A layer that adds its input writes bf16(x + y): compare that with
    x + y_ref. The one rounding of the sum to bf16 moves each element by at
    most half a bf16 spacing of the output; it is allowed on top of the
    output tolerance, which is taken relative to y (the layer's own
    contribution) so that the input does not mask an error in y."""
    out = np.asarray(out_gpu, np.float64)
    want = np.asarray(x_in, np.float64) + y_ref
    err = np.abs(out - want)
    allow = bf16_half_ulp(out)
    l2 = np.linalg.norm(err)
    assert l2 <= RTOL_L2 * np.linalg.norm(y_ref) + np.linalg.norm(allow), (what, l2 / np.linalg.norm(y_ref))
    assert (np.maximum(err - allow, 0.0)).max() <= RTOL_MAX * np.abs(y_ref).max(), what


def note_disagreement(label, dec_replay, dec_indep):
    """Count slots whose fp64 (independent) decision differs from the
    replayed one: a different expert in the slot, or a different skip bit."""
    ids_r, ids_i = dec_replay["ids"], dec_indep["ids"]
    T, k = ids_r.shape
    diff = 0
    tok = 0
    for t in range(T):
        a = {int(e): bool(s) for e, s in zip(ids_r[t], dec_replay["skip"][t])}
        b = {int(e): bool(s) for e, s in zip(ids_i[t], dec_indep["skip"][t])}
        d = sum(1 for e in set(a) | set(b) if a.get(e) != b.get(e))
        diff += d
        tok += d > 0
    DISAGREEMENT.append((label, T * k, diff, T, tok))
    return diff / (T * k)
