"""ACE oracle: a plain, slow CPU implementation of the ACE MoE layer.

TEST INFRASTRUCTURE ONLY. Nothing on the product path may import it.

Source: ACE, "Adaptive Calibration-Free Expert Skipping for MoE-based LLMs".
  * §3.1 Global Spectral Proxy: Eqs. gsp_contribution, swiglu_expert,
    gsp_up_path, gsp_gate_path, gsp_geometric_mean, gsp_layer_normalization,
    gsp_probability; Algorithm 2 (GSP).
  * §3.2 Router-Conditioned Refinement: Eqs. rcr_centered_router,
    rcr_direction_prototype, rcr_raw_amplification, rcr_layer_normalization,
    rcr_contribution, rcr_probability; Algorithm 3 (RCR).
  * §3.2 fusion: Eqs. ace_contribution, ace_candidate_intersection;
    Algorithm 4 (online conservative skipping); Eq. ace_sparse_output.
  * §4.1 Baselines (router-score skipping) and §4.3 ablations (single-view
    GSP / RCR skipping, Min and Mean fusion): the skip-rule variants.
  * App. B.1 budget-to-threshold mapping (quantile rule for tau(q)).

Two families of functions:
  * fp64 ("independent") functions: the layer exactly as the paper defines it,
    every value widened to float64. Library primitives used as steps: matmul,
    sort, exp.
  * fp32 decision spec: the routing/skip decision from given float32 router
    logits, in one fixed IEEE float32 operation order (round to nearest even,
    no fused multiply-add), with its own exp. A GPU kernel that performs the
    same operations in the same order reproduces these bits exactly.

Pins (tests/test_oracle_pins.py): hand-worked examples (tests/golden/), the
skip-ratio-0 reduction to ordinary top-k MoE computed with library softmax and
top-k, a dense brute-force evaluation of all experts on tiny inputs, the
App. A.2.4 identities (max = intersection, skipped-mass ordering, the exact
perturbation identity and its 2*alpha*F_max bound), the App. A.2.1 SwiGLU bound,
router translation invariance (App. A.2.2), the closed-form table means and
scaling laws, the realised skip count of the quantile rule, the exp error
bound against math.exp, and for the skip-rule variants a hand-worked example
(tests/golden/fusion_worked.json), the nesting Max within Mean within Min,
Max / Min as intersection / union of the single views, router-score
skipping as the GSP view with unit tables, and for the layer stack the
identity when every down projection is zero and a dense evaluation of its one
non-zero layer.

Readings where the paper is silent (each also listed in the design notes):
  * gates g are the softmax over the top-k logits (softmax over all experts
    renormalised to the top-k: sum g = 1, as assumed in App. A.2.4);
  * epsilon = 1e-6 everywhere it appears; RMSNorm eps = 1e-6;
  * RCR evaluates f on the prototype q directly (no Gamma), since the expert
    input x is already Gamma-scaled in Eq. swiglu_expert; apply_gamma=True
    gives the other reading;
  * Frobenius norms in GSP exactly as Eqs. gsp_up_path / gsp_gate_path write;
  * top-k ties go to the lower expert index;
  * tau(q) for a given q: tau = the (m+1)-th smallest candidate score, with the
    boundary-tie rule of App. B.1 resolved as documented in tau_from_ratio.
"""
from __future__ import annotations

import math
from decimal import Decimal, getcontext

import numpy as np

__all__ = [
    "rmsnorm", "router_logits", "topk_gates", "silu", "swiglu_expert",
    "FUSIONS", "fused_contribution", "ace_skip", "protected_mask", "tau_from_ratio", "ace_decide", "moe_forward",
    "moe_stack_forward", "permutation", "gsp_table", "rcr_table",
    "exp32", "decide_fp32", "route_fp32", "tau_from_ratio_fp32", "llround_pos",
    "to_f64",
]


def to_f64(a: np.ndarray) -> np.ndarray:
    """Widen a stored array to float64 (uint16 arrays are bf16 bit patterns)."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


# --------------------------------------------------------------------------
# fp64 layer (the paper's definitions)
# --------------------------------------------------------------------------

def rmsnorm(x: np.ndarray, gamma: np.ndarray, rms_eps: float) -> np.ndarray:
    """Expert/router input x = x_bar * Gamma (§3.1, before Eq. swiglu_expert).

    x_bar = x / sqrt(mean(x^2) + rms_eps) is the RMS-normalised direction and
    Gamma = Diag(gamma) the learned RMSNorm scale.
    """
    x = to_f64(x)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + rms_eps) * to_f64(gamma)


def router_logits(h: np.ndarray, router_w: np.ndarray, router_b: np.ndarray | None,
                  temp: float = 1.0) -> np.ndarray:
    """z_e(x) = x^T w_e + b_e (§3.2; App. A.2.2 Eq. app_router_logit), over temp."""
    z = to_f64(h) @ to_f64(router_w).T
    if router_b is not None:
        z = z + to_f64(router_b)
    return z / temp


def topk_gates(z: np.ndarray, k: int) -> tuple[np.ndarray, np.ndarray]:
    """Top-k routed experts and gates {(e_i, g_i)} (§3.1; Algorithm 1).

    Slots are in rank order (logit descending, ties to the lower expert id),
    so slot 0 is the top-1 expert. g is the softmax restricted to the top-k.
    """
    z = np.asarray(z, dtype=np.float64)
    ids = np.argsort(-z, axis=1, kind="stable")[:, :k]
    zt = np.take_along_axis(z, ids, axis=1)
    e = np.exp(zt - zt[:, :1])
    g = e / e.sum(axis=1, keepdims=True)
    return ids.astype(np.int64), g


def silu(u: np.ndarray) -> np.ndarray:
    """SiLU(z) = z * sigma(z) (App. A.2.1 Eq. app_silu_scalar_bound)."""
    return u / (1.0 + np.exp(-u))


def swiglu_expert(x: np.ndarray, w_gate_e: np.ndarray, w_up_e: np.ndarray,
                  w_down_e: np.ndarray) -> np.ndarray:
    """f(x) = (SiLU(x W_gate) ⊙ x W_up) W_down (Eq. swiglu_expert, no bias).

    Weights are stored nn.Linear style: w_gate_e, w_up_e are [m, d] (the
    paper's W_gate, W_up in R^{d x m}, transposed) and w_down_e is [d, m].
    """
    x = to_f64(x)
    u = x @ to_f64(w_gate_e).T
    v = x @ to_f64(w_up_e).T
    return (silu(u) * v) @ to_f64(w_down_e).T


# Skip rules. "max" is ACE (Eq. ace_contribution). The others are the
# variants the paper compares against it: "min" and "mean" fusion
# (§4.3, Tab. fusion_ablation), a single view "gsp" or "rcr" (§4.3,
# Tab. ablation), and router-score skipping "score" (§4.1 Baselines), which
# thresholds the routing gate itself.
FUSIONS = ("max", "min", "mean", "gsp", "rcr", "score")


def fused_contribution(p_gsp: np.ndarray, p_rcr: np.ndarray, g: np.ndarray, fusion: str) -> np.ndarray:
    """Per-slot score c of a skip rule; a slot is a skip candidate when c < tau."""
    if fusion == "max":
        return np.maximum(p_gsp, p_rcr)                 # Eq. ace_contribution
    if fusion == "min":
        return np.minimum(p_gsp, p_rcr)
    if fusion == "mean":
        return (p_gsp + p_rcr) / 2.0
    if fusion == "gsp":
        return p_gsp
    if fusion == "rcr":
        return p_rcr
    if fusion == "score":
        return np.asarray(g, dtype=np.float64)
    raise ValueError(f"unknown fusion {fusion!r}")


def ace_skip(ids: np.ndarray, g: np.ndarray, a_gsp: np.ndarray, a_rcr: np.ndarray,
             tau: float, m_min: int, eps: float, fusion: str = "max"):
    """Algorithm 4 (online conservative expert skipping), vectorised over tokens.

    The candidate set of each rule is formed from the per-view sets as the
    paper describes it: ACE skips a slot only when both views call it
    dispensable (intersection, Eq. ace_candidate_intersection); "min" when
    either does (union); "gsp" / "rcr" use one view; "mean" and "score"
    threshold their score directly.

    Returns (skip [T,k] bool, g_hat [T,k] (0 where skipped), c [T,k],
    p_gsp [T,k], p_rcr [T,k]).
    """
    a_gsp = to_f64(a_gsp)
    a_rcr = to_f64(a_rcr)
    g = np.asarray(g, dtype=np.float64)
    T, k = g.shape
    s_gsp = g * a_gsp[ids]                              # Eq. gsp_contribution
    s_rcr = g * a_rcr[ids]                              # Eq. rcr_contribution
    z_gsp = s_gsp.sum(axis=1, keepdims=True) + eps
    z_rcr = s_rcr.sum(axis=1, keepdims=True) + eps
    p_gsp = s_gsp / z_gsp                               # Eq. gsp_probability
    p_rcr = s_rcr / z_rcr                               # Eq. rcr_probability
    c = fused_contribution(p_gsp, p_rcr, g, fusion)
    low_gsp = p_gsp < tau                               # Eq. gsp_candidate_set
    low_rcr = p_rcr < tau                               # Eq. rcr_candidate_set
    if fusion == "max":
        skip = low_gsp & low_rcr                        # Eq. ace_candidate_intersection
    elif fusion == "min":
        skip = low_gsp | low_rcr
    elif fusion == "gsp":
        skip = low_gsp
    elif fusion == "rcr":
        skip = low_rcr
    else:
        skip = c < tau
    top1 = np.argmax(g, axis=1)                         # top-1 by original gate
    skip[np.arange(T), top1] = False
    if m_min > 1:
        for t in range(T):
            active = k - int(skip[t].sum())
            if active < m_min:
                cand = [i for i in range(k) if skip[t, i]]
                cand.sort(key=lambda i: (-c[t, i], i))   # c descending, lower rank first
                for i in cand[: m_min - active]:
                    skip[t, i] = False
    kept = ~skip
    z_gate = (g * kept).sum(axis=1, keepdims=True) + eps
    g_hat = np.where(kept, g / z_gate, 0.0)
    return skip, g_hat, c, p_gsp, p_rcr


def protected_mask(c: np.ndarray, m_min: int) -> np.ndarray:
    """Slots excluded from the threshold search (App. B.1): the top-1 slot and,
    for m_min > 1, the m_min-1 highest-c other slots of each token (the ones the
    minimum-active rule of Algorithm 4 would restore first)."""
    T, k = c.shape
    prot = np.zeros((T, k), dtype=bool)
    prot[:, 0] = True
    extra = max(0, min(m_min, k) - 1)
    if extra:
        for t in range(T):
            others = sorted(range(1, k), key=lambda i: (-c[t, i], i))
            for i in others[:extra]:
                prot[t, i] = True
    return prot


def llround_pos(x: float) -> int:
    """Round a non-negative double half away from zero (C llround)."""
    n = int(x)
    if x - n >= 0.5:
        n += 1
    return n


def tau_from_ratio(c: np.ndarray, prot: np.ndarray, q: float):
    """Budget-to-threshold mapping (App. B.1), fp64 scores.

    m_q = clip(round(q * N_all), 0, N_cand). tau is placed so that exactly the
    m_q smallest candidate scores satisfy c < tau: tau = c_(m_q+1) when it
    differs from c_(m_q). When the boundary values tie, the two adjacent
    thresholds are tau = v (realising #{c < v}) and the next representable
    value above v (realising #{c <= v}); the one whose count is closer to m_q
    is taken, the lower count on a tie. m_q = 0 gives tau = 0 and m_q = N_cand
    gives tau = +inf.
    Returns (tau, m_q, realised count).
    """
    n_all = c.size
    cand = np.sort(c[~prot].ravel())
    n_cand = cand.size
    m = min(max(llround_pos(float(q) * n_all), 0), n_cand)
    if m == 0:
        return 0.0, m, 0
    if m == n_cand:
        return math.inf, m, n_cand
    v = cand[m]
    lo = int(np.sum(cand < v))
    hi = int(np.sum(cand <= v))
    if lo == m:
        return float(v), m, lo
    if (m - lo) <= (hi - m):
        return float(v), m, lo
    return float(np.nextafter(v, np.inf)), m, hi


def ace_decide(z: np.ndarray, k: int, a_gsp, a_rcr, mode: str, value: float,
               m_min: int = 1, eps: float = 1e-6, fusion: str = "max") -> dict:
    """Routing + skipping decision in fp64 from logits z [T, N]."""
    ids, g = topk_gates(z, k)
    # scores at tau = 0 (no skip) give c for the threshold search
    _, _, c, _, _ = ace_skip(ids, g, a_gsp, a_rcr, 0.0, 1, eps, fusion)
    if mode == "ratio":
        prot = protected_mask(c, m_min)
        tau, m_q, cnt = tau_from_ratio(c, prot, value)
    else:
        tau, m_q, cnt = float(value), None, None
    skip, g_hat, c, p_gsp, p_rcr = ace_skip(ids, g, a_gsp, a_rcr, tau, m_min, eps, fusion)
    return dict(ids=ids, g=g, skip=skip, g_hat=g_hat, c=c, p_gsp=p_gsp, p_rcr=p_rcr,
                tau=tau, m_q=m_q, count=cnt)


def moe_forward(x: np.ndarray, w, mode: str = "threshold", value: float = 0.0,
                decision: dict | None = None, return_decision: bool = False,
                tokens: np.ndarray | None = None, fusion: str = "max"):
    """ACE MoE layer output y_t = sum_{i in I_t} g_hat_i f_{e_i}(x_t)
    (Eq. ace_sparse_output; Algorithm 1 online loop for one layer), fp64.

    `w` is a synth.LayerWeights-like object (router_w, router_b, w_gate, w_up,
    w_down, gamma, spec). `a_gsp`/`a_rcr` tables are read from w.extra.
    No residual connection is inside the layer. With `tokens` (indices), the
    decision is still taken over the whole batch (the per-batch threshold
    needs every token) but the experts are evaluated for those tokens only;
    the returned y then has one row per listed token.
    """
    spec = w.spec
    h = rmsnorm(x, w.gamma, spec.rms_eps)
    if decision is None:
        z = router_logits(h, w.router_w, w.router_b, spec.router_temp)
        decision = ace_decide(z, spec.top_k, w.extra["a_gsp"], w.extra["a_rcr"], mode,
                              value, spec.min_active, spec.eps, fusion)
    ids, skip, g_hat = decision["ids"], decision["skip"], decision["g_hat"]
    rows = np.arange(h.shape[0]) if tokens is None else np.asarray(tokens)
    hs, ids_s, skip_s, gh_s = h[rows], ids[rows], skip[rows], g_hat[rows]
    y = np.zeros_like(hs)
    for e in range(spec.n_experts):
        sel = (ids_s == e) & ~skip_s
        tok, slot = np.nonzero(sel)
        if tok.size == 0:
            continue
        f = swiglu_expert(hs[tok], w.w_gate[e], w.w_up[e], w.w_down[e])
        y[tok] += gh_s[tok, slot][:, None] * f
    if return_decision:
        return y, decision
    return y


def moe_stack_forward(x: np.ndarray, layers, mode: str, value: float) -> np.ndarray:
    """A stack of ACE MoE layers with a residual around each layer:
    x_{l+1} = x_l + y_l(x_l). Each layer applies its own RMSNorm."""
    cur = to_f64(x)
    for w in layers:
        cur = cur + moe_forward(cur, w, mode, value)
    return cur


def permutation(ids: np.ndarray, skip: np.ndarray, n_experts: int):
    """Retained slots grouped by expert: offsets [N+1] (exclusive scan of the
    per-expert counts) and perm [R] = slot ids t*k+i sorted by (expert, token)."""
    T, k = ids.shape
    offsets = np.zeros(n_experts + 1, dtype=np.int64)
    perm = []
    for e in range(n_experts):
        tok, slot = np.nonzero((ids == e) & ~skip)
        order = np.argsort(tok, kind="stable")
        perm.extend((tok[order] * k + slot[order]).tolist())
        offsets[e + 1] = offsets[e] + tok.size
    return offsets, np.asarray(perm, dtype=np.int64)


# --------------------------------------------------------------------------
# Offline tables (Algorithms 2 and 3), fp64, direct products
# --------------------------------------------------------------------------

def gsp_table(gamma, w_gate, w_up, w_down, eps: float = 1e-6) -> np.ndarray:
    """Algorithm 2 (GSP). A^GSP(e) = a_e / (mean_j a_j + eps) with
    a_e = sqrt(a_up * a_gate), a_up = ||U||_F ||G W_down||_F,
    a_gate = ||G||_F ||U W_down||_F, G = Gamma W_gate, U = Gamma W_up
    (Eqs. gsp_up_path, gsp_gate_path, gsp_geometric_mean, gsp_layer_normalization).
    """
    gam = to_f64(gamma)
    n = w_gate.shape[0]
    a = np.zeros(n)
    for e in range(n):
        G = gam[:, None] * to_f64(w_gate[e]).T         # [d, m]
        U = gam[:, None] * to_f64(w_up[e]).T           # [d, m]
        Wd = to_f64(w_down[e]).T                       # [m, d]
        a_up = np.linalg.norm(U, "fro") * np.linalg.norm(G @ Wd, "fro")
        a_gate = np.linalg.norm(G, "fro") * np.linalg.norm(U @ Wd, "fro")
        a[e] = math.sqrt(a_up * a_gate)
    return a / (a.mean() + eps)


def rcr_table(router_w, gamma, w_gate, w_up, w_down, eps: float = 1e-6,
              apply_gamma: bool = False) -> np.ndarray:
    """Algorithm 3 (RCR). Centred router weights (Eq. rcr_centered_router),
    prototypes q_e = rho * w~_e / (RMS(w~_e) + eps) with rho = 1
    (Eq. rcr_direction_prototype), a_e = ||f_e(q_e)||_2 / (||q_e||_2 + eps)
    (Eq. rcr_raw_amplification), A^RCR(e) = a_e / (mean_j a_j + eps)
    (Eq. rcr_layer_normalization).
    """
    wr = to_f64(router_w)
    n, d = wr.shape
    wt = wr - wr.mean(axis=0, keepdims=True)
    a = np.zeros(n)
    for e in range(n):
        r = math.sqrt(float(np.sum(wt[e] ** 2)) / d)
        q = wt[e] / (r + eps)
        xin = q * to_f64(gamma) if apply_gamma else q
        y = swiglu_expert(xin[None, :], w_gate[e], w_up[e], w_down[e])[0]
        a[e] = np.linalg.norm(y) / (np.linalg.norm(q) + eps)
    return a / (a.mean() + eps)


# --------------------------------------------------------------------------
# fp32 decision spec
# --------------------------------------------------------------------------

def _ln2_split():
    """Cody & Waite (1980) split of ln 2 into hi + lo: hi keeps the leading
    9 significant bits (so n*hi is exact in float32 for |n| < 2^15) and lo is
    the float32 rounding of ln2 - hi, both derived here in 50-digit decimal."""
    getcontext().prec = 50
    ln2 = Decimal(2).ln()
    hi = Decimal(int(ln2 * 512)) / Decimal(512) if (ln2 * 512) % 1 < Decimal("0.5") \
        else Decimal(int(ln2 * 512) + 1) / Decimal(512)
    lo = ln2 - hi
    return np.float32(float(hi)), np.float32(float(lo))


_LN2_HI, _LN2_LO = _ln2_split()
_LOG2E = np.float32(1.0 / math.log(2.0))
_INV_FACT = [np.float32(1.0 / math.factorial(j)) for j in range(8)]


def exp32(x: np.ndarray) -> np.ndarray:
    """exp(x) for float32 x <= 0, in a fixed float32 operation sequence.

    Cody-Waite range reduction x = n ln2 + r with n = rint(x log2 e), r in
    about [-ln2/2, ln2/2]; a degree-7 Taylor polynomial sum_j r^j / j! in Horner
    form (separate multiply and add, each rounded); scaling by 2^n through the
    exponent bits. Returns 0 for x < -87.
    """
    x = np.asarray(x, dtype=np.float32)
    n = np.rint(x * _LOG2E).astype(np.float32)
    r = (x - n * _LN2_HI).astype(np.float32)
    r = (r - n * _LN2_LO).astype(np.float32)
    p = np.full_like(r, _INV_FACT[7])
    for j in range(6, -1, -1):
        p = (p * r).astype(np.float32)
        p = (p + _INV_FACT[j]).astype(np.float32)
    ni = np.clip(n, -126, 127).astype(np.int32)
    scale = ((ni + 127).astype(np.uint32) << 23).view(np.float32)
    out = (p * scale).astype(np.float32)
    return np.where(x < np.float32(-87.0), np.float32(0.0), out).astype(np.float32)


def route_fp32(z: np.ndarray, k: int):
    """Top-k slots in rank order (logit descending, ties to the lower expert
    index) and gates g_i = e_i / S with e_i = exp32(z_i - z_0) and
    S = (((e_0 + e_1) + e_2) + ...) summed in rank order, all float32."""
    z = np.asarray(z, dtype=np.float32)
    ids = np.argsort(-z, axis=1, kind="stable")[:, :k]
    zt = np.take_along_axis(z, ids, axis=1)
    e = exp32((zt - zt[:, :1]).astype(np.float32))
    s = e[:, 0].copy()
    for i in range(1, k):
        s = (s + e[:, i]).astype(np.float32)
    g = (e / s[:, None]).astype(np.float32)
    return ids.astype(np.int32), g


def _scores_fp32(ids, g, a_gsp, a_rcr, eps32, fusion="max"):
    k = g.shape[1]
    sg = (g * a_gsp[ids]).astype(np.float32)
    sr = (g * a_rcr[ids]).astype(np.float32)
    zg = sg[:, 0].copy()
    zr = sr[:, 0].copy()
    for i in range(1, k):
        zg = (zg + sg[:, i]).astype(np.float32)
        zr = (zr + sr[:, i]).astype(np.float32)
    zg = (zg + eps32).astype(np.float32)
    zr = (zr + eps32).astype(np.float32)
    pg = (sg / zg[:, None]).astype(np.float32)
    pr = (sr / zr[:, None]).astype(np.float32)
    if fusion == "max":
        c = np.maximum(pg, pr)
    elif fusion == "min":
        c = np.minimum(pg, pr)
    elif fusion == "mean":
        c = (pg + pr).astype(np.float32) * np.float32(0.5)
    elif fusion == "gsp":
        c = pg
    elif fusion == "rcr":
        c = pr
    elif fusion == "score":
        c = g
    else:
        raise ValueError(f"unknown fusion {fusion!r}")
    return np.asarray(c, dtype=np.float32), pg, pr


def _protected_fp32(c: np.ndarray, m_min: int) -> np.ndarray:
    T, k = c.shape
    prot = np.zeros((T, k), dtype=bool)
    prot[:, 0] = True
    extra = max(0, min(m_min, k) - 1)
    if extra:
        for t in range(T):
            others = sorted(range(1, k), key=lambda i: (-float(c[t, i]), i))
            for i in others[:extra]:
                prot[t, i] = True
    return prot


def tau_from_ratio_fp32(c: np.ndarray, prot: np.ndarray, q: float):
    """App. B.1 mapping on float32 scores; same rule as tau_from_ratio with
    float32 thresholds (next representable float32 above v on a tie).
    q is taken as float32 and m_q = llround(double(q) * N_all)."""
    n_all = c.size
    cand = np.sort(c[~prot].ravel().astype(np.float32))
    n_cand = cand.size
    m = min(max(llround_pos(float(np.float32(q)) * float(n_all)), 0), n_cand)
    if m == 0:
        return np.float32(0.0), m, 0
    if m == n_cand:
        return np.float32(np.inf), m, n_cand
    v = cand[m]
    lo = int(np.sum(cand < v))
    hi = int(np.sum(cand <= v))
    if lo == m or (m - lo) <= (hi - m):
        return np.float32(v), m, lo
    return np.nextafter(np.float32(v), np.float32(np.inf)), m, hi


def decide_fp32(ids: np.ndarray, g: np.ndarray, a_gsp, a_rcr, mode: str, value: float,
                m_min: int = 1, eps: float = 1e-6, fusion: str = "max") -> dict:
    """Algorithm 4 in the fixed float32 operation order, from rank-ordered
    (ids, g). tau: the given float32 threshold, or tau_from_ratio_fp32.

    Order: s = g * A[e]; Z = (sum in rank order) + eps; p = s / Z;
    c = max(p_gsp, p_rcr) (other rules: min, (p_gsp + p_rcr) * 0.5, p_gsp,
    p_rcr, or g); skip = rank != 0 and c < tau; minimum-active
    restore in c-descending order (lower rank first on ties);
    Z_gate = (sum of kept g in rank order) + eps; g_hat = g / Z_gate.
    """
    g = np.asarray(g, dtype=np.float32)
    T, k = g.shape
    eps32 = np.float32(eps)
    a_gsp = np.asarray(a_gsp, dtype=np.float32)
    a_rcr = np.asarray(a_rcr, dtype=np.float32)
    c, pg, pr = _scores_fp32(ids, g, a_gsp, a_rcr, eps32, fusion)
    if mode == "ratio":
        prot = _protected_fp32(c, m_min)
        tau, m_q, cnt = tau_from_ratio_fp32(c, prot, value)
    else:
        tau, m_q, cnt = np.float32(value), None, None
    skip = c < tau
    skip[:, 0] = False
    if m_min > 1:
        for t in range(T):
            active = k - int(skip[t].sum())
            if active < m_min:
                cand = [i for i in range(k) if skip[t, i]]
                cand.sort(key=lambda i: (-float(c[t, i]), i))
                for i in cand[: m_min - active]:
                    skip[t, i] = False
    zg = np.zeros(T, dtype=np.float32)
    for i in range(k):
        zg = np.where(skip[:, i], zg, (zg + g[:, i]).astype(np.float32)).astype(np.float32)
    zg = (zg + eps32).astype(np.float32)
    g_hat = np.where(skip, np.float32(0.0), (g / zg[:, None]).astype(np.float32))
    return dict(ids=ids, g=g, skip=skip, g_hat=g_hat.astype(np.float32), c=c,
                p_gsp=pg, p_rcr=pr, tau=np.float32(tau), m_q=m_q, count=cnt)
