"""Offline GSP and RCR tables (ACE Algorithms 2 and 3), host CPU.

The tables are computed once per layer from the frozen weights and handed to
ace_layer_create(). No calibration data is involved.

GSP (§3.1, Eqs. gsp_up_path .. gsp_layer_normalization). With the paper's
row-vector convention G = Gamma W_gate and U = Gamma W_up (d x m) and
W_down (m x d):
    a_up   = ||U||_F * ||G W_down||_F
    a_gate = ||G||_F * ||U W_down||_F
    a~     = sqrt(a_up * a_gate),   A(e) = a~_e / (mean_j a~_j + eps).
The products G W_down are d x d; their Frobenius norms are taken through
m x m Gram matrices instead, ||G W||_F^2 = <G^T G, W W^T>_F, which costs
3 d m^2 multiply-adds per expert instead of 2 d^2 m.

RCR (§3.2, Eqs. rcr_centered_router .. rcr_layer_normalization): centred
router rows w~_e, prototypes q_e = w~_e / (RMS(w~_e) + eps) (rho = 1),
a~_e = ||f_e(q_e)||_2 / (||q_e||_2 + eps), A(e) = a~_e / (mean a~ + eps).
f is applied to q directly; apply_gamma=True scales q by gamma first.

Weights are nn.Linear-shaped: w_gate, w_up [N, m, d]; w_down [N, d, m];
bf16 arrays are uint16 bit patterns.
"""
from __future__ import annotations

import numpy as np


def _f32(a: np.ndarray) -> np.ndarray:
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32)
    return a.astype(np.float32, copy=False)


def gsp_table(gamma, w_gate, w_up, w_down, eps: float = 1e-6) -> np.ndarray:
    gam2 = _f32(gamma).astype(np.float64) ** 2
    n = w_gate.shape[0]
    raw = np.empty(n, dtype=np.float64)
    for e in range(n):
        wg = _f32(w_gate[e]).astype(np.float64)          # [m, d]
        wu = _f32(w_up[e]).astype(np.float64)            # [m, d]
        wd = _f32(w_down[e]).astype(np.float64)          # [d, m]
        gram_g = (wg * gam2) @ wg.T                      # G^T G   [m, m]
        gram_u = (wu * gam2) @ wu.T                      # U^T U   [m, m]
        gram_d = wd.T @ wd                               # W_d W_d^T (paper W_d = wd.T)
        fro_g2 = np.trace(gram_g)
        fro_u2 = np.trace(gram_u)
        fro_gd2 = float(np.vdot(gram_g, gram_d))
        fro_ud2 = float(np.vdot(gram_u, gram_d))
        a_up2 = fro_u2 * max(fro_gd2, 0.0)
        a_gate2 = fro_g2 * max(fro_ud2, 0.0)
        raw[e] = (a_up2 * a_gate2) ** 0.25
    return (raw / (raw.mean() + eps)).astype(np.float32)


def rcr_table(router_w, gamma, w_gate, w_up, w_down, eps: float = 1e-6,
              apply_gamma: bool = False) -> np.ndarray:
    wr = _f32(router_w).astype(np.float64)
    n, d = wr.shape
    centred = wr - wr.mean(axis=0)
    rms = np.sqrt((centred ** 2).sum(axis=1) / d)
    protos = centred / (rms + eps)[:, None]
    raw = np.empty(n, dtype=np.float64)
    gam = _f32(gamma).astype(np.float64)
    for e in range(n):
        q = protos[e]
        xin = q * gam if apply_gamma else q
        u = _f32(w_gate[e]).astype(np.float64) @ xin
        v = _f32(w_up[e]).astype(np.float64) @ xin
        a = u / (1.0 + np.exp(-u)) * v
        y = _f32(w_down[e]).astype(np.float64) @ a
        raw[e] = np.sqrt(y @ y) / (np.sqrt(q @ q) + eps)
    return (raw / (raw.mean() + eps)).astype(np.float32)


def tables(layer, eps: float | None = None, apply_gamma: bool = False):
    """(A^GSP, A^RCR) as float32 arrays for a synth.LayerWeights-like layer."""
    e = layer.spec.eps if eps is None else eps
    a = gsp_table(layer.gamma, layer.w_gate, layer.w_up, layer.w_down, e)
    r = rcr_table(layer.router_w, layer.gamma, layer.w_gate, layer.w_up, layer.w_down, e,
                  apply_gamma)
    return a, r
