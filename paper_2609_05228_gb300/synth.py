"""Seeded synthetic workloads for the ACE MoE layer.

This module only draws random numbers and rounds them to the storage dtype.
It holds none of the layer's arithmetic: no normalisation, routing, skipping
or expert math. The CPU oracle (tests) and the CUDA path both consume exactly
the arrays produced here.

Recipe (the paper evaluates Qwen3-30B-A3B-shaped MoE layers in BF16, §4):
  * x ~ N(0, 1) per element.
  * router, gate, up and down weights ~ N(0, 0.02^2) (standard deviation 0.02).
  * RMSNorm gamma ~ 1 + U(-0.1, 0.1).
  * router bias: zero, or a Zipf-shaped popularity profile
    b_e = -beta * s * log(r_e) with r a seeded permutation of the ranks 1..N.
  * bf16 configurations round every value to bf16 (round to nearest even)
    once; both sides see the same bits.

Large arrays are generated in fixed chunks, each from its own child seed of
one SeedSequence, so the values do not depend on the thread count.

Weights use the nn.Linear convention [out_features, in_features]:
  router_w [N, d], w_gate [N, m, d], w_up [N, m, d], w_down [N, d, m].
bf16 arrays are returned as uint16 bit patterns.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

# Elements per generation chunk. Fixed: changing it changes every value.
_CHUNK = 1 << 22

# Zipf router-bias profile b_e = -beta * ZIPF_S * log(r_e). beta depends on
# the layer shape (the logit noise grows with the hidden size, the ranks with
# the expert count), so each named shape carries its own value, found by a 1-D
# search with the CPU oracle's routing (tests/golden/derive_zipf_beta.py) so
# that the routed-slot counts, sorted, fall with log-log slope -1.1 +- 0.05
# over the popularity ranks 1..N/2; the tests check that slope per shape.
ZIPF_S = 1.1
ZIPF_BETA = 0.59          # hidden 2048, 128 experts, top-8 (4096 tokens: -1.10)
ZIPF_BETA_LARGE = 0.70    # hidden 4096, 256 experts, top-8 (8192 tokens: -1.105; 2048: -1.08)


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float values to bf16 (round to nearest, ties to even); return uint16 bits."""
    f = np.ascontiguousarray(a, dtype=np.float32)
    u = f.view(np.uint32)
    lsb = (u >> 16) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> 16
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _fill_normal(shape, seed: int, scale: float, out_bf16: bool, mean: float = 0.0) -> np.ndarray:
    n = int(np.prod(shape))
    nchunks = max(1, (n + _CHUNK - 1) // _CHUNK)
    children = np.random.SeedSequence(seed).spawn(nchunks)
    out = np.empty(n, dtype=np.uint16 if out_bf16 else np.float32)

    def work(i: int) -> None:
        lo = i * _CHUNK
        hi = min(n, lo + _CHUNK)
        g = np.random.Generator(np.random.PCG64(children[i]))
        v = g.standard_normal(hi - lo, dtype=np.float32)
        if scale != 1.0:
            v *= np.float32(scale)
        if mean != 0.0:
            v += np.float32(mean)
        out[lo:hi] = bf16_bits(v) if out_bf16 else v

    threads = min(nchunks, os.cpu_count() or 1, 32)
    if threads <= 1:
        for i in range(nchunks):
            work(i)
    else:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(work, range(nchunks)))
    return out.reshape(shape)


@dataclass
class LayerSpec:
    hidden: int
    n_experts: int
    top_k: int
    ffn: int
    dtype: str = "bf16"          # "bf16" or "f32"
    zipf: bool = False           # Zipf-skewed router bias
    rms_eps: float = 1e-6
    eps: float = 1e-6            # the paper's numerical constant epsilon
    router_temp: float = 1.0
    min_active: int = 1
    zipf_beta: float = ZIPF_BETA  # scale of the Zipf router bias (used when zipf)


@dataclass
class LayerWeights:
    spec: LayerSpec
    router_w: np.ndarray          # [N, d]
    router_b: np.ndarray          # [N] float32 (zeros when not Zipf)
    w_gate: np.ndarray            # [N, m, d]
    w_up: np.ndarray              # [N, m, d]
    w_down: np.ndarray            # [N, d, m]
    gamma: np.ndarray             # [d]
    seed: int = 0
    extra: dict = field(default_factory=dict)

    @property
    def bf16(self) -> bool:
        return self.spec.dtype == "bf16"

    def f32(self, name: str) -> np.ndarray:
        """A weight array widened exactly to float32."""
        a = getattr(self, name)
        return bf16_to_f32(a) if a.dtype == np.uint16 else a


def make_layer(spec: LayerSpec, seed: int) -> LayerWeights:
    """Seeded layer weights: each tensor gets its own child seed of `seed`."""
    bf = spec.dtype == "bf16"
    d, n, m = spec.hidden, spec.n_experts, spec.ffn
    ss = np.random.SeedSequence(seed)
    s_router, s_gate, s_up, s_down, s_gamma, s_zipf = [
        int(c.generate_state(1, np.uint32)[0]) for c in ss.spawn(6)]
    router_w = _fill_normal((n, d), s_router, 0.02, bf)
    w_gate = _fill_normal((n, m, d), s_gate, 0.02, bf)
    w_up = _fill_normal((n, m, d), s_up, 0.02, bf)
    w_down = _fill_normal((n, d, m), s_down, 0.02, bf)
    g = np.random.Generator(np.random.PCG64(s_gamma))
    gamma = (1.0 + g.uniform(-0.1, 0.1, size=d)).astype(np.float32)
    if bf:
        gamma = bf16_bits(gamma)
    router_b = np.zeros(n, dtype=np.float32)
    if spec.zipf:
        gz = np.random.Generator(np.random.PCG64(s_zipf))
        ranks = gz.permutation(n) + 1
        b = -spec.zipf_beta * ZIPF_S * np.log(ranks.astype(np.float64))
        b -= b.mean()
        router_b = b.astype(np.float32)
    return LayerWeights(spec, router_w, router_b, w_gate, w_up, w_down, gamma, seed)


def make_tokens(spec: LayerSpec, n_tokens: int, seed: int) -> np.ndarray:
    """x ~ N(0,1), [T, d]; uint16 bf16 bits or float32."""
    return _fill_normal((n_tokens, spec.hidden), seed, 1.0, spec.dtype == "bf16")


def make_logits(n_tokens: int, n_experts: int, seed: int, scale: float = 0.9,
                tie_fraction: float = 0.0) -> np.ndarray:
    """fp32 router-logit-like values N(0, scale^2), [T, N].

    With tie_fraction > 0, that fraction of tokens gets duplicated logit values
    (exact ties) so that tie-breaking paths are exercised.
    """
    g = np.random.Generator(np.random.PCG64(seed))
    z = (g.standard_normal((n_tokens, n_experts)) * scale).astype(np.float32)
    if tie_fraction > 0 and n_tokens > 0:
        nt = max(1, int(round(tie_fraction * n_tokens)))
        rows = g.choice(n_tokens, size=min(nt, n_tokens), replace=False)
        for r in rows:
            src = g.integers(0, n_experts)
            dst = g.choice(n_experts, size=min(3, n_experts), replace=False)
            z[r, dst] = z[r, src]
    return z


def make_tables(n_experts: int, seed: int, spread: float = 0.05) -> tuple[np.ndarray, np.ndarray]:
    """Positive per-expert table values around 1 (for tests that need tables only)."""
    g = np.random.Generator(np.random.PCG64(seed))
    a = (1.0 + spread * g.standard_normal(n_experts)).clip(0.05).astype(np.float32)
    b = (1.0 + spread * g.standard_normal(n_experts)).clip(0.05).astype(np.float32)
    return a, b


# Named workloads: the shapes of the paper's evaluated models (Qwen3-30B-A3B
# MoE layer: hidden 2048, 128 experts, top-8, expert FFN 768) plus a tiny
# fp32 layer and a large layer.
def spec_tiny() -> LayerSpec:
    return LayerSpec(256, 16, 4, 128, dtype="f32")


def spec_qwen(zipf: bool = False) -> LayerSpec:
    return LayerSpec(2048, 128, 8, 768, dtype="bf16", zipf=zipf)


def spec_large(zipf: bool = True, n_experts: int = 256) -> LayerSpec:
    """The large layer; n_experts < 256 gives a smaller case with the same
    expert shape (for profiler captures that must stay a few GB)."""
    return LayerSpec(4096, n_experts, 8, 2048, dtype="bf16", zipf=zipf, zipf_beta=ZIPF_BETA_LARGE)
