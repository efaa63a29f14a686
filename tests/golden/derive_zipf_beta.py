"""Derive the Zipf router-bias scale beta of each named layer shape.

The prefill workloads route tokens with a Zipf-skewed expert popularity: the
router bias is b_e = -beta * 1.1 * log(r_e) with r a seeded permutation of the
ranks. For each shape this script bisects beta so that, with the CPU oracle's
RMSNorm, router logits and top-k on the workload's own seeded tokens, the
per-expert routed-slot counts sorted in descending order fall with a log-log
slope of -1.1 over the popularity ranks 1..N/2. It prints the values that
paper_2609_05228_gb300/synth.py holds (rounded to two decimals);
tests/test_oracle_pins.py checks the slope they give.

Run from the repository root:  python tests/golden/derive_zipf_beta.py
"""
import dataclasses
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle as O  # noqa: E402
from paper_2609_05228_gb300 import synth  # noqa: E402

TARGET = -1.1


def routed_slope(spec, beta, T, seed_w=0, seed_x=1):
    # the expert FFN width does not enter the routing: a narrow one keeps this cheap
    s = dataclasses.replace(spec, ffn=64, zipf=True, zipf_beta=beta)
    w = synth.make_layer(s, seed=seed_w)
    x = synth.make_tokens(s, T, seed=seed_x)
    h = O.rmsnorm(x, w.gamma, s.rms_eps)
    z = O.router_logits(h, w.router_w, w.router_b, s.router_temp)
    ids, _ = O.topk_gates(z, s.top_k)
    n = s.n_experts
    counts = np.sort(np.bincount(ids.ravel(), minlength=n))[::-1].astype(np.float64)
    r = np.arange(1, n // 2 + 1)
    return float(np.polyfit(np.log(r), np.log(np.maximum(counts[: n // 2], 1)), 1)[0])


def bisect_beta(spec, T, lo=0.2, hi=1.5, iters=14):
    # the slope falls monotonically as beta grows
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if routed_slope(spec, mid, T) > TARGET:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


if __name__ == "__main__":
    for name, spec, T in [("hidden 2048, 128 experts (4096 tokens)", synth.spec_qwen(zipf=True), 4096),
                          ("hidden 4096, 256 experts (8192 tokens)", synth.spec_large(zipf=True), 8192)]:
        beta = bisect_beta(spec, T)
        print(f"{name}: beta = {beta:.4f} -> {round(beta, 2):.2f} "
              f"(slope at the rounded value {routed_slope(spec, round(beta, 2), T):.3f})")
