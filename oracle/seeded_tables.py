"""GSP / RCR tables (Algorithms 2 and 3) of the seeded benchmark layers,
computed by the CPU oracle and stored in oracle/seeded_tables.json.

TEST INFRASTRUCTURE ONLY: bench.py's reference arm (the oracle timed on the
host) reads them, so that the arm runs the oracle alone and needs no table
tool of the library; the large layer's fp64 direct products take minutes, too
long to recompute on every run. Regenerate from the repository root with
    python -m oracle.seeded_tables
Each entry is keyed by the layer shape and weight seed (the router bias, and
so the Zipf profile, does not enter either table).
"""
from __future__ import annotations

import json
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
PATH = os.path.join(HERE, "seeded_tables.json")


def key(spec, seed: int) -> str:
    return f"d{spec.hidden}_N{spec.n_experts}_m{spec.ffn}_{spec.dtype}_seed{seed}_eps{spec.eps:g}"


def load(spec, seed: int):
    """(a_gsp, a_rcr) float32 for a seeded layer, or None if not stored."""
    try:
        with open(PATH) as f:
            tab = json.load(f)
    except OSError:
        return None
    ent = tab.get(key(spec, seed))
    if ent is None:
        return None
    return np.array(ent["a_gsp"], np.float32), np.array(ent["a_rcr"], np.float32)


def compute(w):
    from oracle import ace_oracle as O
    s = w.spec
    a = O.gsp_table(w.gamma, w.w_gate, w.w_up, w.w_down, s.eps).astype(np.float32)
    r = O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, s.eps).astype(np.float32)
    return a, r


def main() -> None:
    root = os.path.dirname(HERE)
    if root not in sys.path:
        sys.path.insert(0, root)
    from paper_2609_05228_gb300 import synth
    layers = [(synth.spec_qwen(), 0)] + [(synth.spec_qwen(), 100 + l) for l in range(4)] + [(synth.spec_large(), 0)]
    try:
        with open(PATH) as f:
            tab = json.load(f)
    except OSError:
        tab = {}
    for spec, seed in layers:
        k = key(spec, seed)
        if k in tab:
            continue
        t = time.time()
        w = synth.make_layer(spec, seed)
        a, r = compute(w)
        del w
        tab[k] = {"a_gsp": [float(v) for v in a], "a_rcr": [float(v) for v in r]}
        print(f"{k}: {time.time() - t:.1f} s", flush=True)
        with open(PATH, "w") as f:
            json.dump(tab, f, indent=0)


if __name__ == "__main__":
    main()
