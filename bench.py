#!/usr/bin/env python3
"""Benchmark of the ACE MoE-layer forward (token-adaptive expert skipping) on
GB300, one process per GPU.

Default workload: the large MoE layer (hidden 4096, 256 experts, top-8,
expert FFN 2048, bf16; 12.9 GB of expert weights) prefilling 8192 tokens with
Zipf(1.1)-skewed routing at target skip ratio 0.5 (per-batch threshold,
App. B.1). A step is one full layer forward: RMSNorm, router, top-k, skip
decision, threshold, compaction, experts and combine. Inputs are synthetic
(seeded N(0,1) tokens, N(0, 0.02^2) weights) and resident in HBM; the
forward is replayed from a CUDA graph and each step is timed with CUDA
events; L2 is flushed between steps (a 512 MB write, then a 256 MB read so
dirty lines are written back), outside the timed events. The line also
carries per-point records (`points`) for the decode batches 1, 8 and 64 and
the 4096-token Zipf prefill of the hidden-2048 layer, its 4-layer stack
prefilling 16384 tokens and the large layer decoding 128 tokens.

Prints one JSON line (rank 0). `--impl reference` times the CPU oracle
instead, on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

QWEN = "d=2048 N=128 top-8 m=768 bf16"
LARGE = "d=4096 N=256 top-8 m=2048 bf16"
WORKLOADS = {
    "decode": dict(spec="qwen", zipf=False, T=64, q=0.5, layers=1, tables="offline",
                   shape=f"ACE MoE layer decode: {QWEN}"),
    "prefill": dict(spec="qwen", zipf=True, T=4096, q=0.5, layers=1, tables="offline",
                    shape=f"ACE MoE layer prefill: {QWEN}, Zipf(1.1) routing"),
    "stack_prefill": dict(spec="qwen", zipf=False, T=16384, q=0.5, layers=4, tables="offline",
                          shape=f"4-layer stack of the {QWEN} layer (residual), prefill"),
    "stack_decode": dict(spec="qwen", zipf=False, T=32, q=0.5, layers=4, tables="offline",
                         shape=f"4-layer stack of the {QWEN} layer (residual), decode"),
    "large_prefill": dict(spec="large", zipf=True, T=8192, q=0.5, layers=1, tables="gpu",
                          shape=f"large MoE layer {LARGE}, prefill, Zipf(1.1) routing"),
    # the large layer's expert shape with 32 experts (1.6 GB): a case small enough for an
    # ncu --set full capture of the large prefill's GEMMs (traffic scaled to the full layer)
    "large_prefill_e32": dict(spec="large32", zipf=True, T=1024, q=0.5, layers=1, tables="gpu",
                              shape="large MoE layer shape d=4096 top-8 m=2048 bf16 with 32 experts, prefill, "
                                    "Zipf(1.1) routing"),
    "large_decode": dict(spec="large", zipf=True, T=128, q=0.5, layers=1, tables="gpu",
                         shape=f"large MoE layer {LARGE}, decode, Zipf(1.1) routing"),
}


def wl_name(wl, T=None, q=None):
    """A workload named by what it is, with its sizes."""
    T = wl["T"] if T is None else T
    q = wl["q"] if q is None else q
    return f"{wl['shape']}, {T} tokens, skip ratio {q}"


for _wl in WORKLOADS.values():
    _wl["name"] = wl_name(_wl)
METRIC = "ACE MoE-layer tokens/s (prefill, decode) + speedup vs skip=0; % of roofline"
# The paper's own speedups (§4 efficiency, Tab. latency): whole-model TTFT and TPOT
# with and without skipping, on an A100 in bf16 at a 60% skip ratio, five
# (prompt length, batch) points from (256, 1) to (1024, 4). They measure a whole
# model, not this layer, on other hardware: context beside our speedup_vs_q0.
PAPER_SPEEDUPS = {"hardware": "NVIDIA A100, bf16, whole-model latency, skip ratio 0.6",
                  "prefill_ttft_speedup": [1.72, 2.25], "decode_tpot_speedup": [1.27, 1.41],
                  "note": "range over the paper's five (prompt, batch) points; context, not a target"}
L2_FLUSH_BYTES = 512 << 20


class L2Flush:
    """Between timed steps: write a 512 MB buffer (evicts L2), then read a
    256 MB buffer so that the dirty lines are written back before the next
    step starts. Both run outside the timed events."""

    def __init__(self, torch, device):
        self.w = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=device)
        self.r = torch.ones(L2_FLUSH_BYTES // 8, dtype=torch.float32, device=device)
        self.sink = torch.empty(1, dtype=torch.float32, device=device)

    def zero_(self):
        self.w.zero_()
        self.sink.copy_(self.r.sum().reshape(1))


# ncu summaries whose machine-read record gives roofline.traffic, per workload
TRAFFIC_RECORDS = {
    "decode": "profiles/decode_T64_q0.5_expert_decode_full.md",
    "prefill": "profiles/prefill_T4096_q0.5_expert_tc_full.md",
    "stack_prefill": "profiles/stack_prefill_T16384_q0.5_expert_pair_full.md",
    "large_prefill": "profiles/large_prefill_e32_T1024_q0.5_expert_tc_full.md",
}


def _recorded_traffic(path="profiles/decode_T64_q0.5_expert_decode_full.md", alg_bytes=None):
    """DRAM bytes per launch of the dominant kernel from a committed ncu
    summary, or None when the kernel source has changed since the capture.
    A record taken on a smaller case of the workload (it then states
    algorithmic_bytes_per_launch) is scaled by the algorithmic bytes of the
    launch being reported, `alg_bytes`."""
    import hashlib
    try:
        rec = {}
        with open(os.path.join(ROOT, path)) as f:
            for line in f:
                line = line.strip()
                if "=" in line and " " not in line.split("=", 1)[0]:
                    k, v = line.split("=", 1)
                    rec[k] = v
        h = hashlib.sha256()          # the listed sources, concatenated in order
        for src in rec["source"].split(","):
            with open(os.path.join(ROOT, src), "rb") as f:
                h.update(f.read())
        if h.hexdigest() != rec["source_sha256"]:
            return None
        if "algorithmic_bytes_per_launch" in rec:
            if alg_bytes is None:
                return None
            return int(round(int(rec["dram_bytes_per_launch"]) * alg_bytes / int(rec["algorithmic_bytes_per_launch"])))
        return int(rec["dram_bytes_per_launch"])
    except Exception:
        return None


def _peak_sustained():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops_sustained"])
    except Exception:
        return 1700.0


def clocks_rejected(clk):
    """Why a timed region's clock record disqualifies its number, or None: a
    hardware or thermal slowdown, or an SM clock held well below its maximum
    with no reason given (a clock lock left by another user). sw_power_cap
    alone is normal under a long tensor-core load and is kept."""
    if not clk:
        return None
    bad = [r for r in clk.get("reasons", []) if r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")]
    if bad:
        return "+".join(bad)
    mx = clk.get("sm_max_mhz")
    if mx and not clk.get("reasons") and clk["sm_mhz"] < 0.85 * mx:
        return "sm clock held below max with no reason"
    return None


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def smi_gpu_id(props):
    """The nvidia-smi --id of the GPU behind a CUDA device, from its device
    properties (UUID, else PCI address), never from the CUDA ordinal: under
    CUDA_VISIBLE_DEVICES the ordinal names another physical GPU in
    nvidia-smi's numbering. None when the properties carry neither."""
    u = getattr(props, "uuid", None)
    if u is not None and str(u):
        u = str(u)
        return u if u.startswith(("GPU-", "MIG-")) else "GPU-" + u
    bus = getattr(props, "pci_bus_id", None)
    if bus is not None:
        dom = getattr(props, "pci_domain_id", 0) or 0
        dev = getattr(props, "pci_device_id", 0) or 0
        return f"{int(dom):08X}:{int(bus):02X}:{int(dev):02X}.0"
    return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons of one GPU (named by UUID or PCI
    address, see smi_gpu_id) sampled every 100 ms."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.proc = None
        self.gpu = gpu_id
        if gpu_id is None:
            return
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={gpu_id}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            return None
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm), "gpu": self.gpu}


class Stack:
    """The workload's layers on one device; a step chains their forwards.
    In a stack every layer adds its input back (out = x + MoE(x))."""

    fusion = "max"     # skip rule of every forward (ace_skip_ctl.fusion); "max" is ACE

    def __init__(self, wl, max_tokens, tables=None):
        from paper_2609_05228_gb300 import ace, offline, synth
        spec = (synth.spec_qwen(zipf=wl["zipf"]) if wl["spec"] == "qwen" else
                synth.spec_large(zipf=wl["zipf"], n_experts=32 if wl["spec"] == "large32" else 256))
        self.ws, self.layers = [], []
        n = wl["layers"]
        for l in range(n):
            w = synth.make_layer(spec, seed=0 if n == 1 else 100 + l)
            if (tables or wl["tables"]) == "offline":     # host library (fp64)
                w.extra["a_gsp"], w.extra["a_rcr"] = offline.tables(w)
            else:                             # the GPU tables (ace_offline_tables_device)
                w.extra["a_gsp"], w.extra["a_rcr"] = offline.tables_device(w)
            self.ws.append(w)
            self.layers.append(ace.AceLayer(w, w.extra["a_gsp"], w.extra["a_rcr"], max_tokens=max_tokens,
                                            residual=n > 1))
            del w
        self.spec = spec
        # several layers run as one ace_stack (each next layer's RMSNorm inside the combine)
        self.stack = ace.ace_stack_create([l.handle for l in self.layers]) if n > 1 else None

    def buffers(self, torch, x):
        return [torch.empty_like(x) for _ in self.layers]

    def forward(self, x, bufs, T, q, stream=None):
        from paper_2609_05228_gb300 import ace
        if self.stack:
            ace.ace_stack_forward(self.stack, x, bufs[-1], T, "ratio", q, stream, self.fusion)
            return
        cur = x
        for layer, out in zip(self.layers, bufs):
            ace.ace_moe_forward(layer.handle, cur, out, T, "ratio", q, stream, self.fusion)
            cur = out

    def forward_host(self, xp, op, T, q):
        from paper_2609_05228_gb300 import ace
        if self.stack:
            ace.ace_stack_forward_host(self.stack, xp, op, T, "ratio", q, None, self.fusion)
        else:
            ace.ace_moe_forward_host(self.layers[0].handle, xp, op, T, "ratio", q, None, self.fusion)

    def forward_threshold(self, x, bufs, T, taus, stream=None):
        from paper_2609_05228_gb300 import ace
        cur = x
        for layer, out, tau in zip(self.layers, bufs, taus):
            ace.ace_moe_forward(layer.handle, cur, out, T, "threshold", tau, stream, self.fusion)
            cur = out

    def close(self):
        from paper_2609_05228_gb300 import ace
        if self.stack:
            ace.ace_stack_destroy(self.stack)
            self.stack = None
        for layer in self.layers:
            layer.close()


def time_point(torch, model, x, bufs, T, q, steps, warmup, flush):
    """Device time per step (ms) of a graph-replayed forward."""
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    # warm the path once eagerly (outside capture)
    with torch.cuda.stream(s):
        model.forward(x, bufs, T, q, s)
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        model.forward(x, bufs, T, q, torch.cuda.current_stream())
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    with torch.cuda.stream(s):
        for _ in range(warmup):
            flush.zero_()
            g.replay()
        s.synchronize()
        for i in range(steps):
            flush.zero_()
            starts[i].record(s)
            g.replay()
            ends[i].record(s)
    s.synchronize()
    return [a.elapsed_time(b) for a, b in zip(starts, ends)]


def time_threshold(torch, model, x, bufs, T, taus, steps, warmup, flush):
    """Device time per step (ms) of the graph-replayed forward in threshold mode."""
    s = torch.cuda.Stream()
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        model.forward_threshold(x, bufs, T, taus, s)
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        model.forward_threshold(x, bufs, T, taus, torch.cuda.current_stream())
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    with torch.cuda.stream(s):
        for _ in range(warmup):
            flush.zero_()
            g.replay()
        for i in range(steps):
            flush.zero_()
            starts[i].record(s)
            g.replay()
            ends[i].record(s)
    s.synchronize()
    return [a.elapsed_time(b) for a, b in zip(starts, ends)]


def stage_times(torch, model, x, bufs, T, q, steps, flush):
    """Per-kernel-stage device times (ms, summed over the layers) from the
    library's own CUDA events, recorded on the forward's stream inside a
    replayed CUDA graph (external event-record nodes); L2 flushed before
    every replay."""
    from paper_2609_05228_gb300 import ace
    s = torch.cuda.Stream()
    for layer in model.layers:
        ace.ace_layer_set_profiling(layer.handle, True)
    try:
        with torch.cuda.stream(s):
            model.forward(x, bufs, T, q, s)
        s.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            model.forward(x, bufs, T, q, torch.cuda.current_stream())
        out_stages = []
        with torch.cuda.stream(s):
            for i in range(steps + 2):
                flush.zero_()
                g.replay()
                per = [ace.ace_last_stage_times(layer.handle) for layer in model.layers]
                if i >= 2:
                    out_stages.append({k: sum(p[k] for p in per) for k in per[0]})
    finally:
        for layer in model.layers:
            ace.ace_layer_set_profiling(layer.handle, False)
    return out_stages


def aggregate(step_ms: float, tokens_per_rank: int, world: int, dist=None, device=None):
    """Whole-job throughput: every rank's tokens over the slowest rank's step
    time (max over ranks). Returns (tokens/s, max step ms)."""
    t = float(step_ms)
    if world > 1:
        import torch
        x = torch.tensor([t], dtype=torch.float64, device=device)
        dist.all_reduce(x, op=dist.ReduceOp.MAX)
        t = float(x.item())
    return world * tokens_per_rank / (t * 1e-3), t


def algorithmic(w, T, R, D):
    """Algorithmic bytes and flops of one forward (retained work only) and of
    the gate/up expert kernel. D = distinct experts with >= 1 retained slot."""
    s = w.spec
    d, m, N = s.hidden, s.ffn, s.n_experts
    e = 2
    w_bytes = 3 * d * m * e * D
    total_bytes = w_bytes + N * d * e + 2 * T * d * e
    flops = 6 * d * m * R + 2 * d * N * T
    gate_up_bytes = 2 * d * m * e * D + R * d * e + R * m * e
    down_bytes = d * m * e * D + R * m * e + R * d * 4      # batches <= 256: fp32 slot rows
    return total_bytes, flops, gate_up_bytes, down_bytes


def run_ours(args, rank, world, torch, dist):
    from paper_2609_05228_gb300 import ace, synth
    wl = WORKLOADS[args.workload]
    T, q = wl["T"], wl["q"]
    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    model = Stack(wl, max_tokens=max(T, 64))
    model.fusion = args.fusion
    spec, w, layer = model.spec, model.ws[0], model.layers[0]
    xh = synth.make_tokens(spec, T, seed=1 + rank)
    x = torch.from_numpy(xh.view(np.int16)).view(torch.bfloat16).to(dev)
    bufs = model.buffers(torch, x)
    flush = L2Flush(torch, dev)

    # decision statistics of the first layer's batch (R, distinct experts) and launches per step
    model.forward(x, bufs, T, q)
    launches = sum(ace.ace_last_launch_count(l.handle) for l in model.layers)
    skip, ids, gh, tau, R = ace.ace_last_skip_mask(layer.handle, T, spec.top_k)
    off, _ = ace.ace_last_permutation(layer.handle, spec.n_experts, R)
    D = int((np.diff(off) > 0).sum())

    # timed region; a region whose clock record disqualifies it (on any rank)
    # is timed once more, and the line reports the second one
    retry = None
    for attempt in range(2):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()
        clocks = ClockSampler(smi_gpu_id(torch.cuda.get_device_properties(dev)))
        t_wall = time.perf_counter()
        ms = time_point(torch, model, x, bufs, T, q, args.steps, args.warmup, flush)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t_wall
        clk = clocks.stop()
        why = clocks_rejected(clk)
        bad = why is not None
        if world > 1:
            flag = torch.tensor([1 if bad else 0], dtype=torch.int32, device=dev)
            dist.all_reduce(flag, op=dist.ReduceOp.MAX)
            bad = bool(flag.item())
            dist.barrier()
        # why the reported attempt's own clock record was rejected (any rank's), null when clean
        clock_rejected = (why or "another rank's clocks") if bad else None
        if not bad or attempt == 1:
            break
        retry = {"first_clocks": clk, "reason": why or "another rank's clocks"}
    step_ms = float(np.mean(ms))
    pct = {f"ms_p{p}": round(float(np.percentile(ms, p)), 5) for p in (10, 50, 90)}
    value, step_ms_max = aggregate(step_ms, T, world, dist, dev)

    # the dominant kernel's duration, from events on its own stream
    stages = stage_times(torch, model, x, bufs, T, q, min(args.steps, 200), flush)
    # skip ratio 0 with the same kernels, for the speedup
    ms0 = time_point(torch, model, x, bufs, T, 0.0, max(10, min(args.steps // 2, 200)), 3, flush)
    t0 = float(np.mean(ms0))

    # threshold mode with tau calibrated on a separate seed-2 batch (App. B.1 mapping)
    from paper_2609_05228_gb300 import calibrate
    xc = torch.from_numpy(synth.make_tokens(spec, T, seed=2).view(np.int16)).view(torch.bfloat16).to(dev)
    taus = [calibrate.calibrate_taus(l, xc, T, [q], fusion=args.fusion)[float(q)] for l in model.layers]
    thr_ms = time_threshold(torch, model, x, bufs, T, taus, max(10, min(args.steps // 2, 200)), 3, flush)
    model.forward_threshold(x, bufs, T, taus)
    _, _, _, _, R_thr = ace.ace_last_skip_mask(layer.handle, T, spec.top_k)
    threshold_point = {"tau_layer0": taus[0], "calibration": "seed-2 batch, ratio mode at q",
                       "realised_skip_ratio": round((T * spec.top_k - R_thr) / (T * spec.top_k), 6),
                       "ms_per_step": round(float(np.mean(thr_ms)), 5),
                       "tokens_per_s": round(T / (float(np.mean(thr_ms)) * 1e-3), 1)}

    # Zipf check: log-log slope of the sorted routed (top-k) slot counts over ranks 1..N/2
    zipf_slope = None
    if wl["zipf"]:
        model.forward(x, bufs, T, q)
        _, ids_r, _, _, _ = ace.ace_last_skip_mask(layer.handle, T, spec.top_k)
        cnt = np.sort(np.bincount(ids_r.ravel(), minlength=spec.n_experts))[::-1][: spec.n_experts // 2]
        ranks = np.arange(1, cnt.size + 1)
        ok = cnt > 0
        zipf_slope = round(float(np.polyfit(np.log(ranks[ok]), np.log(cnt[ok]), 1)[0]), 3)

    # end to end through the host-buffer C call (pinned buffers, copies included:
    # ace_moe_forward_host for one layer, ace_stack_forward_host for a stack)
    xp = torch.from_numpy(xh.view(np.int16)).pin_memory()
    op = torch.empty_like(xp).pin_memory()
    for _ in range(3):
        model.forward_host(xp, op, T, q)
    e2e_steps = max(10, min(args.steps, 300))
    t = time.perf_counter()
    for _ in range(e2e_steps):
        model.forward_host(xp, op, T, q)
    e2e_s = (time.perf_counter() - t) / e2e_steps

    hbm, bf16, peak_kind = _peaks()
    bf16_sust = _peak_sustained()
    n_layers = len(model.layers)
    total_bytes, flops, gu_bytes, down_bytes = algorithmic(w, T, R, D)
    gu_flops = 4 * spec.hidden * spec.ffn * R
    # the "gate_up" stage: batches <= 256 run both GEMMs in one launch (k_expert_decode)
    gu_ms = float(np.mean([st["gate_up"] for st in stages])) / n_layers if stages else float("nan")
    stage_avg = {k: round(float(np.mean([st[k] for st in stages])) * 1e3, 2) for k in stages[0]} if stages else {}
    tensor_bound = R / max(D, 1) > 280           # tokens per expert above the ridge (FLOP/B)
    pair = T > 256 and T * spec.top_k * (1.0 - q) >= 256 * spec.n_experts   # the library's CTA-pair rule
    if tensor_bound:
        achieved = gu_flops / (gu_ms * 1e-3) / 1e12
        kname = "k_expert_pair gate/up (tcgen05 cta_group::2)" if pair else "k_expert_tc gate/up (tcgen05)"
        roof = {"bound": "tensor", "kernel": kname, "achieved": round(achieved, 1),
                "peak": bf16_sust, "unit": "TFLOP/s", "frac": round(achieved / bf16_sust, 4),
                "peak_source": peak_kind + " (sustained bf16)",
                "traffic": _recorded_traffic(TRAFFIC_RECORDS[args.workload]) if args.workload in TRAFFIC_RECORDS else None,
                "algorithmic_flops": gu_flops, "kernel_us": round(gu_ms * 1e3, 2)}
    elif T <= 256:
        kb = gu_bytes + down_bytes
        achieved = kb / (gu_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "kernel": "k_expert_decode gate/up + down (tcgen05, one launch)",
                "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "peak_source": peak_kind,
                "traffic": _recorded_traffic(TRAFFIC_RECORDS[args.workload]) if args.workload in TRAFFIC_RECORDS else None,
                "algorithmic_bytes": kb, "kernel_us": round(gu_ms * 1e3, 2)}
    else:
        achieved = gu_bytes / (gu_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "kernel": "k_expert_tc gate/up (tcgen05)",
                "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s", "frac": round(achieved / hbm, 4),
                "peak_source": peak_kind,
                "traffic": _recorded_traffic(TRAFFIC_RECORDS[args.workload], gu_bytes)
                if args.workload in TRAFFIC_RECORDS else None,
                "algorithmic_bytes": gu_bytes, "kernel_us": round(gu_ms * 1e3, 2)}

    result = {
        "metric": METRIC,
        "value": round(value, 1),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(step_ms_max, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) tokens, N(0,0.02^2) weights, " +
                ("offline GSP/RCR tables from the host library)" if wl["tables"] == "offline"
                 else "offline GSP/RCR tables computed on the GPU)"),
        "config": {"workload": wl["name"], "tokens_per_step": T, "layers": n_layers, "skip_ratio": q,
                   "skip_rule": args.fusion,
                   "parallelism": f"replicas{world}" if world > 1 else "single GPU",
                   "l2": "flushed between timed steps (512 MB write, then a 256 MB read)", "graph": "CUDA graph replay"},
        "realised_skip_ratio": round((T * spec.top_k - R) / (T * spec.top_k), 6),
        "retained_slots": R,
        "distinct_experts": D,
        **pct,
        "speedup_vs_q0": round(t0 / step_ms, 4),
        "paper_speedups": PAPER_SPEEDUPS,
        "threshold_mode": threshold_point,
        "zipf_slope": zipf_slope,
        "q0_ms_per_step": round(t0, 5),
        "stage_us": stage_avg,
        "wall_s": round(wall, 3),
        "roofline": roof,
        "layer_roofline": {"bytes": total_bytes * n_layers, "flops": flops * n_layers,
                           "hbm_frac": round(total_bytes * n_layers / (step_ms * 1e-3) / 1e9 / hbm, 4),
                           "tensor_frac": round(flops * n_layers / (step_ms * 1e-3) / 1e12 / bf16_sust, 5)},
        "e2e": {"value": round(T / e2e_s, 1), "unit": "tokens/s",
                "h2d_bytes_per_step": int(T * spec.hidden * 2),
                "d2h_bytes_per_step": int(T * spec.hidden * 2)},
        "gpu_launches": args.steps * launches,
        "clocks": clk,
        "clock_retry": retry,
        "clock_rejected": clock_rejected,
        "offline_tables": time_tables(torch, w) if rank == 0 else None,
    }
    if rank == 0 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(model.ws, wl, budget_s=args.cpu_seconds, fusion=args.fusion)
    if rank == 0 and not args.no_points:
        result["points"] = measure_points(torch, args, {"large_decode": model} if args.workload == "large_prefill"
                                          else None)
    if rank == 0 and args.sweep:
        result["sweep"] = sweep(torch, args)
    model.close()
    return result


# Per-point records of the default run: the other batch sizes and workloads
# (tokens/s, retained slots R, distinct retained experts D, fractions of the
# binding roofline, speedup over the same kernels at skip ratio 0).
POINTS = [("decode", 1), ("decode", 8), ("decode", 64), ("prefill", 4096), ("stack_prefill", 16384),
          ("large_decode", 128)]


def layer_roofline(spec, T, R, D, n_layers=1):
    """Algorithmic bytes and FLOPs of a forward (retained work only), summed
    over layers: B = 6 d m D + 2 d N + 4 d T per layer (bf16 weights of the
    distinct retained experts, the router, tokens in and out), F = 6 d m R +
    2 d N T. R and D are lists (one entry per layer)."""
    d, m, N = spec.hidden, spec.ffn, spec.n_experts
    B = sum(6 * d * m * Dl + 2 * d * N + 4 * d * T for Dl in D)
    F = sum(6 * d * m * Rl + 2 * d * N * T for Rl in R)
    return B, F


def roofline_point(spec, T, R, D, ms, hbm_gbs, tensor_tflops):
    """Fractions of the HBM and tensor rooflines for one step of `ms` ms, and
    of t* = max(B / BW, F / P), the binding one."""
    B, F = layer_roofline(spec, T, R, D)
    t_hbm = B / (hbm_gbs * 1e9)
    t_tc = F / (tensor_tflops * 1e12)
    t = ms * 1e-3
    tstar = max(t_hbm, t_tc)
    return {"bytes": B, "flops": F, "bound": "hbm" if t_hbm >= t_tc else "tensor",
            "tstar_us": round(tstar * 1e6, 2), "frac_of_tstar": round(tstar / t, 4),
            "hbm_frac": round(t_hbm / t, 4), "tensor_frac": round(t_tc / t, 4)}


def decision_stats(model, T):
    """Retained slots and distinct retained experts of each layer's last forward."""
    from paper_2609_05228_gb300 import ace
    spec = model.spec
    R, D = [], []
    for layer in model.layers:
        _, _, _, _, r = ace.ace_last_skip_mask(layer.handle, T, spec.top_k)
        off, _ = ace.ace_last_permutation(layer.handle, spec.n_experts, r)
        R.append(int(r))
        D.append(int((np.diff(off) > 0).sum()))
    return R, D


def measure_points(torch, args, models=None):
    """The POINTS at skip ratio 0.5 and 0, each timed as in the main line
    (graph replay, L2 flushed between steps, median of the replays). Layers are
    built per workload and freed after it (the GPU tables, as the large layer
    uses); `models` maps a workload to a Stack that is already built."""
    from paper_2609_05228_gb300 import synth
    hbm, _, _ = _peaks()
    sust = _peak_sustained()
    flush = L2Flush(torch, "cuda")
    groups = {}
    for wl, T in POINTS:
        groups.setdefault(wl, []).append(T)
    out = []
    for wl, Ts in groups.items():
        own = not (models and wl in models)
        model = Stack(WORKLOADS[wl], max_tokens=max(Ts), tables="gpu") if own else models[wl]
        model.fusion = args.fusion
        q = WORKLOADS[wl]["q"]
        for T in Ts:
            xh = synth.make_tokens(model.spec, T, seed=1)
            x = torch.from_numpy(xh.view(np.int16)).view(torch.bfloat16).cuda()
            bufs = model.buffers(torch, x)
            ms = float(np.median(time_point(torch, model, x, bufs, T, q, 30, 3, flush)))
            model.forward(x, bufs, T, q)
            R, D = decision_stats(model, T)
            ms0 = float(np.median(time_point(torch, model, x, bufs, T, 0.0, 15, 3, flush)))
            rec = {"workload": wl_name(WORKLOADS[wl], T), "tokens": T, "layers": len(model.layers), "skip_ratio": q,
                   "tokens_per_s": round(T / (ms * 1e-3), 1), "us_per_step": round(ms * 1e3, 2),
                   "retained_slots": R, "distinct_experts": D,
                   "speedup_vs_q0": round(ms0 / ms, 4), "q0_us_per_step": round(ms0 * 1e3, 2)}
            rec.update(roofline_point(model.spec, T, R, D, ms, hbm, sust))
            out.append(rec)
            del x, bufs
        if own:
            model.close()
            del model
            torch.cuda.empty_cache()
    return out


def sweep(torch, args):
    """Tokens/s and speedup vs q=0 over the configurations' batch sizes and
    skip ratios: the d=2048 layer (decode batches, 4096-token prefill), or the
    large layer (decode 1/16/128, prefill 2048/8192; q from 0 to 0.625 in
    steps of 0.125) when the workload is a large-layer one. Each point also
    carries its retained slots, distinct retained experts and roofline
    fractions, as the main line's points do."""
    from paper_2609_05228_gb300 import synth
    hbm, _, _ = _peaks()
    sust = _peak_sustained()
    if args.workload.startswith("large"):
        qs = [0.0, 0.125, 0.25, 0.375, 0.5, 0.625]
        plan = [("large_prefill", [1, 16, 128, 2048, 8192], qs)]
    else:
        plan = [("decode", [1, 8, 32, 64], [0.0, 0.25, 0.5]),
                ("prefill", [4096], [0.0, 0.25, 0.5, 0.625])]
    pts = []
    for wlname, Ts, qs in plan:
        model = Stack(WORKLOADS[wlname], max_tokens=max(Ts))
        model.fusion = args.fusion
        flush = L2Flush(torch, "cuda")
        for T in Ts:
            xh = synth.make_tokens(model.spec, T, seed=1)
            x = torch.from_numpy(xh.view(np.int16)).view(torch.bfloat16).cuda()
            bufs = model.buffers(torch, x)
            base = None
            for q in qs:
                ms = time_point(torch, model, x, bufs, T, q, 20, 3, flush)
                t = float(np.median(ms))
                base = t if q == 0.0 else base
                model.forward(x, bufs, T, q)
                R, D = decision_stats(model, T)
                rec = {"workload": wlname, "T": T, "q": q, "us": round(t * 1e3, 2),
                       "tokens_per_s": round(T / (t * 1e-3), 1),
                       "speedup_vs_q0": round(base / t, 4) if base else None,
                       "retained_slots": R, "distinct_experts": D}
                rec.update(roofline_point(model.spec, T, R, D, t, hbm, sust))
                pts.append(rec)
        model.close()
    return pts


def time_tables(torch, w, reps=3):
    """Wall time of ace_offline_tables_device (Algorithms 2 and 3 on the GPU)
    for layer `w`, weights resident on the device; the call allocates its
    scratch, packs, runs and synchronises. GSP GEMM FLOPs: two d x d x m
    products per expert."""
    from paper_2609_05228_gb300 import ace
    spec = w.spec
    d, n, m = spec.hidden, spec.n_experts, spec.ffn

    def up(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).cuda()

    ts = [up(a) for a in (w.gamma, w.router_w, w.w_gate, w.w_up, w.w_down)]
    torch.cuda.synchronize()
    ace.ace_offline_tables_device(d, n, m, *ts, spec.eps)
    times = []
    for _ in range(reps):
        t = time.perf_counter()
        ace.ace_offline_tables_device(d, n, m, *ts, spec.eps)
        times.append(time.perf_counter() - t)
    del ts
    torch.cuda.empty_cache()
    t = float(np.median(times))
    flops = 2 * 2 * d * d * m * n
    return {"call_ms": round(t * 1e3, 3), "gsp_gemm_tflop": round(flops / 1e12, 4),
            "gsp_gemm_tflops_over_call": round(flops / t / 1e12, 1),
            "note": "whole call: scratch allocation, packing, GSP GEMM, norms, RCR GEMV, normalisation"}


def cpu_baseline(ws, wl, budget_s=12.0, fusion="max"):
    """The CPU oracle (fp64) on a bounded sample of the same workload: the
    stacked layers over a sample of tokens (64, or 256 for prefill)."""
    import oracle as O
    from paper_2609_05228_gb300 import synth
    T = wl["T"] if wl["T"] <= 64 else 256
    x = synth.make_tokens(ws[0].spec, T, seed=1)
    n = 0
    t0 = time.perf_counter()
    while True:
        cur = O.to_f64(x)
        for i, w in enumerate(ws):
            y = O.moe_forward(cur, w, "ratio", wl["q"], fusion=fusion)
            cur = cur + y if len(ws) > 1 else y
        n += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    return {"value": round(n * T / dt, 2), "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} forwards of {T} tokens through {len(ws)} layer(s) ({dt:.1f} s), numpy fp64 "
                      "with its default BLAS threads"}


def run_reference(args):
    """The reference arm: the CPU oracle on a bounded sample, per step."""
    import oracle as O
    from oracle import seeded_tables
    from paper_2609_05228_gb300 import synth
    wl = WORKLOADS[args.workload]
    spec = synth.spec_qwen(zipf=wl["zipf"]) if wl["spec"] == "qwen" else synth.spec_large(zipf=wl["zipf"])
    ws = []
    for l in range(wl["layers"]):
        seed = 0 if wl["layers"] == 1 else 100 + l
        w = synth.make_layer(spec, seed=seed)
        # the oracle's own tables (Algorithms 2 and 3): stored by oracle/seeded_tables.py, else computed here
        tabs = seeded_tables.load(spec, seed)
        w.extra["a_gsp"], w.extra["a_rcr"] = tabs if tabs is not None else seeded_tables.compute(w)
        ws.append(w)
    xall = synth.make_tokens(spec, min(wl["T"], 256), seed=1)

    def step(T):
        cur = O.to_f64(xall[:T])
        for w in ws:
            y = O.moe_forward(cur, w, "ratio", wl["q"], fusion=args.fusion)
            cur = cur + y if len(ws) > 1 else y

    # tokens per step: the whole run (warm-up + steps) is sized to about two
    # minutes of oracle time, from a one-step rate estimate on 8 tokens
    t = time.perf_counter()
    step(min(8, xall.shape[0]))
    rate = min(8, xall.shape[0]) / (time.perf_counter() - t)
    T = int(max(1, min(xall.shape[0], rate * 120.0 / (args.steps + args.warmup))))
    for _ in range(args.warmup):
        step(T)
    times = []
    for _ in range(args.steps):
        t = time.perf_counter()
        step(T)
        times.append(time.perf_counter() - t)
    st = float(np.mean(times))
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    val = round(T / st, 2)
    return {"impl": "reference", "metric": METRIC, "value": val, "unit": "tokens/s", "n_gpus": 1,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(st * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl["name"], "tokens_per_step": T, "layers": len(ws),
                                            "skip_ratio": wl["q"], "skip_rule": args.fusion,
                                            "sample": f"{T} tokens per step"},
            "cpu_baseline": {"value": val, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": f"{args.steps} steps of {T} tokens"},
            "e2e": {"value": val, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="large_prefill", choices=sorted(WORKLOADS))
    ap.add_argument("--no-points", action="store_true",
                    help="skip the per-point records (other batch sizes and workloads) of the default run")
    ap.add_argument("--sweep", action="store_true", help="add decode/prefill sweep points")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--fusion", default="max", choices=["max", "min", "mean", "gsp", "rcr", "score"],
                    help="skip rule (max = ACE; the others are the paper's ablation variants and router-score skipping)")
    ap.add_argument("--tables-only", action="store_true",
                    help="time only the GPU offline tables (ace_offline_tables_device) of the workload's layer")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))

    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return

    import torch
    import torch.distributed as dist
    if args.tables_only:
        if rank == 0:
            from paper_2609_05228_gb300 import synth
            wl = WORKLOADS[args.workload]
            spec = (synth.spec_qwen(zipf=wl["zipf"]) if wl["spec"] == "qwen" else
                synth.spec_large(zipf=wl["zipf"], n_experts=32 if wl["spec"] == "large32" else 256))
            w = synth.make_layer(spec, seed=0)
            print(json.dumps({"workload": wl["name"], "offline_tables": time_tables(torch, w, reps=args.steps)}),
                  flush=True)
        return
    if world > 1:
        dist.init_process_group("nccl")
    try:
        res = run_ours(args, rank, world, torch, dist)
        if rank == 0:
            print(json.dumps(res), flush=True)
    finally:
        if world > 1:
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
