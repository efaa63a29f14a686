"""Host-side pieces of bench.py that need no GPU: the reference arm's JSON
line (the oracle on a bounded sample), the ncu traffic record guard, and the
algorithmic byte counts of the roofline."""
import json
import os
import re
import shutil
import subprocess
import sys

import numpy as np

import bench
from paper_2609_05228_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_recorded_traffic_follows_the_kernel_sources(tmp_path, monkeypatch):
    """A record gives its DRAM bytes only while the hash of its listed sources
    matches; a stale hash, a missing file or a missing source gives None."""
    import hashlib
    srcs = ("ace_expert_tc.cu", "ace_tc.cuh", "ace_device.cuh")
    os.makedirs(tmp_path / "paper_2609_05228_gb300" / "csrc", exist_ok=True)
    h = hashlib.sha256()
    for src in srcs:
        path = os.path.join(ROOT, "paper_2609_05228_gb300", "csrc", src)
        shutil.copy(path, tmp_path / "paper_2609_05228_gb300" / "csrc" / src)
        h.update(open(path, "rb").read())
    listed = ",".join("paper_2609_05228_gb300/csrc/" + s for s in srcs)
    record = ("Machine-read record:\n\n"
              "    kernel=k_expert_decode\n"
              f"    source={listed}\n"
              f"    source_sha256={h.hexdigest()}\n"
              "    dram_bytes_per_launch=1044777984\n")
    (tmp_path / "good.md").write_text(record)
    (tmp_path / "bad.md").write_text(record.replace("source_sha256=", "source_sha256=0"))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._recorded_traffic("good.md") == 1044777984
    assert bench._recorded_traffic("bad.md") is None
    assert bench._recorded_traffic("missing.md") is None
    os.remove(tmp_path / "paper_2609_05228_gb300" / "csrc" / "ace_tc.cuh")
    assert bench._recorded_traffic("good.md") is None
    # every committed record names the files it hashes, and those files exist
    monkeypatch.setattr(bench, "ROOT", ROOT)
    for rec in bench.TRAFFIC_RECORDS.values():
        text = open(os.path.join(ROOT, rec)).read()
        listed = re.search(r"source=(\S+)", text).group(1).split(",")
        assert all(os.path.exists(os.path.join(ROOT, s)) for s in listed)
        assert re.search(r"dram_bytes_per_launch=\d+", text)


def test_clock_records_that_disqualify_a_timed_region():
    ok = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 17}
    capped = {"sm_mhz": 1850.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 30}
    assert bench.clocks_rejected(ok) is None
    assert bench.clocks_rejected(capped) is None          # power cap under load is kept
    assert bench.clocks_rejected(None) is None            # no nvidia-smi: nothing to reject
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert r in bench.clocks_rejected(dict(ok, reasons=[r, "sw_power_cap"]))
    locked = dict(ok, sm_mhz=1200.0)                      # held low with no reason: a clock lock
    assert bench.clocks_rejected(locked) is not None
    assert bench.clocks_rejected(dict(locked, reasons=["sw_power_cap"])) is None


def test_algorithmic_bytes_of_the_decode_layer():
    """Retained-expert weight bytes: 3 matrices of d x m bf16 per distinct expert."""
    w = synth.LayerWeights(synth.spec_qwen(), None, None, None, None, None, None)
    d, m, N = 2048, 768, 128
    total, flops, gu, down = bench.algorithmic(w, 64, 256, 110)
    assert total == 3 * d * m * 2 * 110 + N * d * 2 + 2 * 64 * d * 2
    assert flops == 6 * d * m * 256 + 2 * d * N * 64
    assert gu == 2 * d * m * 2 * 110 + 256 * d * 2 + 256 * m * 2
    assert down == d * m * 2 * 110 + 256 * m * 2 + 256 * d * 4


def test_reference_arm_json_line():
    """`bench.py --impl reference` prints one JSON line with the contract's
    keys, timing the oracle on the host (tokens per step sized to the steps)."""
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "decode",
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, cwd=ROOT, timeout=900)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "tokens/s" and d["value"] > 0
    assert d["steps"] == 2 and d["warmup"] >= 3 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert 1 <= d["config"]["tokens_per_step"] <= 64
    assert "libace" not in r.stderr


def test_smi_gpu_id_names_the_device_not_the_ordinal():
    """nvidia-smi is pointed at the GPU by UUID (else PCI address) from the
    device's properties; the CUDA ordinal is never used."""
    class P:
        uuid = "1a2b3c4d-0000-1111-2222-333344445555"
        pci_bus_id, pci_domain_id, pci_device_id = 0x41, 0, 0
    assert bench.smi_gpu_id(P()) == "GPU-1a2b3c4d-0000-1111-2222-333344445555"

    class Q:
        pci_bus_id, pci_domain_id, pci_device_id = 0x41, 2, 0
    assert bench.smi_gpu_id(Q()) == "00000002:41:00.0"
    assert bench.smi_gpu_id(object()) is None
    assert bench.ClockSampler(None).stop() is None        # unknown GPU: no samples rather than another GPU's


def test_reference_arm_reads_oracle_tables_only():
    """The reference arm's tables are the oracle's (Algorithms 2 and 3), stored
    by oracle/seeded_tables.py for every benchmark layer: check one stored
    entry against a fresh oracle computation on a subset of experts."""
    import oracle as O
    from oracle import seeded_tables
    spec = synth.spec_qwen()
    for seed in (0, 100, 101, 102, 103):
        assert seeded_tables.load(spec, seed) is not None, seed
    assert seeded_tables.load(synth.spec_large(), 0) is not None
    a, r = seeded_tables.load(spec, 0)
    w = synth.make_layer(spec, seed=0)
    # the normalisation is one constant per table, so ratios of entries are those of the raw scores
    idx = [0, 5, 77]
    sub = O.gsp_table(w.gamma, w.w_gate[idx], w.w_up[idx], w.w_down[idx], 0.0)
    np.testing.assert_allclose(a[idx] / a[idx[0]], sub / sub[0], rtol=1e-6)
    r_full = O.rcr_table(w.router_w, w.gamma, w.w_gate, w.w_up, w.w_down, spec.eps)
    np.testing.assert_allclose(r, r_full.astype(np.float32), rtol=1e-6)
