import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: larger CPU cases")
TESTS = os.path.dirname(os.path.abspath(__file__))
if TESTS not in sys.path:
    sys.path.insert(0, TESTS)


def pytest_terminal_summary(terminalreporter):
    """Disagreement of the independent fp64 decision with the replayed fp32
    decision, per GPU parity case (reported, not asserted)."""
    try:
        import _replay
    except Exception:
        return
    rows = _replay.DISAGREEMENT
    if not rows:
        return
    slots = sum(r[1] for r in rows)
    diff = sum(r[2] for r in rows)
    terminalreporter.write_line(f"fp64-vs-replayed decision disagreement: {diff} of {slots} slots "
                                f"({diff / max(slots, 1):.2e}) over {len(rows)} forwards")
    for label, n, d, T, tok in rows:
        if d:
            terminalreporter.write_line(f"  {label}: {d} of {n} slots, {tok} of {T} tokens")
