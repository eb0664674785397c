import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def pytest_terminal_summary(terminalreporter):
    """Per-row output errors of the GPU parity checks: for every check, the
    global figure of the contract (max|gpu - ref| / max|ref| over the output)
    and the worst row (max over h of |gpu - ref| / max over h of |ref|)."""
    mod = sys.modules.get("tests.gpu_harness")
    rep = getattr(mod, "REPORT", None)
    if not rep:
        return
    tw = terminalreporter
    tw.write_line(f"parity checks: {len(rep)}, rows compared: {sum(r[3] for r in rep)}")
    g = max(rep, key=lambda r: r[4])
    w = max(rep, key=lambda r: r[5])
    tw.write_line(f"worst global error {g[4]:.2e} ({g[0]}); worst row error {w[5]:.2e} ({w[0]})")
    for r in rep:
        if "ties" in r[0] or "heavy" in r[0] or "full_batch" in r[0]:
            tw.write_line(f"  {r[0].split('::')[-1]}: fmt {r[1]} T={r[2]} rows={r[3]} "
                          f"global {r[4]:.2e} worst row {r[5]:.2e}")
