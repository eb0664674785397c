"""The warp-MMA expert engine (selected with MOE_ENGINE=mma; the library reads
the variable once, so each check runs in a fresh process) against the oracle,
for both weight formats, fused and with wide chunks."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys
sys.path.insert(0, {root!r})
from tests.gpu_harness import Case
FP8, FP4 = 1, 2
Case(FP4, T=8, H=4096, E=128, k=8, I=1536, seed=0).run().check_output()
Case(FP8, T=13, H=768, E=16, k=4, I=384, seed=3).run().check_output()
Case(FP4, T=77, H=1024, E=24, k=6, I=512, seed=5, residual=True).run().check_output(tokens=[0, 40, 76])
print("ENGINE_OK")
"""


def test_warp_mma_engine_matches_oracle():
    env = dict(os.environ, MOE_ENGINE="mma")
    r = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT)], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "ENGINE_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
