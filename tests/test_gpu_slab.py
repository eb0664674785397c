"""GPU tests of the FP8 engine's slab order: in a step whose whole items would not keep their
weight tiles in L2, an expert with several token chunks runs every chunk over one slab of
K-blocks before the next slab, and each chunk's partial sums are added out at the end of its
run in a slab.  Each case routes Zipf-hot experts of several chunks and compares every token
with the oracle, with the default slab length and (in subprocesses, MOE_F8_SLAB) with lengths
that do and do not divide the step's K-blocks."""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2609_11133_gb300 import synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP8 = 1
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

# (T, H, E, k, I) on a GB300 (152 SMs, ~126 MB of L2): H = 6144 puts the gate/up step in slab
# order (48 K-blocks: 152 CTAs' whole tiles 239 MB), I = 4096 the down step (32 K-blocks:
# 159 MB), the other step of each shape keeps whole items; batches above 64 tokens run in
# gathered 32-token chunks, the only chunk width with slab order
SHAPES = [(120, 6144, 32, 4, 256), (200, 6144, 32, 4, 256), (120, 256, 32, 4, 4096),
          (200, 256, 32, 4, 4096)]


def _case(T, H, E, k, I, seed):
    bias = synth.make_zipf_bias(E, H, s=1.1, seed=seed)
    return Case(FP8, T=T, H=H, E=E, k=k, I=I, seed=seed, bias=bias, residual=True)


@pytest.mark.parametrize("T,H,E,k,I", SHAPES)
def test_hot_experts_in_slab_order(T, H, E, k, I):
    c = _case(T, H, E, k, I, seed=60 + T + H).run()
    n = np.bincount(c.ids.cpu().numpy().reshape(-1), minlength=E)
    assert (n > 2 * 32).sum() >= 2  # hot experts of three chunks or more
    c.check_output(row_tol=2e-2)


SCRIPT = r"""
import sys
sys.path.insert(0, {root!r})
from paper_2609_11133_gb300 import synth
from tests.gpu_harness import Case
for T, H, E, k, I in {shapes!r}:
    bias = synth.make_zipf_bias(E, H, s=1.1, seed=70 + T + H)
    c = Case(1, T=T, H=H, E=E, k=k, I=I, seed=70 + T + H, bias=bias, residual=True).run()
    c.check_output(row_tol=2e-2)
print("SLAB_OK")
"""


@pytest.mark.parametrize("slab", ["0", "1", "5", "40"])
def test_other_slab_lengths(slab):
    """0: whole items; 1: every chunk one K-block at a time; 5: slabs dividing neither 48 nor
    32; 40: one slab of 40 and one of 8 in the gate/up step, one slab of all 32 in the down
    step (whole items)."""
    env = dict(os.environ, MOE_F8_SLAB=slab)
    r = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT, shapes=SHAPES)], env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0 and "SLAB_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
