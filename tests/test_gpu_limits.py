"""GPU parity at the limits include/moe.h states: E = 512 experts with k = 32,
H = 8192, I = 8192, and T*k = 65536 assignments - one limit per case, the
other sizes small so that the oracle finishes in seconds."""
import numpy as np
import pytest
import torch

from paper_2609_11133_gb300 import binding
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2


@pytest.mark.parametrize("fmt", [FP8, FP4])
def test_most_experts_and_largest_k(fmt):
    c = Case(fmt, T=20, H=256, E=512, k=32, I=256, seed=11).run()
    c.check_output(tokens=[0, 7, 19])


@pytest.mark.parametrize("fmt", [FP8, FP4])
def test_widest_hidden(fmt):
    c = Case(fmt, T=9, H=8192, E=6, k=2, I=256, seed=12).run()
    c.check_output()


@pytest.mark.parametrize("fmt", [FP8, FP4])
def test_widest_intermediate(fmt):
    c = Case(fmt, T=9, H=256, E=6, k=2, I=8192, seed=13).run()
    c.check_output()


@pytest.mark.parametrize("fmt", [FP8, FP4])
def test_most_assignments(fmt):
    """T*k = 65536 (T = 8192 tokens, top-8 of 16 experts): many token chunks,
    gathered activation rows, several hundred chunks per expert."""
    c = Case(fmt, T=8192, H=256, E=16, k=8, I=256, seed=14).run()
    ids = c.ids.cpu().numpy()
    assert np.bincount(ids.reshape(-1), minlength=16).sum() == 65536
    c.check_output(tokens=[0, 1, 4095, 8191])


def test_one_more_assignment_is_rejected():
    c = Case(FP8, T=8193, H=256, E=16, k=8, I=256, seed=15)
    with pytest.raises(binding.MoeError) as ei:
        binding.moe_workspace_size(c.w, 8193, 8)
    assert ei.value.status == -2  # MOE_ERR_UNSUPPORTED_SHAPE
