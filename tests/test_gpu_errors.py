"""Device-side failure reporting, tested without faulting the GPU: a bounded
wait that is made to expire (the producer withholds one stage through a test
flag) returns an error status the host reads, and the context stays usable."""
import os

import pytest
import torch

from paper_2609_11133_gb300 import binding
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu


def test_expired_wait_is_reported_and_context_survives():
    c = Case(1, T=4, H=512, E=8, k=2, I=256, seed=0)
    n = binding.moe_workspace_size(c.w, 4, 2)
    ws = binding.alloc_workspace(n)
    out = torch.empty((4, 512), dtype=torch.bfloat16, device="cuda")
    binding.moe_decode_layer(c.x, c.wr, None, c.w, 2, out, ws, flags=binding._FLAG_TEST_STALL)
    torch.cuda.synchronize()
    assert binding.moe_read_status(ws) == -5  # MOE_ERR_DEVICE_TIMEOUT
    assert binding.moe_read_status(ws) == 0   # reading clears it
    # the same workspace and context still compute the layer correctly
    c.run()
    c.check_output()


def test_workspace_too_small_is_rejected():
    c = Case(1, T=4, H=512, E=8, k=2, I=256, seed=0)
    n = binding.moe_workspace_size(c.w, 4, 2)
    ws = binding.alloc_workspace(n - 256)
    out = torch.empty((4, 512), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.MoeError) as ei:
        binding.moe_decode_layer(c.x, c.wr, None, c.w, 2, out, ws[: n - 512])
    assert ei.value.status == -3
