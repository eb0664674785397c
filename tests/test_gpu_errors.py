"""Device-side failure reporting, tested without faulting the GPU: a bounded
wait that is made to expire (the producer withholds one stage through a test
flag) returns an error status the host reads, and the context stays usable.
Each engine has its own waits and its own wind-down (tensor memory freed,
copies in flight drained), so each is made to time out: the FP8 and NVFP4
tensor-core engines in this process (1 s limit), and all three engines in a
subprocess with a 50 ms limit (MOE_WAIT_LIMIT_MS is read once per process)."""
import os
import subprocess
import sys

import pytest
import torch

from paper_2609_11133_gb300 import binding
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def stall_then_recover(fmt, T, H, E, k, I, seed):
    """A layer call whose first gate/up stage never arrives: the status word
    reports the expired wait, reading clears it, and after moe_workspace_init
    the same workspace computes the layer within tolerance of the oracle."""
    c = Case(fmt, T=T, H=H, E=E, k=k, I=I, seed=seed)
    ws = binding.alloc_workspace(binding.moe_workspace_size(c.w, T, k))
    out = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    binding.moe_decode_layer(c.x, c.wr, None, c.w, k, out, ws, flags=binding._FLAG_TEST_STALL)
    torch.cuda.synchronize()
    assert binding.moe_read_status(ws) == -5  # MOE_ERR_DEVICE_TIMEOUT
    assert binding.moe_read_status(ws) == 0   # reading clears it
    binding.moe_workspace_init(ws)
    c.run(out=out, ws=ws)
    c.check_output()


@pytest.mark.parametrize("fmt,T,H,E,k,I", [(1, 4, 512, 8, 2, 256), (2, 8, 1024, 16, 4, 512),
                                           (2, 72, 1024, 16, 4, 512)])
def test_expired_wait_is_reported_and_context_survives(fmt, T, H, E, k, I):
    """FP8 engine (T=4) and the NVFP4 block-scaled engine (T=8, and T=72 with
    the gathered activation rows and 16-token chunks)."""
    stall_then_recover(fmt, T, H, E, k, I, seed=T)


SCRIPT = r"""
import sys
sys.path.insert(0, {root!r})
from tests.test_gpu_errors import stall_then_recover
stall_then_recover(1, 4, 512, 8, 2, 256, seed=1)
stall_then_recover(2, 8, 1024, 16, 4, 512, seed=2)
print("STALL_OK")
"""


@pytest.mark.parametrize("engine", ["mma", "tensor"])
def test_expired_wait_with_a_short_limit_in_each_engine(engine):
    env = dict(os.environ, MOE_WAIT_LIMIT_MS="50")
    if engine == "mma":
        env["MOE_ENGINE"] = "mma"
    r = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT)], env=env,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "STALL_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]


def test_workspace_too_small_is_rejected():
    c = Case(1, T=4, H=512, E=8, k=2, I=256, seed=0)
    n = binding.moe_workspace_size(c.w, 4, 2)
    ws = binding.alloc_workspace(n - 256)
    out = torch.empty((4, 512), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.MoeError) as ei:
        binding.moe_decode_layer(c.x, c.wr, None, c.w, 2, out, ws[: n - 512])
    assert ei.value.status == -3
