"""moe_decode_layer_noalloc: the fused layer for callers that must not allocate
device memory while they run it (an engine plugin's enqueue path, which is
handed a stream and tensors but no allocator; a serving loop that cannot
afford a cudaMalloc that may synchronise the device).  It runs on the
library's own 16 MiB scratch array.

The tests check it against the workspace-taking moe_decode_layer and against
the oracle on two calls in a row (the second call reuses the array the first
one left behind), at the largest batch whose workspace fits the array (found
from moe_workspace_size) and one token beyond it, and after a call whose
bounded wait expired (read through moe_noalloc_read_status).  This file is
collected last, so a run that stops at the first failure has run every other
test by then; it also passes on its own in a fresh process."""
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

REL_TOL = 2e-2  # the output tolerance of the other layer tests
SCRATCH_BYTES = 16 << 20  # the array's size, as moe.h states it


def _inputs(fmt, T, H, E, k, I, seed):
    w = synth.make_weights(fmt, E, H, I, seed=seed, device="cuda")
    x = synth.make_x(T, H, seed=seed, device="cuda")
    wr = synth.make_router(E, H, seed=seed, device="cuda")
    return w, x, wr


@pytest.mark.parametrize("fmt,T,H,E,k,I", [(2, 8, 4096, 128, 8, 1536), (1, 13, 768, 16, 4, 384)])
def test_noalloc_matches_workspace_layer_on_consecutive_calls(fmt, T, H, E, k, I):
    c = Case(fmt, T=T, H=H, E=E, k=k, I=I, seed=7).run()
    c.check_output()  # the workspace layer against the oracle
    ref = c.out.clone()
    scale = ref.float().abs().max().item()
    for _ in range(2):
        out = torch.full((T, H), float("nan"), dtype=torch.bfloat16, device="cuda")
        binding.moe_decode_layer_noalloc(c.x, c.wr, None, c.w, k, out)
        torch.cuda.synchronize()
        assert binding.moe_noalloc_read_status() == 0
        assert torch.isfinite(out.float()).all()
        assert (out.float() - ref.float()).abs().max().item() <= REL_TOL * scale
        c.out = out
        c.check_output()  # and against the oracle (same routing, checked bit-exactly)


def test_noalloc_with_residual_after_a_different_shape():
    """A call with another shape in between leaves nothing that disturbs the next."""
    w, x, wr = _inputs(1, 5, 512, 8, 2, 256, seed=3)
    res = synth.make_x(5, 512, seed=4, device="cuda")
    ref = torch.empty((5, 512), dtype=torch.bfloat16, device="cuda")
    ws = binding.alloc_workspace(binding.moe_workspace_size(w, 5, 2))
    binding.moe_decode_layer(x, wr, None, w, 2, ref, ws, residual=res)
    w2, x2, wr2 = _inputs(2, 21, 1024, 12, 3, 512, seed=5)
    out2 = torch.empty((21, 1024), dtype=torch.bfloat16, device="cuda")
    binding.moe_decode_layer_noalloc(x2, wr2, None, w2, 3, out2)
    out = torch.empty_like(ref)
    binding.moe_decode_layer_noalloc(x, wr, None, w, 2, out, residual=res)
    torch.cuda.synchronize()
    assert binding.moe_noalloc_read_status() == 0
    assert (out.float() - ref.float()).abs().max().item() <= REL_TOL * ref.float().abs().max().item()


@pytest.fixture(scope="module")
def layer_235b():
    w = synth.make_weights(2, 128, 4096, 1536, seed=0, device="cuda")
    wr = synth.make_router(128, 4096, seed=0, device="cuda")
    yield w, wr
    del w
    torch.cuda.empty_cache()


def largest_batch_that_fits(w, k):
    T = 1
    while binding.moe_workspace_size(w, T + 1, k) <= SCRATCH_BYTES:
        T += 1
    return T


def test_noalloc_at_the_largest_batch_that_fits(layer_235b):
    """The 235B-shaped NVFP4 layer at the last T whose workspace fits the
    array (74 tokens), against the workspace layer and the oracle."""
    w, wr = layer_235b
    k = 8
    T = largest_batch_that_fits(w, k)
    assert T >= 64
    x = synth.make_x(T, 4096, seed=11, device="cuda")
    c = Case(2, T=T, H=4096, E=128, k=k, I=1536, w=w, wr=wr, x=x).run()
    ref = c.out.clone()
    for _ in range(2):
        out = torch.empty_like(ref)
        binding.moe_decode_layer_noalloc(x, wr, None, w, k, out)
        torch.cuda.synchronize()
        assert binding.moe_noalloc_read_status() == 0
        assert (out.float() - ref.float()).abs().max().item() <= \
            REL_TOL * ref.float().abs().max().item()
    c.out = out
    c.check_output(tokens=[0, T // 2, T - 1])


def test_noalloc_rejects_one_token_beyond_its_scratch(layer_235b):
    w, wr = layer_235b
    k = 8
    T = largest_batch_that_fits(w, k) + 1
    x = torch.zeros((T, 4096), dtype=torch.bfloat16, device="cuda")
    out = torch.empty((T, 4096), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.MoeError) as ei:
        binding.moe_decode_layer_noalloc(x, wr, None, w, k, out)
    assert ei.value.status == -3  # MOE_ERR_WORKSPACE_TOO_SMALL


@pytest.mark.parametrize("fmt", [1, 2])
def test_noalloc_reports_an_expired_wait_and_recovers(fmt):
    """The test flag makes the first gate/up stage never arrive: the bounded
    wait expires, moe_noalloc_read_status reports it once, and the next call
    on the same array matches the oracle (each call clears its counters)."""
    H, I = (768, 384) if fmt == 1 else (1024, 512)
    c = Case(fmt, T=9, H=H, E=16, k=4, I=I, seed=13)
    out = torch.empty((9, H), dtype=torch.bfloat16, device="cuda")
    binding.moe_decode_layer_noalloc(c.x, c.wr, None, c.w, 4, out,
                                     flags=binding._FLAG_TEST_STALL)
    torch.cuda.synchronize()
    assert binding.moe_noalloc_read_status() == -5  # MOE_ERR_DEVICE_TIMEOUT
    assert binding.moe_noalloc_read_status() == 0   # reading clears it
    c.run()  # the routing the oracle is given, from the workspace layer
    binding.moe_decode_layer_noalloc(c.x, c.wr, None, c.w, 4, out)
    torch.cuda.synchronize()
    assert binding.moe_noalloc_read_status() == 0
    c.out = out
    c.check_output()
