"""moe_decode_layer_noalloc: the fused layer for callers that must not allocate
device memory while they run it (an engine plugin's enqueue path, a serving
loop that cannot afford a synchronising cudaMalloc).  It runs on the
library's own 16 MiB scratch array, so the test checks it against the
workspace-taking moe_decode_layer on the same inputs, on two calls in a row
(the second call reuses the array the first one left behind)."""
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth

pytestmark = pytest.mark.gpu

REL_TOL = 2e-2  # the output tolerance of the other layer tests


def _inputs(fmt, T, H, E, k, I, seed):
    w = synth.make_weights(fmt, E, H, I, seed=seed, device="cuda")
    x = synth.make_x(T, H, seed=seed, device="cuda")
    wr = synth.make_router(E, H, seed=seed, device="cuda")
    return w, x, wr


@pytest.mark.parametrize("fmt,T,H,E,k,I", [(2, 8, 4096, 128, 8, 1536), (1, 13, 768, 16, 4, 384)])
def test_noalloc_matches_workspace_layer_on_consecutive_calls(fmt, T, H, E, k, I):
    w, x, wr = _inputs(fmt, T, H, E, k, I, seed=7)
    ref = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    ws = binding.alloc_workspace(binding.moe_workspace_size(w, T, k))
    binding.moe_decode_layer(x, wr, None, w, k, ref, ws)
    scale = ref.float().abs().max().item()
    for _ in range(2):
        out = torch.full((T, H), float("nan"), dtype=torch.bfloat16, device="cuda")
        binding.moe_decode_layer_noalloc(x, wr, None, w, k, out)
        torch.cuda.synchronize()
        assert torch.isfinite(out.float()).all()
        assert (out.float() - ref.float()).abs().max().item() <= REL_TOL * scale


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
    assert (out.float() - ref.float()).abs().max().item() <= REL_TOL * ref.float().abs().max().item()


def test_noalloc_rejects_shapes_beyond_its_scratch():
    w = synth.make_weights(2, 128, 4096, 1536, seed=0, device="cuda", experts=[0])
    T = 200  # needs more than 16 MiB of scratch
    x = torch.zeros((T, 4096), dtype=torch.bfloat16, device="cuda")
    wr = torch.zeros((128, 4096), dtype=torch.float32, device="cuda")
    out = torch.empty((T, 4096), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.MoeError) as ei:
        binding.moe_decode_layer_noalloc(x, wr, None, w, 8, out)
    assert ei.value.status == -3  # MOE_ERR_WORKSPACE_TOO_SMALL
