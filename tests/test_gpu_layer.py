"""GPU parity of the fused decode layer (moe_decode_layer) against the oracle."""
import numpy as np
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2


def test_tiny_fp8_layer_all_tokens():
    """The small case: H=512, E=8, top-2, I=256, T=4, seed 0."""
    c = Case(FP8, T=4, H=512, E=8, k=2, I=256, seed=0).run()
    c.check_output()


@pytest.mark.parametrize("T", [1, 8])
def test_qwen3_235b_nvfp4_layer(T):
    c = Case(FP4, T=T, H=4096, E=128, k=8, I=1536, seed=0).run()
    c.check_output()


def test_qwen3_235b_nvfp4_t64_full_batch():
    """Every token of the 235B-shaped NVFP4 layer at T=64, each row also
    within 2e-2 of its own maximum."""
    c = Case(FP4, T=64, H=4096, E=128, k=8, I=1536, seed=1).run()
    c.check_output(row_tol=2e-2)


def test_qwen3_480b_fp8_t64_full_batch():
    """Every token of the 480B-shaped FP8 layer at T=64 (the bench's layer)."""
    c = Case(FP8, T=64, H=6144, E=160, k=8, I=2560, seed=0).run()
    c.check_output(row_tol=2e-2)


@pytest.mark.parametrize("fmt,T,E,k", [(FP8, 13, 16, 4), (FP4, 37, 12, 3), (FP8, 3, 5, 5),
                                       (FP4, 1, 1, 1), (FP8, 9, 1, 1)])
def test_ragged_and_degenerate_shapes(fmt, T, E, k):
    H, I = (768, 384) if fmt == FP8 else (512, 512)
    c = Case(fmt, T=T, H=H, E=E, k=k, I=I, seed=T + E).run()
    c.check_output()


@pytest.mark.parametrize("fmt", [FP8, FP4])
def test_hot_experts_span_several_token_chunks(fmt):
    """A bias makes every token pick the same 4 experts: n_e = T > 32 tokens."""
    E, H = 16, 512
    bias = torch.zeros(E)
    bias[[3, 7, 8, 12]] = 50.0
    c = Case(fmt, T=77, H=H, E=E, k=4, I=256 if fmt == FP8 else 512, seed=5, bias=bias).run()
    assert set(np.unique(c.ids.cpu().numpy())) == {3, 7, 8, 12}
    c.check_output()


def test_no_renorm_bias_and_residual():
    bias = torch.linspace(-0.2, 0.2, 24)
    c = Case(FP4, T=11, H=1024, E=24, k=6, I=512, seed=9, bias=bias, residual=True,
             flags=binding.MOE_FLAG_NO_RENORM).run()
    c.check_output()


def test_prenorm_rms():
    c = Case(FP8, T=10, H=512, E=8, k=2, I=256, seed=11, residual=True,
             flags=binding.MOE_FLAG_PRENORM_RMS)
    c.x = synth.make_x(10, 512, seed=11, device="cuda", std=3.0)
    c.run()
    c.check_output()


def test_empty_batch_is_a_no_op():
    w = synth.make_weights(FP8, 8, 512, 256, device="cuda")
    x = torch.empty((0, 512), dtype=torch.bfloat16, device="cuda")
    out = torch.empty((0, 512), dtype=torch.bfloat16, device="cuda")
    ws = binding.alloc_workspace(binding.moe_workspace_size(w, 0, 2))
    wr = synth.make_router(8, 512, device="cuda")
    binding.moe_decode_layer(x, wr, None, w, 2, out, ws)
    torch.cuda.synchronize()


def test_repeated_calls_reuse_the_workspace():
    c = Case(FP4, T=8, H=1024, E=16, k=4, I=512, seed=21).run()
    first = c.out.clone()
    for _ in range(3):
        binding.moe_decode_layer(c.x, c.wr, None, c.w, c.k, c.out, c.ws)
    torch.cuda.synchronize()
    assert binding.moe_read_status(c.ws) == 0
    # the same inputs give the same bf16 outputs up to the order of fp32 atomics
    assert (c.out.float() - first.float()).abs().max() <= 1e-2 * first.float().abs().max()
    c.check_output()


def test_layer_replays_from_a_cuda_graph():
    """The layer enqueues only kernels on the caller's stream, so a captured
    graph replays it with new inputs in place."""
    c = Case(FP4, T=16, H=1024, E=16, k=4, I=512, seed=31).run()
    eager = c.out.clone()
    x_new = synth.make_x(16, 1024, seed=32, device="cuda")
    x_buf = c.x.clone()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        binding.moe_decode_layer(x_buf, c.wr, None, c.w, c.k, c.out, c.ws)
    g.replay()
    torch.cuda.synchronize()
    assert (c.out.float() - eager.float()).abs().max() <= 1e-2 * eager.float().abs().max()
    x_buf.copy_(x_new)
    g.replay()
    torch.cuda.synchronize()
    from_graph = c.out.clone()
    assert binding.moe_read_status(c.ws) == 0
    c.x = x_new
    c.run()  # eager call on the new input, checked against the oracle
    c.check_output()
    assert (from_graph.float() - c.out.float()).abs().max() <= 1e-2 * c.out.float().abs().max()
