"""GPU parity of the fused layer on the remaining workload shapes: the
235B-shaped NVFP4 layer at T=32 and T=128, the 480B-shaped FP8 layer under
Zipf-skewed routing across the batch sweep, and the 94-layer NVFP4 stack
with RMS pre-norm and the residual stream threaded between layers (each layer
checked teacher-forced: the oracle takes the GPU's input of that layer)."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case
from tests.util_np import np_, oracle_weights

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2
Q235 = dict(H=4096, E=128, k=8, I=1536)
Q480 = dict(H=6144, E=160, k=8, I=2560)


def test_qwen3_235b_nvfp4_t32_sampled_tokens():
    c = Case(FP4, T=32, seed=2, **Q235).run()
    c.check_output(tokens=[0, 13, 31])


def test_qwen3_235b_nvfp4_t128_prenorm_residual():
    """The layer of the 94-layer stack in its launch configuration (T=128)."""
    c = Case(FP4, T=128, seed=3, residual=True, flags=binding.MOE_FLAG_PRENORM_RMS,
             **Q235).run()
    c.check_output(tokens=[0, 64, 127])


@pytest.fixture(scope="module")
def zipf_layer():
    H, E, I = Q480["H"], Q480["E"], Q480["I"]
    w = synth.make_weights(FP8, E, H, I, seed=0, device="cuda")
    wr = synth.make_router(E, H, seed=0, device="cuda")
    bias = synth.make_zipf_bias(E, H, s=1.1, seed=0, device="cuda")
    ow = oracle_weights(w)
    yield w, wr, bias, ow
    del w, ow
    torch.cuda.empty_cache()


@pytest.mark.parametrize("T", [1, 8, 32, 128, 256])
def test_qwen3_480b_fp8_zipf_routing(zipf_layer, T):
    w, wr, bias, ow = zipf_layer
    x = synth.make_x(T, Q480["H"], seed=T, device="cuda")
    c = Case(FP8, T=T, w=w, wr=wr, x=x, ow=ow, bias=bias, **Q480).run()
    counts = np.bincount(c.ids.cpu().numpy().reshape(-1), minlength=Q480["E"])
    if T >= 128:
        # the bias concentrates the batch: the hottest expert spans several
        # 32-token chunks of the expert kernels
        assert counts.max() > 64, counts.max()
    hot = int(np.argmax(counts))
    on_hot = np.nonzero((c.ids.cpu().numpy() == hot).any(axis=1))[0]
    toks = sorted({0, T - 1, int(on_hot[-1])}) if T > 8 else None
    c.check_output(tokens=toks)


def test_94_layer_nvfp4_stack_teacher_forced():
    """94 fresh-weight 235B-shaped NVFP4 layers at T=128, x_{l+1} =
    bf16(x_l + MoE(RMSNorm(x_l))); layers 0, 1, 46 and 93 are checked against
    the oracle on the GPU's own input of that layer, the rest must stay finite
    and grow smoothly (the pre-norm keeps the stream bounded)."""
    L, T = 94, 128
    H, E, k, I = Q235["H"], Q235["E"], Q235["k"], Q235["I"]
    check = {0: [0, 127], 1: [5], 46: [64], 93: [0, 100]}
    xs = [synth.make_x(T, H, seed=0, device="cuda")]
    ws = None
    rms = []
    for l in range(L):
        w = synth.make_weights(FP4, E, H, I, seed=1009 * l, device="cuda")
        wr = synth.make_router(E, H, seed=1009 * l, device="cuda")
        if ws is None:
            ws = binding.alloc_workspace(binding.moe_workspace_size(w, T, k))
        out = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
        if l in check:
            c = Case(FP4, T=T, w=w, wr=wr, x=xs[l], residual=xs[l],
                     flags=binding.MOE_FLAG_PRENORM_RMS, **Q235).run(out=out)
            c.check_output(tokens=check[l])
        else:
            binding.moe_decode_layer(xs[l], wr, None, w, k, out, ws,
                                     flags=binding.MOE_FLAG_PRENORM_RMS, residual=xs[l])
        xs.append(out)
        rms.append(float(out.float().pow(2).mean().sqrt()))
        del w, wr
    torch.cuda.synchronize()
    assert binding.moe_read_status(ws) == 0
    assert all(np.isfinite(rms))
    # the increment of each layer is small next to the stream it is added to
    ratio = np.array(rms[1:]) / np.array(rms[:-1])
    assert (ratio > 0.9).all() and (ratio < 1.5).all(), ratio
    del xs
    torch.cuda.empty_cache()
