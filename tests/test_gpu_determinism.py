"""GPU tests of MOE_FLAG_DETERMINISTIC: every item of the expert kernels is
summed by one CTA over its whole K range and each token's k down rows are
added by the combine kernel in a fixed order, so the same call gives the same
output bits however the CTAs are scheduled.  Each case checks parity with the
float64 oracle, bit-identical outputs over repeated calls (same workspace, a
fresh workspace, while another stream loads the memory system, and from a CUDA
graph), and - where it holds by construction - that permuting the batch rows
permutes the output rows bit for bit."""
import numpy as np
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2
DET = binding.MOE_FLAG_DETERMINISTIC

# (format, T, H, E, k, I): the two served layers at decode batches, a batch
# whose activation terms are gathered (T > 64), and small shapes whose stage
# counts are below the SM count (many CTAs get no item)
SHAPES = [
    pytest.param(FP4, 1, 4096, 128, 8, 1536, id="nvfp4_235b_T1"),
    pytest.param(FP4, 64, 4096, 128, 8, 1536, id="nvfp4_235b_T64"),
    pytest.param(FP8, 8, 6144, 160, 8, 2560, id="fp8_480b_T8"),
    pytest.param(FP8, 64, 6144, 160, 8, 2560, id="fp8_480b_T64"),
    pytest.param(FP8, 160, 6144, 160, 8, 2560, id="fp8_480b_T160_gathered"),
    pytest.param(FP4, 96, 1024, 64, 4, 512, id="nvfp4_small_T96_gathered"),
    pytest.param(FP4, 5, 256, 8, 2, 256, id="nvfp4_tiny"),
    pytest.param(FP8, 3, 256, 4, 2, 128, id="fp8_tiny"),
]


def _sample(T):
    return sorted({0, T // 3, T // 2, T - 1})


def _call(c, out, ws, stream=None):
    binding.moe_decode_layer(c.x, c.wr, c.bias, c.w, c.k, out, ws, flags=c.flags,
                             residual=c.residual, stream=stream)


@pytest.mark.parametrize("fmt,T,H,E,k,I", SHAPES)
def test_repeated_calls_are_bit_identical(fmt, T, H, E, k, I):
    c = Case(fmt, T=T, H=H, E=E, k=k, I=I, seed=90 + T, residual=True, flags=DET).run()
    c.check_output(tokens=None if T * H <= 64 * 4096 else _sample(T))
    first = c.out.clone()
    outs = []
    out = torch.empty_like(first)
    # the same workspace again, then a fresh one
    for ws in (c.ws, binding.alloc_workspace(binding.moe_workspace_size(c.w, T, k, DET))):
        out.fill_(float("nan"))
        _call(c, out, ws)
        torch.cuda.synchronize()
        assert binding.moe_read_status(ws) == 0
        outs.append(out.clone())
    # while a copy on another stream competes for HBM and the SMs' L2 slices
    noise = torch.cuda.Stream()
    big = torch.empty(256 << 20, dtype=torch.uint8, device="cuda")
    dst = torch.empty_like(big)
    with torch.cuda.stream(noise):
        for _ in range(4):
            dst.copy_(big)
    out.fill_(float("nan"))
    _call(c, out, c.ws)
    torch.cuda.synchronize()
    outs.append(out.clone())
    # replayed from a CUDA graph
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        _call(c, out, c.ws, stream=s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            _call(c, out, c.ws, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    out.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert binding.moe_read_status(c.ws) == 0
    outs.append(out.clone())
    for i, o in enumerate(outs):
        assert torch.equal(o.view(torch.int16), first.view(torch.int16)), f"call {i + 1} differs"


@pytest.mark.parametrize("fmt,T,H,E,k,I", [
    pytest.param(FP4, 64, 4096, 128, 8, 1536, id="nvfp4_235b_T64"),
    pytest.param(FP8, 64, 6144, 160, 8, 2560, id="fp8_480b_T64"),
    pytest.param(FP8, 160, 6144, 160, 8, 2560, id="fp8_480b_T160_gathered"),
])
def test_permuted_batch_gives_permuted_rows(fmt, T, H, E, k, I):
    """A token's output depends on its own row only: the expert kernels sum
    each token column over the whole K range in one order whatever chunk the
    token lands in, and every other step works row by row."""
    w = synth.make_weights(fmt, E, H, I, seed=95, device="cuda")
    wr = synth.make_router(E, H, seed=95, device="cuda")
    x = synth.make_x(T, H, seed=96, device="cuda")
    perm = torch.from_numpy(np.random.default_rng(97).permutation(T)).cuda()
    a = Case(fmt, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x, flags=DET).run()
    b = Case(fmt, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x[perm].contiguous(), flags=DET).run()
    assert torch.equal(b.ids, a.ids[perm])
    assert torch.equal(b.out.view(torch.int16), a.out[perm].view(torch.int16))


@pytest.mark.parametrize("fmt,H,E,k,I", [
    pytest.param(FP4, 4096, 128, 8, 1536, id="nvfp4_235b"),
    pytest.param(FP8, 6144, 160, 8, 2560, id="fp8_480b"),
])
def test_token_rows_do_not_depend_on_the_batch(fmt, H, E, k, I):
    """Up to 64 tokens (8-token chunks, activation terms read per token) a
    token's output bits are the same in a batch of 1, 8, 17 or 64 tokens: the
    router's per-token sums do not depend on how many tokens share its blocks,
    and the expert kernels sum each token column alone over the whole K."""
    w = synth.make_weights(fmt, E, H, I, seed=103, device="cuda")
    wr = synth.make_router(E, H, seed=103, device="cuda")
    x = synth.make_x(64, H, seed=104, device="cuda")
    outs = {T: Case(fmt, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x[:T].contiguous(),
                    flags=DET).run().out for T in (1, 8, 17, 64)}
    for T in (1, 8, 17):
        assert torch.equal(outs[T].view(torch.int16), outs[64][:T].view(torch.int16)), T


@pytest.mark.parametrize("fmt,T,H,E,k,I", [
    pytest.param(FP4, 64, 4096, 128, 8, 1536, id="nvfp4_235b_T64"),
    pytest.param(FP8, 64, 6144, 160, 8, 2560, id="fp8_480b_T64"),
])
def test_same_result_as_the_default_mode_within_rounding(fmt, T, H, E, k, I):
    """The flag changes the order of the fp32 additions only: both modes route
    alike and agree with each other far inside the oracle tolerance."""
    w = synth.make_weights(fmt, E, H, I, seed=98, device="cuda")
    wr = synth.make_router(E, H, seed=98, device="cuda")
    x = synth.make_x(T, H, seed=99, device="cuda")
    a = Case(fmt, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x).run()
    b = Case(fmt, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x, flags=DET).run()
    assert torch.equal(a.ids, b.ids)
    ya = a.out.float()
    d = (ya - b.out.float()).abs()
    # fp32 sums reordered, then one bf16 rounding each: a few bf16 ulps of the
    # element, or of the fp32 rounding left over by cancellation in its row
    rowmax = ya.abs().amax(dim=1, keepdim=True)
    assert (d <= 4 * 2.0 ** -8 * ya.abs() + 2.0 ** -14 * rowmax).all()
    a.check_output(tokens=_sample(T))
    b.check_output(tokens=_sample(T))


def test_prefill_batch_is_bit_identical():
    """A prefill-shaped NVFP4 batch runs on the prefill engine, which stores
    whole-K sums and combines in a fixed order with or without the flag."""
    c = Case(FP4, T=2048, H=4096, E=128, k=8, I=1536, seed=100, flags=DET).run()
    c.check_output(tokens=[0, 1000, 2047], row_tol=2e-2)
    first = c.out.clone()
    for flags in (DET, 0):
        out = torch.empty_like(first)
        binding.moe_decode_layer(c.x, c.wr, c.bias, c.w, c.k, out, c.ws, flags=flags)
        torch.cuda.synchronize()
        assert torch.equal(out.view(torch.int16), first.view(torch.int16))


def test_noalloc_entry_point_takes_the_flag():
    """moe_decode_layer_noalloc sizes its scratch with the flag: a batch that
    fits runs bit-identical to the workspace call; one that does not is
    refused on the host."""
    T, H, E, k, I = 16, 4096, 128, 8, 1536
    c = Case(FP4, T=T, H=H, E=E, k=k, I=I, seed=101, flags=DET).run()
    out = torch.empty_like(c.out)
    binding.moe_decode_layer_noalloc(c.x, c.wr, c.bias, c.w, k, out, flags=DET)
    torch.cuda.synchronize()
    assert binding.moe_noalloc_read_status() == 0
    assert torch.equal(out.view(torch.int16), c.out.view(torch.int16))
    big = 64
    assert binding.moe_workspace_size(c.w, big, k, DET) > 16 << 20
    x = synth.make_x(big, H, seed=102, device="cuda")
    o = torch.empty((big, H), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.MoeError) as ei:
        binding.moe_decode_layer_noalloc(x, c.wr, None, c.w, k, o, flags=DET)
    assert ei.value.status == -3
