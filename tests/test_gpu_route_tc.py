"""GPU tests of the tensor-core router (route_tc.cu), which batches with
T * H >= 2^21 and E <= 256 use: the fp32 router split into three bf16 parts, a
tcgen05 bf16 GEMM over eight K slices, the slices added in order by the router
kernel.  Each case checks the routing as every layer case does (the oracle's
top-k of the GPU's logits equals the GPU's ids bit for bit; the logits lie
within the fp32 dot-product bound of the float64 ones) and the layer output
against the oracle."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case
from tests.test_gpu_ties import brute_topk, signed_zero_router

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_one_hot_rows_give_the_router_weights_exactly():
    """x rows with a single 1.0: the fp32 GEMV gives the router weight itself,
    and so must the GEMM, which holds only if the three bf16 parts of every
    weight add up to it exactly (two parts would leave up to 8 bits out)."""
    T, H, E, k = 2048, 1024, 160, 8
    g = torch.Generator().manual_seed(80)
    wr = torch.randn((E, H), generator=g) * 0.05  # full 24-bit significands
    cols = (np.arange(T) * 37) % H
    x = torch.zeros((T, H))
    x[np.arange(T), cols] = 1.0
    c = Case(FP8, T=T, H=H, E=E, k=k, I=256, seed=80, wr=wr.cuda(),
             x=x.to(torch.bfloat16).cuda()).run()
    want = wr.numpy()[:, cols].T
    assert np.array_equal(c.logits.cpu().numpy().view(np.uint32), want.view(np.uint32))
    c.check_output(tokens=[0, 1, 777, T - 1], row_tol=2e-2)


@pytest.mark.parametrize("fmt,T,H,E,k,I,pre", [
    pytest.param(FP4, 512, 4096, 128, 8, 1536, True, id="nvfp4_235b_T512_prenorm"),
    pytest.param(FP8, 342, 6144, 160, 8, 256, False, id="fp8_H6144_E160_T342"),
    pytest.param(FP4, 520, 4096, 100, 6, 256, False, id="nvfp4_E100_padded_T520"),
    pytest.param(FP8, 8192, 256, 256, 8, 128, True, id="fp8_E256_H256_T8192"),
    pytest.param(FP4, 1030, 2048, 64, 4, 512, False, id="nvfp4_E64_T1030"),
])
def test_layer_routes_on_the_tensor_cores(fmt, T, H, E, k, I, pre):
    bias = torch.linspace(-0.1, 0.1, E)
    flags = binding.MOE_FLAG_PRENORM_RMS if pre else 0
    c = Case(fmt, T=T, H=H, E=E, k=k, I=I, seed=81 + T, bias=bias, residual=pre,
             flags=flags).run()
    assert binding.moe_layer_kernel_count(c.w, T, k) == 8  # prep and GEMM in the launch list
    c.check_output(tokens=[0, 1, T // 3, T // 2, T - 1], row_tol=2e-2)


SCRIPT = r"""
import sys, torch
sys.path.insert(0, {root!r})
from tests.gpu_harness import Case
for fmt, T, H, E, k in [(2, 1, 1024, 160, 8), (1, 5, 256, 100, 4), (2, 64, 2048, 128, 8),
                        (1, 127, 1024, 16, 2)]:
    c = Case(fmt, T=T, H=H, E=E, k=k, I=256, seed=90 + T, bias=torch.linspace(-1, 1, E)).run()
    c.check_output(row_tol=2e-2)
print("TC_SMALL_OK")
"""


def test_forced_on_small_batches():
    """MOE_ROUTE_TC=1 (in a subprocess) puts small batches on the tensor-core
    router too: one partial token tile of 1 to 127 rows."""
    env = dict(os.environ, MOE_ROUTE_TC="1")
    r = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT)], env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0 and "TC_SMALL_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]


@pytest.mark.parametrize("fmt,E", [(FP4, 128), (FP8, 160)])
def test_ties_on_the_tensor_cores(fmt, E):
    """Duplicated router rows give bit-identical logits (identical B rows of the
    GEMM), an all-zero router gives zero logits, and rows of -2^-149 (whose
    three bf16 parts are all -0) tie with zero rows: the top-k takes the zero
    logits in index order whatever the sign the tensor cores give them."""
    T, H, k = 2048, 1024, 8
    wr = synth.make_router(E, H, seed=95, device="cpu")
    grp = [3, 35, 127, 96]
    wr[grp] = wr[grp[0]].clone()
    bias = torch.zeros(E)
    bias[grp] = 10.0
    c = Case(fmt, T=T, H=H, E=E, k=k, I=256, seed=95, wr=wr.cuda(), bias=bias).run()
    lg = c.logits.cpu().numpy()
    assert (lg[:, grp] == lg[:, grp[:1]]).all()
    assert np.array_equal(c.ids.cpu().numpy(), brute_topk(lg, k))
    assert (c.ids.cpu().numpy()[:, :4] == np.sort(grp)).all()
    c.check_output(tokens=[0, 5, T - 1], row_tol=2e-2)

    z = Case(fmt, T=T, H=H, E=E, k=k, I=256, seed=96,
             wr=torch.zeros((E, H), device="cuda")).run()
    assert (z.logits.cpu().numpy() == 0).all()
    assert (z.ids.cpu().numpy() == np.arange(k)).all()
    z.check_output(tokens=[0, 5, T - 1], row_tol=2e-2)

    wr, bias, neg, pos = signed_zero_router(E, H, seed=97)
    g = torch.Generator().manual_seed(98)
    x = (torch.rand((T, H), generator=g) * 0.5).to(torch.bfloat16)
    s = Case(fmt, T=T, H=H, E=E, k=k, I=256, seed=99, wr=wr.cuda(), x=x.cuda(),
             bias=bias).run()
    lg = s.logits.cpu().numpy()
    assert (lg[:, neg + pos] == 0).all()
    assert np.array_equal(s.ids.cpu().numpy(), brute_topk(lg, k))
    assert (s.ids.cpu().numpy() == np.sort(neg + pos)[:k]).all()
    s.check_output(tokens=[0, 5, T - 1], row_tol=2e-2)
