"""GPU parity of the NVFP4 prefill engine (ffn_pf.cuh): batches with at least
32 tokens per expert on average (T * k >= 32 * E, more than 64 tokens) take
items of one 128-row weight tile against a group of up to 64 tokens, with the
first three of the four activation terms, and the combine kernel sums each
assignment's down row.  Every case is compared with the float64 oracle, on
every token unless the shape is the full 235B-shaped layer."""
import os
import subprocess
import sys

import numpy as np
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP4 = 2
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_small_prefill_shape_every_token():
    """T=256, 16 experts, top-4: ~64 tokens per expert (one or two groups)."""
    c = Case(FP4, T=256, H=1024, E=16, k=4, I=512, seed=61).run()
    n = np.bincount(c.ids.cpu().numpy().reshape(-1), minlength=16)
    assert n.max() > 64  # some experts span two token groups
    c.check_output(row_tol=2e-2)


def test_ragged_groups_hot_and_empty_experts():
    """A bias sends every token to expert 3 (five groups of 64, the last one
    partial) and no token to experts 0-1; the others get ragged groups."""
    E = 8
    bias = torch.zeros(E)
    bias[3] = 50.0
    bias[0] = bias[1] = -50.0
    c = Case(FP4, T=300, H=768, E=E, k=2, I=512, seed=62, bias=bias).run()
    n = np.bincount(c.ids.cpu().numpy().reshape(-1), minlength=E)
    assert n[3] == 300 and n[0] == 0 and n[1] == 0
    c.check_output(row_tol=2e-2)


def test_prenorm_residual_and_no_renorm():
    bias = torch.linspace(-0.2, 0.2, 12)
    flags = binding.MOE_FLAG_PRENORM_RMS | binding.MOE_FLAG_NO_RENORM
    c = Case(FP4, T=160, H=1024, E=12, k=3, I=768, seed=63, bias=bias, residual=True,
             flags=flags).run()
    c.check_output(row_tol=2e-2)


def test_outlier_channels_with_three_terms():
    """Four channels of x at 10^3 times the others: the terms keep what the
    outliers leave of each 16-element block."""
    T, H = 192, 1024
    x = synth.make_x(T, H, seed=64, device="cuda").float()
    x[:, [5, 300, 301, 777]] *= 1000.0
    x = x.to(torch.bfloat16)
    c = Case(FP4, T=T, H=H, E=8, k=2, I=512, seed=64, x=x).run()
    c.check_output(row_tol=2e-2)


def test_qwen3_235b_prefill_rows():
    """The 235B-shaped layer at T=2048 (~128 tokens per expert), sampled
    tokens, each row within 2e-2 of its own maximum."""
    c = Case(FP4, T=2048, H=4096, E=128, k=8, I=1536, seed=65).run()
    c.check_output(tokens=[0, 1, 700, 1023, 1500, 2046, 2047], row_tol=2e-2)


def test_consecutive_calls_and_graph_replay():
    """Two calls with different batches on one workspace, then a CUDA graph
    of a call replayed: the per-expert counters and the combine start from
    zero each time."""
    T, H, E, k, I = 256, 1024, 16, 4, 512
    w = synth.make_weights(FP4, E, H, I, seed=66, device="cuda")
    wr = synth.make_router(E, H, seed=66, device="cuda")
    ws = binding.alloc_workspace(binding.moe_workspace_size(w, T, k))
    for i in range(2):
        x = synth.make_x(T, H, seed=67 + i, device="cuda")
        Case(FP4, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x).run(ws=ws).check_output()
    x = synth.make_x(T, H, seed=69, device="cuda")
    out = torch.empty((T, H), dtype=torch.bfloat16, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        binding.moe_decode_layer(x, wr, None, w, k, out, ws)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            binding.moe_decode_layer(x, wr, None, w, k, out, ws)
    torch.cuda.current_stream().wait_stream(s)
    out.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert binding.moe_read_status(ws) == 0
    ref = Case(FP4, T=T, H=H, E=E, k=k, I=I, w=w, wr=wr, x=x).run()
    a, b = out.float(), ref.out.float()
    assert torch.isfinite(a).all()
    assert (a - b).abs().max() <= 2e-2 * b.abs().max()
    ref.check_output()


def test_expired_wait_is_reported_and_context_survives():
    from tests.test_gpu_errors import stall_then_recover
    stall_then_recover(FP4, T=256, H=1024, E=16, k=4, I=512, seed=70)


SCRIPT = r"""
import sys, torch
sys.path.insert(0, {root!r})
from tests.gpu_harness import Case
c = Case(2, T=2048, H=4096, E=128, k=8, I=1536, seed=71).run()
c.check_output(tokens=[3, 1029, 2040])
torch.save({{"ids": c.ids.cpu(), "out": c.out.cpu()}}, {path!r})
print("DECODE_OK")
"""


def test_same_routing_and_outputs_as_the_decode_engine(tmp_path):
    """The decode engine (MOE_PF=0, in a subprocess) and the prefill engine
    route every token alike and agree within the oracle's tolerance."""
    path = str(tmp_path / "decode.pt")
    env = dict(os.environ, MOE_PF="0")
    r = subprocess.run([sys.executable, "-c", SCRIPT.format(root=ROOT, path=path)], env=env,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0 and "DECODE_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
    dec = torch.load(path)
    c = Case(FP4, T=2048, H=4096, E=128, k=8, I=1536, seed=71).run()
    assert torch.equal(dec["ids"], c.ids.cpu())
    a, b = dec["out"].float(), c.out.cpu().float()
    assert (a - b).abs().max() <= 2e-2 * b.abs().max()
    c.check_output(tokens=[3, 1029, 2040])
