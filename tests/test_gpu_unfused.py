"""GPU parity of the four separate entry points against the oracle and the
fused layer: route_topk -> permute -> expert_ffn -> combine."""
import numpy as np
import pytest
import torch

from oracle import oracle
from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import GATE_TOL, REL_TOL, Case
from tests.util_np import np_, oracle_weights

pytestmark = pytest.mark.gpu


def unfused(c):
    T, H, E, k = c.T, c.H, c.E, c.k
    dev = "cuda"
    rws = binding.alloc_workspace(binding.moe_route_workspace_size(T, E))
    ids = torch.empty((T, k), dtype=torch.int32, device=dev)
    gw = torch.empty((T, k), dtype=torch.float32, device=dev)
    logits = torch.empty((T, E), dtype=torch.float32, device=dev)
    binding.moe_route_topk(c.x, c.wr, c.bias, k, ids, gw, rws, logits_out=logits)
    counts = torch.empty(E, dtype=torch.int32, device=dev)
    offsets = torch.empty(E + 1, dtype=torch.int32, device=dev)
    srt = torch.empty(T * k, dtype=torch.int32, device=dev)
    inv = torch.empty(T * k, dtype=torch.int32, device=dev)
    active = torch.empty(E + 1, dtype=torch.int32, device=dev)
    binding.moe_permute(ids, E, counts, offsets, srt, inv, active)
    ws = binding.alloc_workspace(binding.moe_workspace_size(c.w, T, k))
    y = torch.empty((T * k, H), dtype=torch.float32, device=dev)
    binding.moe_expert_ffn(c.x, c.w, offsets, srt, active, k, y, ws)
    out = torch.empty((T, H), dtype=torch.bfloat16, device=dev)
    binding.moe_combine(y, gw, inv, out, residual=c.residual)
    torch.cuda.synchronize()
    assert binding.moe_read_status(ws) == 0
    return dict(ids=ids, gw=gw, logits=logits, counts=counts, offsets=offsets, sorted=srt,
                inv=inv, active=active, y=y, out=out)


@pytest.mark.parametrize("fmt,T,H,E,k,I", [(1, 4, 512, 8, 2, 256), (2, 19, 1024, 32, 8, 512),
                                          (1, 40, 768, 12, 3, 384)])
def test_separate_entry_points_match_oracle(fmt, T, H, E, k, I):
    c = Case(fmt, T=T, H=H, E=E, k=k, I=I, seed=3, residual=True)
    r = unfused(c)
    # routing: bit-exact on the GPU's own logits
    o_ids, o_g = oracle.topk(r["logits"].double().cpu().numpy(), k)
    assert np.array_equal(o_ids, r["ids"].cpu().numpy())
    assert np.abs(o_g - r["gw"].double().cpu().numpy()).max() <= GATE_TOL
    # permutation: bit-exact
    cnt, off, srt, inv, act = oracle.permute(r["ids"].cpu().numpy(), E)
    assert np.array_equal(cnt, r["counts"].cpu().numpy())
    assert np.array_equal(off, r["offsets"].cpu().numpy())
    assert np.array_equal(srt, r["sorted"].cpu().numpy())
    assert np.array_equal(inv, r["inv"].cpu().numpy())
    assert np.array_equal(act[:1 + act[0]], r["active"].cpu().numpy()[:1 + act[0]])
    # expert outputs row by row
    ow = oracle_weights(c.w)
    xv = np_(c.x)
    from tests import indep
    xf = indep.bf16_to_f64(xv)
    y = r["y"].double().cpu().numpy()
    ids = r["ids"].cpu().numpy().reshape(-1)
    for p in range(0, T * k, max(1, T * k // 12)):
        a = srt[p]
        ref = oracle.expert_vec(ow, int(ids[a]), xf[a // k])
        assert np.abs(y[p] - ref).max() <= 1e-2 * max(np.abs(ref).max(), 1e-30)
    # combined output
    ref = oracle.moe_tokens(ow, xv, o_ids, o_g, residual_bits=np_(c.residual))
    got = r["out"].double().cpu().numpy()
    assert np.abs(got - ref).max() <= REL_TOL * np.abs(ref).max()


def test_unfused_matches_fused():
    c = Case(2, T=24, H=1024, E=16, k=4, I=512, seed=8, residual=True)
    r = unfused(c)
    c.run()
    assert torch.equal(r["ids"], c.ids)
    d = (r["out"].float() - c.out.float()).abs().max().item()
    assert d <= 1e-2 * c.out.float().abs().max().item()


def test_permute_reports_bad_expert_ids():
    dev = "cuda"
    E = 8
    ids = torch.tensor([[0, 1], [2, 9]], dtype=torch.int32, device=dev)
    outs = [torch.empty(n, dtype=torch.int32, device=dev) for n in (E, E + 1, 4, 4, E + 1)]
    binding.moe_permute(ids, E, *outs)
    torch.cuda.synchronize()
    assert outs[4][0].item() == -1


def test_permute_large_batch_against_oracle():
    dev = "cuda"
    T, k, E = 2000, 8, 160
    g = torch.Generator().manual_seed(0)
    ids = torch.stack([torch.randperm(E, generator=g)[:k] for _ in range(T)]).int()
    outs = [torch.empty(n, dtype=torch.int32, device=dev) for n in (E, E + 1, T * k, T * k, E + 1)]
    binding.moe_permute(ids.to(dev), E, *outs)
    torch.cuda.synchronize()
    ref = oracle.permute(ids.numpy(), E)
    for a, b in zip(ref, outs):
        assert np.array_equal(a, b.cpu().numpy())
