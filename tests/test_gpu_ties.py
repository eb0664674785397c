"""Exact logit ties on the device.

The selection rule is top-k by (logit desc, expert index asc), with -0 and +0
equal.  Random N(0, 0.02) routers practically never tie, so these routers are
built to:

- duplicated rows: expert groups whose router rows (and biases) are identical
  give bit-identical fp32 logits, whatever the summation order, because every
  expert's dot product runs through the same code path;
- an all-zero router: every logit is +0, so the top-k is experts 0..k-1 with
  gates 1/k;
- +0 and -0: x in [0, 0.5] against router rows of -2^-149 makes every product
  round to -0, and the bias -0 keeps the sum at -0; all-zero rows give +0
  (H = 1024, so that every lane of the router's reduction holds products).
  The other experts get negative logits, so the top-k is a set of signed
  zeros, taken in index order.

E = 128 and E = 160 put the tied experts on different lanes and on different
slots of a lane in the top-k warp (4 and 8 logits per lane).  T = 1, 8, 24 and
80 run the router with 1, 1, 4 and 8 experts per CTA.  Each case checks the
GPU's ids against a brute-force sort of the GPU's own fp32 logits, and the
layer output against the oracle."""
import numpy as np
import pytest
import torch

from paper_2609_11133_gb300 import binding, synth
from tests.gpu_harness import Case

pytestmark = pytest.mark.gpu

FP8, FP4 = 1, 2
NEG_TINY = -(2.0 ** -149)  # the negative fp32 subnormal of least magnitude


def brute_topk(logits, k):
    """ids [T, k] by (value desc, index asc); -0.0 == 0.0 in Python's order."""
    out = []
    for row in logits:
        order = sorted(range(row.size), key=lambda e: (-float(row[e]), e))
        out.append(order[:k])
    return np.array(out, dtype=np.int32)


def check_ids(c):
    lg = c.logits.cpu().numpy()
    ids = c.ids.cpu().numpy()
    assert np.array_equal(ids, brute_topk(lg, c.k))


def shape(fmt, E):
    # I small: the routing is under test, the expert path is checked as usual.
    # H = 1024: every lane of every router warp adds products (a lane with
    # none would add its +0 start value, and -0 + +0 = +0 in IEEE arithmetic)
    return dict(H=1024, I=256)


@pytest.mark.parametrize("fmt,E", [(FP4, 128), (FP8, 160)])
@pytest.mark.parametrize("T", [1, 8, 24, 80])
def test_ties_duplicated_router_rows(fmt, E, T):
    sh = shape(fmt, E)
    H, k = sh["H"], 8
    wr = synth.make_router(E, H, seed=40 + T, device="cpu")
    # group A (biased to the top) spans lanes 3, 3, 31, 0 and every lane slot;
    # group B (second) has six members, so the k-th place falls inside it
    grp_a = [3, 35, 127, 96]
    grp_b = [5, 37, 69, 64, 1, 100]
    if E > 128:
        grp_a += [131]
        grp_b += [159, 132]
    # plain duplicates (no bias): ties wherever such a pair lands in a top-k
    pairs = [(10, 42), (11, 74), (20, 21), (50, 114)]
    bias = torch.zeros(E)
    wr[grp_a] = wr[grp_a[0]].clone()
    wr[grp_b] = wr[grp_b[0]].clone()
    bias[grp_a] = 10.0
    bias[grp_b] = 5.0
    for a, b in pairs:
        wr[b] = wr[a].clone()
    c = Case(fmt, T=T, E=E, k=k, seed=41 + T, wr=wr.cuda(), bias=bias, **sh).run()
    lg = c.logits.cpu().numpy()
    for g in (grp_a, grp_b) + tuple(pairs):
        assert (lg[:, g] == lg[:, g[:1]]).all(), "duplicated rows gave different logits"
    check_ids(c)
    na = len(grp_a)
    ids = c.ids.cpu().numpy()
    assert (ids[:, :na] == np.sort(grp_a)).all()
    assert (ids[:, na:] == np.sort(grp_b)[:k - na]).all()
    c.check_output(row_tol=2e-2)


@pytest.mark.parametrize("fmt,E", [(FP4, 128), (FP8, 160)])
@pytest.mark.parametrize("T", [1, 24, 80])
def test_ties_all_zero_router(fmt, E, T):
    sh = shape(fmt, E)
    k = 8
    wr = torch.zeros((E, sh["H"]), dtype=torch.float32, device="cuda")
    c = Case(fmt, T=T, E=E, k=k, seed=50 + T, wr=wr, **sh).run()
    assert (c.logits.cpu().numpy() == 0).all()
    check_ids(c)
    assert (c.ids.cpu().numpy() == np.arange(k)).all()
    assert np.abs(c.gates.cpu().numpy() - 1.0 / k).max() <= 1e-7
    c.check_output(row_tol=2e-2)


def signed_zero_router(E, H, seed):
    """Router rows and bias whose logits are -0 for `neg`, +0 for `pos` and
    negative elsewhere, for any x in [0, 0.5]."""
    g = torch.Generator().manual_seed(seed)
    wr = -0.01 * (torch.rand((E, H), generator=g) + 0.5)
    neg = [2, 33, 66, 97, 98, 127] + ([129, 158] if E > 128 else [])
    pos = [0, 31, 34, 65, 100, 126] + ([130, 159] if E > 128 else [])
    wr[neg] = NEG_TINY
    wr[pos] = 0.0
    bias = torch.full((E,), -0.0)
    return wr, bias, neg, pos


@pytest.mark.parametrize("fmt,E", [(FP4, 128), (FP8, 160)])
@pytest.mark.parametrize("T", [1, 8, 24, 80])
def test_ties_signed_zero_logits(fmt, E, T):
    sh = shape(fmt, E)
    H, k = sh["H"], 8
    wr, bias, neg, pos = signed_zero_router(E, H, seed=60 + T)
    g = torch.Generator().manual_seed(61 + T)
    x = (torch.rand((T, H), generator=g) * 0.5).to(torch.bfloat16)
    c = Case(fmt, T=T, E=E, k=k, seed=62 + T, wr=wr.cuda(), x=x.cuda(), bias=bias, **sh).run()
    lg = c.logits.cpu().numpy()
    assert (lg[:, neg] == 0).all() and np.signbit(lg[:, neg]).all(), "expected -0 logits"
    assert (lg[:, pos] == 0).all() and not np.signbit(lg[:, pos]).any(), "expected +0 logits"
    check_ids(c)
    assert (c.ids.cpu().numpy() == np.sort(neg + pos)[:k]).all()
    c.check_output(row_tol=2e-2)


@pytest.mark.parametrize("E", [128, 160])
@pytest.mark.parametrize("T", [1, 24, 80])
def test_ties_standalone_route_topk(E, T):
    """moe_route_topk (the unfused router) on duplicated rows and signed zeros."""
    H, k = 1024, 8
    wr, bias, neg, pos = signed_zero_router(E, H, seed=70 + T)
    wr[[3, 35, 67, 99]] = 0.0  # four more +0 experts
    g = torch.Generator().manual_seed(71 + T)
    x = (torch.rand((T, H), generator=g) * 0.5).to(torch.bfloat16).cuda()
    ids = torch.empty((T, k), dtype=torch.int32, device="cuda")
    gates = torch.empty((T, k), dtype=torch.float32, device="cuda")
    logits = torch.empty((T, E), dtype=torch.float32, device="cuda")
    ws = binding.alloc_workspace(binding.moe_route_workspace_size(T, E))
    binding.moe_route_topk(x, wr.cuda(), bias.cuda(), k, ids, gates, ws, logits_out=logits)
    torch.cuda.synchronize()
    lg = logits.cpu().numpy()
    assert np.array_equal(ids.cpu().numpy(), brute_topk(lg, k))
    tied = np.sort(neg + pos + [3, 35, 67, 99])[:k]
    assert (ids.cpu().numpy() == tied).all()
    assert np.abs(gates.cpu().numpy() - 1.0 / k).max() <= 1e-7
