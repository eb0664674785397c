"""The FP8 tensor-core kernel's stage order, run on the host from the compiled library.

moe_stage_order runs the kernel's own cursor on the plan the kernel builds from the per-expert
token counts.  Here it is checked against the order written out from its definition:
- groups (active expert in increasing id order, then row tile) in the same places as in the
  item order of moe_cost_split_stage (chunk, then K-block);
- inside a group of several chunks, K-blocks cut into slabs of `slab` (the last one shorter),
  and every chunk over one slab before any chunk over the next;
- a group of one chunk, or slab 0 or >= KB: the item order.
The epilogue relies on one property of it: until run_end, the next stage continues the same
chunk's run (same item, next K-block), so partial sums are added out only at run_end."""
import numpy as np
import pytest

from paper_2609_11133_gb300 import binding


def expected_order(counts, NT, rtiles, KB, slab):
    item, kb, end = [], [], []
    it0 = 0
    for c in counts:
        if c == 0:
            continue
        nch = -(-c // NT)
        g = slab if (nch > 1 and 0 < slab < KB) else KB
        for _rt in range(rtiles):
            for lo in range(0, KB, g):
                hi = min(lo + g, KB)
                for ch in range(nch):
                    for k in range(lo, hi):
                        item.append(it0 + ch)
                        kb.append(k)
                        end.append(1 if k == hi - 1 else 0)
            it0 += nch
    return item, kb, end


def zipf_counts(E, assignments, s, seed):
    rng = np.random.default_rng(seed)
    p = 1.0 / np.arange(1, E + 1) ** s
    p = rng.permutation(p / p.sum())
    return np.bincount(rng.choice(E, size=assignments, p=p), minlength=E).tolist()


CASES = [
    # (counts, NT, rtiles, KB, slab)
    (zipf_counts(160, 256 * 8, 1.1, 1), 32, 20, 48, 8),   # 480B gate/up, Zipf T=256
    (zipf_counts(160, 256 * 8, 1.1, 1), 32, 24, 20, 8),   # 480B down: slabs of 8, 8, 4
    (zipf_counts(160, 128 * 8, 1.1, 2), 32, 20, 48, 7),   # slab not dividing KB
    (zipf_counts(160, 32 * 8, 1.1, 3), 8, 20, 48, 8),     # 8-token chunks
    (zipf_counts(160, 64 * 8, 0.0, 4), 8, 24, 20, 8),     # uniform decode batch
    ([0, 40, 0, 3, 17, 0, 64, 1], 8, 3, 5, 1),            # slabs of one K-block
    ([0, 40, 0, 3, 17, 0, 64, 1], 8, 3, 5, 5),            # slab = KB: item order
    ([0, 40, 0, 3, 17, 0, 64, 1], 8, 3, 5, 9),            # slab > KB: item order
    ([9, 0, 0, 33], 16, 2, 6, 4),                         # 4 + 2
    ([5] * 12, 8, 4, 16, 8),                              # one chunk everywhere
]


def _stages(counts, NT, rtiles, KB):
    return sum(-(-c // NT) for c in counts if c > 0) * rtiles * KB


@pytest.mark.parametrize("counts,NT,rtiles,KB,slab", CASES)
def test_order_matches_the_definition(counts, NT, rtiles, KB, slab):
    n = _stages(counts, NT, rtiles, KB)
    want = expected_order(counts, NT, rtiles, KB, slab)
    got = binding.moe_stage_order(counts, NT, rtiles, KB, slab, 0, n)
    assert got[0] == want[0] and got[1] == want[1] and got[2] == want[2]
    # every (item, K-block) exactly once: the same stages as the item order
    items = sum(-(-c // NT) for c in counts if c > 0) * rtiles
    pairs = set(zip(got[0], got[1]))
    assert len(pairs) == n == items * KB
    # the epilogue's invariant: inside a run the next stage continues it
    it, kb, end = (np.asarray(v) for v in got)
    inside = np.nonzero(end[:-1] == 0)[0]
    assert (it[inside + 1] == it[inside]).all() and (kb[inside + 1] == kb[inside] + 1).all()
    assert end[-1] == 1


@pytest.mark.parametrize("counts,NT,rtiles,KB,slab", CASES)
def test_seek_from_any_stage(counts, NT, rtiles, KB, slab):
    """A CTA starts at its share's first stage and jumps to the shared tail's units: the cursor
    placed at any stage gives the same stages as the walk from the start."""
    n = _stages(counts, NT, rtiles, KB)
    want = expected_order(counts, NT, rtiles, KB, slab)
    rng = np.random.default_rng(n)
    starts = sorted(set(rng.integers(0, n, size=40).tolist()) | {0, n - 1})
    for s in starts:
        m = min(n - s, 300)
        got = binding.moe_stage_order(counts, NT, rtiles, KB, slab, s, m)
        assert got == (want[0][s:s + m], want[1][s:s + m], want[2][s:s + m]), s


def test_whole_items_without_slabs():
    counts = zipf_counts(160, 256 * 8, 1.1, 5)
    NT, rtiles, KB = 32, 20, 48
    n = _stages(counts, NT, rtiles, KB)
    it, kb, end = binding.moe_stage_order(counts, NT, rtiles, KB, 0, 0, n)
    s = np.arange(n)
    assert (np.asarray(it) == s // KB).all() and (np.asarray(kb) == s % KB).all()
    assert (np.asarray(end) == (s % KB == KB - 1)).all()


def test_groups_keep_their_place():
    """Slabs reorder stages only inside an (expert, row tile) group, so the cost split's
    boundaries between groups mean the same stages in both orders."""
    counts = zipf_counts(160, 128 * 8, 1.1, 6)
    NT, rtiles, KB = 32, 20, 48
    n = _stages(counts, NT, rtiles, KB)
    a = binding.moe_stage_order(counts, NT, rtiles, KB, 0, 0, n)
    b = binding.moe_stage_order(counts, NT, rtiles, KB, 8, 0, n)
    nch = [-(-c // NT) for c in counts if c > 0]
    bounds = np.cumsum([0] + [ch * KB for ch in nch for _ in range(rtiles)])
    for lo, hi in zip(bounds[:-1], bounds[1:]):
        assert sorted(zip(a[0][lo:hi], a[1][lo:hi])) == sorted(zip(b[0][lo:hi], b[1][lo:hi]))


def test_rejects_bad_arguments():
    with pytest.raises(binding.MoeError):
        binding.moe_stage_order([4, 4], 8, 2, 3, -1, 0, 1)
    with pytest.raises(binding.MoeError):
        binding.moe_stage_order([4, 4], 8, 2, 3, 2, 0, 13)  # 12 stages
    with pytest.raises(binding.MoeError):
        binding.moe_stage_order([4, -4], 8, 2, 3, 2, 0, 1)
    with pytest.raises(binding.MoeError):
        binding.moe_stage_order([1] * 513, 8, 2, 3, 2, 0, 1)
    assert binding.moe_stage_order([4, 4], 8, 2, 3, 2, 12, 0) == ([], [], [])
