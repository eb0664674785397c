"""The stage split of the tensor-core expert kernels, run on the host from the compiled library.

The kernels cut the work of one phase into stages and give each CTA a contiguous run of them.
moe_cost_split_stage runs the kernels' own split function on the host, on the plan the kernels
build from the per-expert token counts.  Here it is checked against the definition, written out
stage by stage:
- stage order: active experts in increasing id order, then row tile, then chunk of NT tokens,
  then K-block;
- a stage of a chunk with n tokens costs a + b * n;
- the split for num / den is the first stage whose preceding stages cost at least
  floor(C * num / den), C the total cost.

The kernels call it as: CTA i of G runs the stages from split(i * snum, G * sden) up to
split((i + 1) * snum, G * sden); snum / sden = 1 for the static split alone, 4 / 5 when the
FP8 engine leaves the rest to a shared tail starting at split(snum, sden)."""
import numpy as np
import pytest

from paper_2609_11133_gb300 import binding


def stage_costs(counts, NT, rtiles, KB, a, b):
    """Cost of every stage, in the kernels' stage order."""
    out = []
    for c in counts:
        if c == 0:
            continue
        chunks = [NT] * (c // NT) + ([c % NT] if c % NT else [])
        for _rt in range(rtiles):
            for n in chunks:
                out.extend([a + b * n] * KB)
    return np.asarray(out, dtype=np.int64)


def expected_split(P, num, den):
    """First stage s with P[s] >= floor(P[-1] * num / den); P[s] = cost of stages before s."""
    X = int(P[-1]) * num // den
    return int(np.searchsorted(P, X, side="left"))


def zipf_counts(rng, E, assignments, s):
    p = 1.0 / np.arange(1, E + 1) ** s
    p = rng.permutation(p / p.sum())
    return np.bincount(rng.choice(E, size=assignments, p=p), minlength=E)


CASES = [
    # (E, assignments, Zipf s, NT, rtiles, KB, a, b, grid, snum, sden)
    (128, 512, 0.0, 8, 12, 32, 24, 1, 152, 1, 1),    # 235B-like gate/up, per-token rows
    (128, 512, 1.1, 16, 8, 12, 64, 1, 152, 1, 1),    # 235B-like down, skewed
    (160, 512, 0.0, 8, 20, 48, 24, 1, 152, 4, 5),    # 480B-like gate/up with the shared tail
    (160, 512, 1.1, 8, 24, 20, 64, 1, 152, 4, 5),    # 480B-like down, skewed, with the tail
    (32, 256, 1.1, 8, 4, 8, 24, 1, 152, 1, 1),       # hot experts of many chunks
    (8, 8, 0.0, 32, 1, 2, 64, 1, 152, 1, 1),         # fewer stages than CTAs
    (64, 64, 0.5, 16, 3, 7, 1, 0, 19, 1, 1),         # plain stage count (b = 0)
    (16, 300, 1.5, 8, 5, 9, 3, 5, 7, 2, 3),          # token cost above stage cost
]


@pytest.mark.parametrize("case", CASES)
def test_split_matches_the_definition(case):
    E, m, s, NT, rtiles, KB, a, b, grid, snum, sden = case
    rng = np.random.default_rng(hash(case) % 2**32)
    counts = zipf_counts(rng, E, m, s)
    cost = stage_costs(counts, NT, rtiles, KB, a, b)
    P = np.concatenate([[0], np.cumsum(cost)])
    total, C = len(cost), int(P[-1])
    den = grid * sden

    def split(num, d=den):
        return binding.moe_cost_split_stage(counts, NT, rtiles, KB, a, b, num, d)

    bounds = [split(i * snum) for i in range(grid + 1)]
    assert bounds == [expected_split(P, i * snum, den) for i in range(grid + 1)]
    assert bounds[0] == 0 and all(x <= y for x, y in zip(bounds, bounds[1:]))
    # the static part ends where the shared tail begins; the whole range is every stage
    tail = split(snum, sden)
    assert bounds[-1] == tail == expected_split(P, snum, sden)
    assert split(den) == split(1, 1) == total
    # each CTA's cost is within one stage of its share
    share = C * snum / den
    per_cta = P[bounds[1:]] - P[bounds[:-1]]
    assert per_cta.max() <= share + cost.max() and per_cta.min() >= share - cost.max()


def test_every_fraction_on_a_small_plan():
    counts = [0, 3, 0, 17, 1, 8, 0, 0, 9]
    for NT in (1, 4, 8):
        for a, b in ((24, 1), (1, 0), (2, 7)):
            cost = stage_costs(counts, NT, 2, 3, a, b)
            P = np.concatenate([[0], np.cumsum(cost)])
            den = int(P[-1])
            for num in range(den + 1):  # every integer cost threshold
                got = binding.moe_cost_split_stage(counts, NT, 2, 3, a, b, num, den)
                assert got == expected_split(P, num, den), (NT, a, b, num)


def test_no_active_expert_gives_no_stages():
    for num in (0, 3, 7):
        assert binding.moe_cost_split_stage([0] * 12, 8, 4, 16, 24, 1, num, 7) == 0


def test_argument_checks():
    with pytest.raises(binding.MoeError) as e:
        binding.moe_cost_split_stage([1, 2], 8, 4, 16, 24, 1, 3, 2)  # num > den
    assert e.value.status == -1
    with pytest.raises(binding.MoeError) as e:
        binding.moe_cost_split_stage([1, -2], 8, 4, 16, 24, 1, 0, 2)
    assert e.value.status == -1
    with pytest.raises(binding.MoeError) as e:
        binding.moe_cost_split_stage([1] * 513, 8, 4, 16, 24, 1, 0, 2)
    assert e.value.status == -2
    with pytest.raises(binding.MoeError) as e:  # 2^31 stages
        binding.moe_cost_split_stage([1 << 20] * 4, 1, 1 << 10, 1 << 1, 24, 1, 0, 2)
    assert e.value.status == -2
