"""The N>1 launch of the benchmark on the host: two ranks over gloo on CPU.

The layer does not shard across GPUs, so an N-GPU run is N independent
replicas: every rank holds the same weights (seeded by layer), decodes its own
batch (activations seeded by seed + rank), and the only cross-rank traffic is
the barrier and the max-over-ranks of the step time.  These tests run that
host logic with world size 2: the rank environment, the all-reduce max on a
gloo group, the whole-job throughput, that the reference arm does its work on
rank 0 only, and that each replica's result is the one a single process
computes for its seed (the float64 oracle stands in for the device path)."""
import contextlib
import io
import json
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench

WORLD = 2
SEED = 5


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _replica_output(rank):
    """What rank `rank` decodes: the tiny FP8 layer on its own activations."""
    from oracle import oracle
    from paper_2609_11133_gb300 import synth
    wl = bench.WORKLOADS["tiny_fp8"]
    fmt, H, E, k, I, T = (wl[n] for n in ("fmt", "H", "E", "k", "I", "T"))
    s0 = bench.layer_seed(SEED, 0)
    w = synth.make_weights(fmt, E, H, I, seed=s0)
    wr = synth.make_router(E, H, seed=s0).numpy()
    x = synth.make_x(T, H, seed=SEED + rank)
    xb = x.view(torch.int16).numpy().view(np.uint16)
    out, ids, _, _ = oracle.layer(bench._oracle_weights(w), xb, wr, k)
    wsum = float(w.w_gate.float().sum() + w.w_down.float().sum())
    return out, ids, wsum


def _rank_main(rank, port, outdir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(WORLD), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        r, world, local = bench.dist_env()
        # each rank's step time differs; all of them report the slowest
        ms = bench.barrier_max(1.0 + 0.25 * rank, world)
        bench.barrier(world)
        # the reference arm: ranks other than 0 return at once, printing nothing
        buf = io.StringIO()
        if rank != 0:
            with contextlib.redirect_stdout(buf):
                bench.run_reference(bench.parse(["--impl", "reference",
                                                 "--workload", "tiny_fp8"]))
        out, ids, wsum = _replica_output(rank)
        outs = [None] * world
        dist.all_gather_object(outs, (out.tolist(), ids.tolist(), wsum))
        with open(os.path.join(outdir, f"rank{rank}.json"), "w") as f:
            json.dump({"env": [r, world, local], "ms": ms, "ref_stdout": buf.getvalue(),
                       "all": outs}, f)
    finally:
        dist.destroy_process_group()


@pytest.fixture(scope="module")
def ranks(tmp_path_factory):
    d = str(tmp_path_factory.mktemp("gloo"))
    mp.spawn(_rank_main, args=(_free_port(), d), nprocs=WORLD, join=True)
    return [json.load(open(os.path.join(d, f"rank{r}.json"))) for r in range(WORLD)]


def test_rank_environment(ranks):
    for r, res in enumerate(ranks):
        assert res["env"] == [r, WORLD, r]


def test_step_time_is_the_slowest_rank(ranks):
    assert [res["ms"] for res in ranks] == [1.25, 1.25]


def test_job_throughput_counts_every_replica():
    # two replicas of 64 tokens each at 0.25 ms per step: 512k tokens/s
    assert bench.job_throughput(0.25, 64, 2) == pytest.approx(512000.0)
    assert bench.job_throughput(0.25, 64, 1) == pytest.approx(256000.0)


def test_reference_arm_runs_on_rank_zero_only(ranks):
    assert ranks[1]["ref_stdout"] == ""


def test_replicas_share_weights_and_decode_their_own_batch(ranks):
    gathered = ranks[0]["all"]
    assert gathered == ranks[1]["all"]
    (o0, i0, w0), (o1, i1, w1) = gathered
    assert w0 == w1  # one set of weights on every rank
    assert not np.array_equal(np.asarray(o0), np.asarray(o1))  # distinct batches
    for r in range(WORLD):
        out, ids, _ = _replica_output(r)  # the same replica, decoded alone
        np.testing.assert_array_equal(np.asarray(gathered[r][0]), out)
        np.testing.assert_array_equal(np.asarray(gathered[r][1]), ids)
