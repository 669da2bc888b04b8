"""World-size-2 runs on CPU (gloo) of the multi-rank host logic.

The path shards over independent samples with no collective on the data
path; the bench launches one process per GPU and its only collectives are the
whole-job aggregation (max of the times, sum of tokens and FLOPs). Here two
CPU ranks check that aggregation, that each rank draws its own batch, and
that a rank's result for a sample is the single-process result for the same
sample (replicas compute the same function)."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import smartvl_oracle as O
from paper_2607_20357_gb300 import synth


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _sample0_logits(seed: int):
    wl = synth.WORKLOADS["tiny"]
    w = O.to_numpy_weights(synth.make_weights(wl.dims, 0))
    b = O.to_numpy_batch(synth.make_batch(wl, seed))
    return O.forward_batch(wl.dims, w, b, mode="fp64", samples=[0])[0]["logits"]


def _worker(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        (mx,), (tok, fl) = bench.job_aggregate([10.0 + rank], [100.0 * (rank + 1), 1.5], "cpu")
        seed = bench.rank_seed(rank)
        b = synth.make_batch(synth.WORKLOADS["tiny"], seed)
        digest = float(b["vis"].float().sum())
        digests = [None] * world
        dist.all_gather_object(digests, digest)
        q.put((rank, mx, tok, fl, digests, seed, _sample0_logits(seed).tolist()))
    except Exception as e:  # reported to the parent, which fails the test
        q.put((rank, "error", repr(e)))
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo_aggregation_and_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    try:
        results = sorted((q.get(timeout=300) for _ in procs), key=lambda r: r[0])
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
    for r in results:
        assert r[1] != "error", r
    for p in procs:
        assert p.exitcode == 0
    for rank, mx, tok, fl, digests, seed, logits in results:
        assert mx == 11.0                 # the slowest rank's time
        assert tok == 300.0 and fl == 3.0  # tokens and FLOPs of the whole job
        assert digests[0] != digests[1]   # each rank runs its own batch
        np.testing.assert_array_equal(np.asarray(logits), _sample0_logits(seed))


def test_single_process_aggregation_is_identity():
    import bench
    assert not dist.is_initialized()
    assert bench.job_aggregate([3.0], [4.0, 5.0]) == ([3.0], [4.0, 5.0])


def test_reference_arm_runs_on_rank_zero_only(capsys):
    """Under torchrun the reference arm (the oracle on the host cores) runs
    and prints on rank 0 alone; the other ranks return without work."""
    import argparse

    import bench
    ns = argparse.Namespace(workload="llava", steps=1, warmup=0, gpus=2)
    assert bench.run_reference(ns, rank=1, world=2) is None
    assert capsys.readouterr().out == ""
