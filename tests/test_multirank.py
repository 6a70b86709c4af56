"""Multi-rank host logic of bench.py on CPU: two gloo ranks (world size 2).

The contraction shards by batch with no data-path collective (each rank works on its own
synthetic batch); what the ranks share is the step timing: a barrier on both sides of the
timed region, the maximum of the per-rank times, and a whole-job rate over all ranks'
units.  These tests run that logic with the gloo backend and CPU tensors.
"""
import io
import json
import os
import socket
import sys
import time
from contextlib import redirect_stdout

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, outdir):
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist

    import bench
    from paper_1705_01462_gb300 import synth

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    cpu = torch.device("cpu")
    res = {"rank": rank}
    # slowest rank decides the step time
    res["max_ms"] = bench.max_over_ranks(dist, 10.0 + 3.0 * rank, cpu)
    res["rate"] = bench.whole_job_rate(1e12, world, res["max_ms"])
    # each rank draws its own batch
    layer = synth.conv2x_3x3()
    x = synth.activations((1, 4, 4, layer.C), synth.layer_seed(3, bench.rank_seed_offset(rank) + 1))
    digests = [None] * world
    dist.all_gather_object(digests, float(np.abs(x).sum()))
    res["digests"] = digests
    # a barrier holds every rank until the slowest arrives
    if rank == 1:
        time.sleep(0.5)
    t0 = time.perf_counter()
    dist.barrier()
    res["barrier_wait_s"] = time.perf_counter() - t0
    # the reference arm prints only on rank 0: other ranks exit without work
    if rank != 0:
        buf = io.StringIO()

        class A:
            steps, warmup, gpus = 1, 0, world

        with redirect_stdout(buf):
            bench.run_reference(A, world, rank)
        res["reference_stdout"] = buf.getvalue()
    dist.barrier()
    dist.destroy_process_group()
    with open(os.path.join(outdir, f"rank{rank}.json"), "w") as f:
        json.dump(res, f)


def test_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp

    world = 2
    port = _free_port()
    mp.start_processes(_rank_main, args=(world, port, str(tmp_path)), nprocs=world, join=True,
                       start_method="spawn")
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    for r in res:
        assert r["max_ms"] == 13.0  # max over ranks, seen identically by every rank
        assert r["rate"] == pytest.approx(1e12 * 2 / 13e-3 / 1e12)
        assert r["digests"] == res[0]["digests"]
    assert res[0]["digests"][0] != res[0]["digests"][1]  # distinct batches per rank
    assert res[0]["barrier_wait_s"] >= 0.3  # rank 0 waited for the late rank
    assert res[1]["reference_stdout"] == ""


def test_single_rank_helpers():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(None, 4.5, None) == 4.5
    assert bench.whole_job_rate(2e12, 1, 1000.0) == pytest.approx(2.0)
    assert len({bench.rank_seed_offset(r) for r in range(8)}) == 8
