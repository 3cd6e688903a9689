"""The N > 1 path of bench.py is replicas only (each rank trains its own batch
of 256 on its own GPU; the only collectives are the timing barrier and the max
over ranks).  Its host logic runs here as two gloo ranks on the CPU: the max of
the ranks' times, the whole-job throughput, distinct synthetic inputs per rank,
and a reference arm that only rank 0 runs."""
import contextlib
import io
import os
import socket

import numpy as np
import torch.multiprocessing as mp

import bench
from paper_1911_07384_gb300 import synthetic as syn


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import torch.distributed as dist

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms = 10.0 + 5.0 * rank  # rank 1 is the slower replica
        ms_max = bench.max_over_ranks(ms, dist, "cpu")
        dist.barrier()
        x = syn.images_f16(syn.seed_for(4, "x", rank), 1, 8, 8, 3)
        out[rank] = (ms_max, bench.job_throughput(world, 256, 20, ms_max), x.tobytes())
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas_agree_on_the_slowest_time():
    world, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.start_processes(_rank, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0
    assert res[0][1] == res[1][1] == 2 * 256 * 20 / 0.015
    assert res[0][2] != res[1][2]  # each replica draws its own batch


def test_single_process_needs_no_collective():
    assert bench.max_over_ranks(12.5, None, "cpu") == 12.5
    assert np.isclose(bench.job_throughput(1, 256, 20, 16.5 * 20), 256 / 0.0165)


def test_reference_arm_runs_on_rank_zero_only():
    class A:
        steps, warmup, gpus = 2, 1, 2

    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        assert bench.run_reference(A(), 1, 2) == 0
    assert buf.getvalue() == ""
