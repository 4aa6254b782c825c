"""The multi-rank logic of bench.py on CPU with the gloo backend (world size
2): one process per rank, the job's time is the slowest rank's, throughput
counts every rank's units, every rank draws its own queries, and only rank 0
runs the reference arm; the clock record keeps only samples of the timed
region."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = 1.5 + rank                        # rank 1 is the slow one
        t = bench.slowest(dist, mine, "cpu")
        seeds = [None] * world
        dist.all_gather_object(seeds, bench.query_seed(3, rank))
        out[rank] = (t, bench.job_rate(1000.0, world, t), seeds, bench.dist_env())
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_slowest_time_and_job_rate():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        t, rate, seeds, env = res[rank]
        assert t == 2.5                          # max over ranks
        assert rate == pytest.approx(1000.0 * world / 2.5)
        assert len(set(seeds)) == world           # queries differ per rank
        assert env == (rank, world, rank)


def test_slowest_without_a_process_group_is_the_local_time():
    assert bench.slowest(None, 3.25, "cpu") == 3.25
    assert bench.job_rate(10.0, 1, 2.0) == 5.0


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    bench.reference_arm(object())                # returns before reading any argument
    assert capsys.readouterr().out == ""


def test_clock_summary_keeps_the_samples_of_the_timed_region():
    """The clock record of a bench line: only samples that arrived between the
    region's start and one sampling period after its end count; throttle
    reasons are collected from those samples alone."""
    cs = bench.ClockSampler(0)
    cs.t0, cs.t1 = 10.0, 11.0
    row = "0, {sm}, 2070, 900.00, 0x0, {hw}, Not Active, Not Active, {pc}\n"
    cs.rows = [
        (9.5, row.format(sm=1200, hw="Active", pc="Not Active")),      # before: dropped
        (10.2, row.format(sm=2070, hw="Not Active", pc="Not Active")),
        (10.6, row.format(sm=2055, hw="Not Active", pc="Active")),
        (11.05, row.format(sm=2070, hw="Not Active", pc="Not Active")),  # last period: kept
        (11.5, row.format(sm=900, hw="Active", pc="Not Active")),       # after: dropped
    ]
    s = cs.summary()
    assert s["samples"] == 3
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["sw_power_cap"]
    cs.rows = [(12.0, row.format(sm=2070, hw="Not Active", pc="Not Active"))]
    assert cs.summary()["reasons"] == ["unsampled"]
