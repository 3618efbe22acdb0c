"""The multi-GPU bench path on CPU: two gloo ranks run the host logic bench.py
uses under torchrun (one independent replica per rank, slowest rank's time,
whole-job throughput) and the reference arm's rank rule."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import tracegen as tg
    cfg = bench.replica_cfg(tg.CONFIGS["tiny"], rank, world)
    ms = 10.0 + 5.0 * rank                      # rank 1 is the slow one
    ms_max = bench.max_over_ranks(ms, world, torch.device("cpu"))
    value = bench.job_throughput(1000, world, ms_max)
    out[rank] = (cfg.trace_seed, ms_max, value)
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_rank, args=(world, _free_port(), out), nprocs=world, start_method="spawn", join=True)
    seeds = {out[r][0] for r in range(world)}
    assert len(seeds) == world                               # independent replicas
    for r in range(world):
        assert out[r][1] == 15.0                             # every rank reports the slowest time
        assert out[r][2] == pytest.approx(1000 * world / 0.015)  # units of all ranks / slowest time


def test_single_rank_is_unchanged():
    import bench
    import tracegen as tg
    cfg = tg.CONFIGS["tiny"]
    assert bench.replica_cfg(cfg, 0, 1) is cfg
    assert bench.max_over_ranks(7.5, 1, torch.device("cpu")) == 7.5
    assert bench.job_throughput(300, 1, 3.0) == pytest.approx(100000.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    bench.run_reference(bench.parse_args(["--impl", "reference", "--steps", "1", "--warmup", "0"]))
    assert capsys.readouterr().out == ""                     # other ranks exit without work


def test_plan_stats_without_plans():
    # replica sets with no plan-based policy (e.g. --policies P2C) build no plans
    import numpy as np
    import bench
    assert bench.plan_stats(np.zeros((3, 0))) == {"median": None, "max": None, "builds_per_step": 0}
    st = bench.plan_stats(np.array([[1.0, 3.0], [2.0, 5.0]]))
    assert st == {"median": 2.5, "max": 5.0, "builds_per_step": 2}


def test_schedule_defaults_follow_interval_size():
    # a CUDA graph and long replay groups for many short intervals; the Large sweep's
    # ~1M-request intervals run without a graph, two intervals per replay call
    import tracegen as tg
    import bench
    got = {}
    for name in ("tiny", "70b", "8b", "burst", "large"):
        args = bench.parse_args(["--config", name])
        bench.auto_schedule(args, tg.Trace(tg.CONFIGS[name]))
        got[name] = (args.graph, args.trace_min_interval, args.replay_group)
    assert got["large"] == (False, 65536, 2)
    assert got["8b"] == (True, 0, 13)
    assert got["70b"][0] and got["burst"][0] and got["tiny"][0]
    args = bench.parse_args(["--config", "8b", "--no-graph", "--replay-group", "1"])
    bench.auto_schedule(args, tg.Trace(tg.CONFIGS["8b"]))
    assert (args.graph, args.trace_min_interval, args.replay_group) == (False, 65536, 1)
    args = bench.parse_args(["--sm-split", "8"])
    assert args.graph is False
