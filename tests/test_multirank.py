"""The bench's multi-GPU path is replicas only (one process per GPU, no
collective on the data path); what crosses ranks is host-side: the barrier,
the max-over-ranks time and the whole-job rate.  Those run here as two gloo
ranks on the CPU (rendezvous on 127.0.0.1); the reference arm's rank gating is
checked too."""
import importlib.util
import json
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mr", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    b = _bench()
    ms = [40.0, 55.0][rank]                      # rank 1 is the slow one
    b.barrier(True, device="cpu")
    job_ms = b.max_over_ranks(ms, True, device="cpu")
    rate = b.whole_job_rate(world, 20, job_ms)
    with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
        json.dump({"job_ms": job_ms, "rate": rate}, f)
    dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_time(tmp_path):
    world, port = 2, _free_port()
    mp.spawn(_rank, args=(world, port, str(tmp_path)), nprocs=world, join=True)
    got = [json.load(open(tmp_path / f"r{r}.json")) for r in range(world)]
    for g in got:
        assert g["job_ms"] == 55.0
        assert g["rate"] == pytest.approx(2 * 20 / 0.055)


def test_single_process_needs_no_process_group():
    b = _bench()
    assert b.max_over_ranks(12.5, False, device="cpu") == 12.5
    assert b.whole_job_rate(1, 10, 500.0) == pytest.approx(20.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    b = _bench()
    monkeypatch.setenv("RANK", "1")

    class Args:
        steps, warmup, gpus = 1, 0, 2
    assert b.reference_arm(Args, None) == 0      # returns before touching the workload
    assert capsys.readouterr().out == ""
