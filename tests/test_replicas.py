"""The multi-GPU path of bench.py is replicas only: each rank runs its own copy of the layer
(it shards along tokens with no exchange), a barrier brackets the timed region, each timing is
the maximum over ranks, and the reported value is the whole job's throughput.  Checked here on
CPU with two gloo ranks; no GPU and no collective on the data path."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    # rank r timed (r + 1) ms per step and a slower or faster e2e loop
    t = bench.max_over_ranks([1.0 + rank, 5.0 - rank], torch.device("cpu"))
    dist.barrier()
    out[rank] = t
    dist.destroy_process_group()


def test_timings_are_the_max_over_two_gloo_ranks():
    world, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as m:  # no fork of this (multi-threaded) process
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1] == [2.0, 5.0]


def test_single_process_is_the_identity_and_value_counts_every_replica():
    import bench
    assert not dist.is_initialized()
    assert bench.max_over_ranks([3.5, 1.25], torch.device("cpu")) == [3.5, 1.25]
    # 4 replicas of 10 steps of 2e12 ops each in 2 s (the slowest rank) -> 40 TOPS for the job
    assert bench.whole_job_tops(4, 2e12, 10, 2.0) == pytest.approx(40.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                                      "--warmup", "3"])
    assert bench.main() == 0
    assert capsys.readouterr().out == ""  # rank 1 exits without work or output


@pytest.mark.parametrize("workload,unit", [("dllm", "TOPS"), ("quant_dllm", "GB/s")])
def test_reference_arm_line_on_rank_zero(monkeypatch, capsys, workload, unit):
    # the reference arm times the oracle on the host cores and prints the contract's JSON line
    import json
    import bench
    monkeypatch.delenv("RANK", raising=False)
    monkeypatch.delenv("WORLD_SIZE", raising=False)
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--workload", workload, "--steps", "1",
                                      "--warmup", "3", "--ref-seconds", "0.2", "--ref-single-seconds", "0.2"])
    assert bench.main() == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == unit and line["n_gpus"] == 1
    assert line["steps"] == 1 and line["warmup"] == 3 and line["higher_is_better"] is True
    assert line["value"] > 0 and line["config"]["workload"]
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
