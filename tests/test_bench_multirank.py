"""The multi-rank logic of bench.py on the CPU with the gloo backend (world size 2):
max-over-ranks timing, the whole-job rate, independent replicas per rank, and the
reference arm running on rank 0 only."""

import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    elapsed = [1.5, 4.0][rank]
    got = bench.dist_max(elapsed)
    out[rank] = (got, bench.replica_workers(rank, 8))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_replicas():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == 4.0 and res[1][0] == 4.0
    assert res[0][1] == list(range(8)) and res[1][1] == list(range(8, 16))


def test_whole_job_rate_and_single_process():
    import bench
    assert bench.whole_job_rate(2, 8, 1000, 10, 2.0) == 2 * 8 * 1000 * 10 / 2.0
    assert bench.dist_max(3.25) == 3.25   # no process group: the value itself


def test_reference_arm_only_on_rank_zero(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = type("A", (), {"config": "tiny-2^20", "steps": 1, "warmup": 0})()
    bench.run_reference(args)
    assert capsys.readouterr().out == ""


def test_cpu_baseline_sample_fits_every_workload():
    """The bounded oracle sample never asks for more coordinates than the workload has."""
    import bench
    import workloads
    w = workloads.get_config("tiny-2^20")
    cpu = bench.cpu_baseline(w, steps=1, d_s=1 << 22)
    assert cpu["value"] > 0 and cpu["kind"] == "oracle"
    assert f"first {w.d} coordinates" in cpu["sample"]
