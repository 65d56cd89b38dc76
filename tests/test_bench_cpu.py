"""Host logic of bench.py: the multi-rank aggregation (gloo, world size 2, CPU) and the
reference arm's rank handling.  No GPU is used."""
import os
import socket
import sys
import types

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        slowest = bench.max_over_ranks(10.0 + 5.0 * rank, world, "cpu")
        out.put((rank, slowest, bench.per_image_us(slowest, steps=4, world=world)))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # both ranks see the slowest rank's time; per-image time divides by all images of the job
    assert res == [(0, 15.0, 15.0 * 1e3 / 8), (1, 15.0, 15.0 * 1e3 / 8)]


def test_single_rank_aggregation():
    assert bench.max_over_ranks(3.25, 1, "cpu") == 3.25
    assert bench.per_image_us(10.0, steps=5, world=1) == pytest.approx(2000.0)


def test_reference_arm_only_rank0_works(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    args = types.SimpleNamespace(gpus=2, steps=1, warmup=3, ref_vit_rows=64)
    assert bench.run_reference(args) == 0
    assert capsys.readouterr().out == ""      # other ranks print nothing and do no work
