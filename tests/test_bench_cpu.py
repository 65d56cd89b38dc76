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


def test_reference_arm_times_one_part_per_step(monkeypatch, capsys):
    """Rank 0 of the reference arm: step s times part s mod 5 only (a bounded sample per step),
    the per-image value is the sum of the parts' means over the timed steps, and a run with
    fewer steps than parts still measures every part once."""
    import json
    from paper_2608_27206_gb300 import synth

    calls = []

    class FakeTimer:
        PARTS = ("density", "resample", "vit", "llm", "select")
        cost = {"density": 1.0, "resample": 2.0, "vit": 30.0, "llm": 0.5, "select": 0.25}

        def __init__(self, *a, **k):
            self.n = 0

        def time(self, part):
            self.n += 1
            calls.append(part)
            # per-image seconds drift with the call count, so the mean over timed steps is checked
            return {part: self.cost[part] + 0.01 * self.n}, 0.1

        def description(self):
            return "fake"

    class FakePool:
        def close(self):
            pass

        def join(self):
            pass

    monkeypatch.setenv("RANK", "0")
    monkeypatch.setattr(bench, "OracleTimer", FakeTimer)
    monkeypatch.setattr(bench, "oracle_pool", lambda n=None: (FakePool(), 4))
    monkeypatch.setattr(bench, "workload_config", lambda wl, keep: {"workload": "fake"})
    monkeypatch.setattr(synth, "make_workload", lambda *a, **k: object())

    args = types.SimpleNamespace(gpus=1, steps=10, warmup=2, ref_vit_rows=64)
    assert bench.run_reference(args) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert calls == [FakeTimer.PARTS[s % 5] for s in range(12)]
    # timed steps are calls 3..12 (n = 3..12); part p was timed at the n with (n - 1) % 5 == index
    expect = 0.0
    for i, p in enumerate(FakeTimer.PARTS):
        ns = [n for n in range(3, 13) if (n - 1) % 5 == i]
        expect += sum(FakeTimer.cost[p] + 0.01 * n for n in ns) / len(ns)
    assert line["impl"] == "reference" and line["steps"] == 10 and line["warmup"] == 2
    assert line["value"] == pytest.approx(expect * 1e6)
    assert line["ms_per_step"] == pytest.approx(100.0)

    calls.clear()
    args = types.SimpleNamespace(gpus=1, steps=1, warmup=0, ref_vit_rows=64)
    assert bench.run_reference(args) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert calls == list(FakeTimer.PARTS)          # one timed step, four extra to cover every part
    assert set(line["cpu_baseline"]["parts_s_per_image"]) == set(FakeTimer.PARTS)


def test_oracle_timer_parts_on_a_small_workload():
    """The per-part oracle timer behind cpu_baseline and the reference arm, on the 448^2
    workload with a two-process spawn pool: every part reports a time, and a row sample of the
    ViT map is scaled by N / rows (all rows: no scaling)."""
    from paper_2608_27206_gb300 import synth
    wl = synth.make_workload("img448", seed=0)
    pool, _ = bench.oracle_pool(2)
    try:
        full = bench.OracleTimer(wl, 0.1, pool, vit_rows=0)
        seen = {}
        for part in bench.OracleTimer.PARTS:
            t, dt = full.time(part)
            assert dt >= 0.0 and all(v >= 0.0 for v in t.values())
            seen.update(t)
        assert set(seen) == {"density", "resample", "vit", "llm", "select", "gather"}
        n = wl.vit_q.shape[0]
        t, dt = full.time("vit")
        assert t["vit"] == pytest.approx(dt)                     # every row: measured, not scaled
        part = bench.OracleTimer(wl, 0.1, pool, vit_rows=n // 4)
        t, dt = part.time("vit")
        assert t["vit"] == pytest.approx(dt * 4)                 # a quarter of the rows, scaled by 4
        assert "first %d of %d query rows" % (n // 4, n) in part.description()
        assert "all %d query rows" % n in full.description()
    finally:
        pool.close()
        pool.join()
