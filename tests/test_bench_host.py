"""Host logic of bench.py on the CPU: replica timing over gloo ranks, the reference arm's rank
handling, and the algorithmic byte count the roofline divides by."""
import json
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

import bench  # noqa: E402
from workloads import synth  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, elapsed, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        m = bench.max_over_ranks(elapsed[rank], "cpu")
        out.put((rank, m, bench.replica_throughput(m, 10, 18432, world)))
    finally:
        dist.destroy_process_group()


def test_replicas_take_the_slowest_rank_over_gloo():
    world, elapsed = 2, [40.0, 52.5]
    ctx = mp.get_context("spawn")
    q = ctx.SimpleQueue()
    mp.start_processes(_rank_main, args=(world, _free_port(), elapsed, q), nprocs=world, join=True,
                       start_method="spawn")
    got = sorted(q.get() for _ in range(world))
    for rank, m, (ms, value) in got:
        assert m == 52.5                               # every rank sees the max
        assert ms == pytest.approx(5.25)
        assert value == pytest.approx(2 * 18432 / 5.25e-3)   # whole-job tokens over both replicas


def test_replica_throughput_weak_scaling():
    ms1, v1 = bench.replica_throughput(100.0, 100, 18432, 1)
    ms4, v4 = bench.replica_throughput(100.0, 100, 18432, 4)
    assert ms1 == ms4 == 1.0 and v4 == pytest.approx(4 * v1)


def test_reference_arm_other_ranks_do_no_work(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--gpus", "2", "--steps", "3",
                                      "--warmup", "3"])
    monkeypatch.setattr(bench, "workload", lambda: pytest.fail("rank 1 must not build the workload"))
    bench.main()
    assert capsys.readouterr().out == ""


def test_warmup_below_three_is_rejected(monkeypatch):
    monkeypatch.setattr(sys, "argv", ["bench.py", "--warmup", "2"])
    with pytest.raises(SystemExit):
        bench.main()


def test_algorithmic_bytes_of_the_bench_batch():
    w = bench.workload()
    sn = sum(r.n for r in w.reqs)
    sm = sum(r.m for r in w.reqs)
    assert sn == 32 * 576 and w.d == 4096
    b = bench.algorithmic_bytes(w)
    # Z and T read once (bf16), s_v read once, the K1 kept indices written once
    assert b["score_kernel"] == sn * 4096 * 2 + sm * 4096 * 2 + sn * 4 + 32 * 64 * 4
    assert b["score_kernel"] == 162_430_976
    # stage 2: Q (L rows x 32 heads x 128) and K (64 x 32 x 128) read; K2 rows of hidden, K, V moved
    sl = sum(r.l for r in w.reqs)
    s2 = sl * 32 * 128 * 2 + 32 * 64 * 32 * 128 * 2 + 2 * 32 * 32 * (4096 + 2 * 32 * 128) * 2 + 32 * 32 * 4
    assert b["stage2"] == s2
    assert b["step"] == b["stage1"] + b["stage2"] == 257_675_264


def test_config_names_the_workload():
    w = synth.llava15_batch32(k1=64, ratio=0.5, k2=32)
    cfg = bench.config_of(w)
    json.dumps(cfg)
    assert cfg["workload"].startswith("llava15_576_b32") and cfg["requests"] == 32
