"""The multi-rank path of bench.py on CPU with gloo, world size 2: ranks share no
data (token-parallel replicas), the timing reduction is a max over ranks, the
whole-job value counts every rank's tokens, and the reference arm runs on
rank 0 only."""
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


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r took (10 + r) ms per step and (20 - r) ms end to end
        got = bench.reduce_max([10.0 + rank, 20.0 - rank])
        dist.barrier()
        q.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_reduce_max_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert out[0] == out[1] == [11.0, 20.0]


def test_reduce_max_single_process_is_identity():
    assert bench.reduce_max([1.5, 2.5]) == [1.5, 2.5]


def test_weak_scaling_value_counts_all_ranks():
    # 2 ranks x 4096 tokens in a 0.1 ms slowest step
    assert bench.whole_job_tokens_per_s(2, 4096, 0.1) == pytest.approx(81.92e6)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    monkeypatch.setenv("RANK", "1")

    class A:
        workload = "tiny_fp32"
        T = 0
        steps = 1
        warmup = 0
        gpus = 2

    assert bench.run_reference(A()) == 0
    assert capsys.readouterr().out == ""
