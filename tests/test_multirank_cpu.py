"""The multi-rank logic of bench.py on CPU: two gloo ranks, no GPU.

Sequences are independent, so N GPUs run N independent batches (weak scaling) with no
collective on the data path; the process group only carries the timing (max over ranks).
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    r, lr, w = bench.dist_env()
    local = [12.5, 20.0][rank]                     # this rank's timed region, ms
    slowest = bench.max_over_ranks(local, w, "cpu")
    value = bench.job_throughput(1000, w, slowest * 1e-3)
    seeds = {bench.rank_cache_seed(1, r, c) for c in range(4)}
    out.put((r, lr, w, slowest, value, sorted(seeds)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_report_the_slowest_and_own_distinct_sequences():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    results = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, lr0, w0, s0, v0, seeds0), (r1, lr1, w1, s1, v1, seeds1) = results
    assert (r0, r1, lr0, lr1, w0, w1) == (0, 1, 0, 1, 2, 2)
    assert s0 == s1 == 20.0                          # max over ranks
    assert v0 == v1 == pytest.approx(2 * 1000 / 0.020)
    assert not set(seeds0) & set(seeds1)             # each rank owns different sequences


def test_reference_arm_other_ranks_do_no_work(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class Args:
        steps, warmup = 10, 3

    bench.run_reference(Args, bench.workload("llama8b_layer_b8_s4096"))
    assert capsys.readouterr().out == ""
