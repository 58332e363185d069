"""The multi-rank bench arithmetic on CPU: two gloo ranks, each an independent
replica with its own prompt, agree on the slowest rank's time and report the
whole job's tokens over it (no collective on the data path)."""
import os
import socket

import pytest

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, times, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        slowest = bench.max_over_ranks(times[rank], dist, device="cpu")
        out.put((rank, slowest, bench.job_tokens_per_s(world, 3, slowest)))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time():
    mp = pytest.importorskip("torch.multiprocessing")
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    times = [1.25, 2.5]
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, times, out)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, slowest, value in got:
        assert slowest == 2.5
        assert value == pytest.approx(2 * 3 * bench.GEN * bench.BATCH / 2.5)


def test_one_rank_needs_no_collective():
    assert bench.max_over_ranks(0.75) == 0.75
    assert bench.job_tokens_per_s(1, 2, 0.5) == 4 * bench.GEN * bench.BATCH


def test_replicas_get_distinct_prompts():
    import synth
    a = synth.make_prompt(0, bench.N_PH, bench.N_AC, bench.MODEL.phone_vocab)
    b = synth.make_prompt(1, bench.N_PH, bench.N_AC, bench.MODEL.phone_vocab)
    assert any((x != y).any() for x, y in zip(a, b))
