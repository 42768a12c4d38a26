"""The N-GPU bench path is N independent replicas (sequences shard with no
exchange): its whole-job figures are the slowest rank's time and the sum of
every rank's tokens.  Checked with two gloo ranks on the CPU."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q, ms_all, toks_all):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = ms_all[rank]
        toks = toks_all[rank]
        q.put((rank, bench.combine_over_ranks(ms, toks, world)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,ms_all,toks_all", [
    (2, [12.5, 17.25], [100, 140]),
    (3, [12.5, 17.25, 9.0], [100, 140, 90]),
    (2, [12.5, 0.0], [100, 0]),          # a rank that had no sequences to verify
])
def test_replicas_take_the_slowest_rank_and_all_tokens(world, ms_all, toks_all):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q, ms_all, toks_all)) for r in range(world)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    want = (max(ms_all), float(sum(toks_all)))
    assert all(v == want for v in got.values()), got


def test_single_rank_passes_through():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.combine_over_ranks(3.5, 7, 1) == (3.5, 7.0)
