"""The N > 1 path of bench.py on CPU: two gloo ranks, each with its own
instances, combined only through the max-over-ranks timing reduction."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2609_04971_gb300 import synth
    from paper_2609_04971_gb300.workloads import TINY

    # every rank draws different instances from its own seed
    inp = synth.step_inputs(TINY, bench.rank_seed(0, rank), "cpu")
    digest = float(inp["K"].float().sum())
    t = bench.max_over_ranks(10.0 + rank * 5.0, world, torch.device("cpu"))
    digests = [None] * world
    dist.all_gather_object(digests, digest)
    out[rank] = (t, digests, bench.aggregate_throughput(TINY.tokens_per_step(), world, 4, t))
    dist.destroy_process_group()


def test_two_ranks_gloo():
    mp_ctx = mp.get_context("spawn")
    mgr = mp_ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [mp_ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    from paper_2609_04971_gb300.workloads import TINY
    for r in range(2):
        t, digests, value = out[r]
        assert t == 15.0                                   # max over ranks
        assert digests[0] != digests[1]                    # distinct instances per rank
        assert value == pytest.approx(TINY.tokens_per_step() * 2 * 4 / 0.015)
