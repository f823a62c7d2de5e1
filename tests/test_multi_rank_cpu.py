"""The multi-GPU bench path on CPU ranks (gloo, world size 2): replicas time
independently and the job takes the slowest rank's times and every rank's
tokens.  No GPU: the reduction is the same collective on another backend."""
import multiprocessing as mp
import os
import socket

import bench


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank: int, world: int, port: int, q) -> None:
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank 0: faster timed region, slower end to end; rank 1 the reverse
        got = bench.job_totals(1.0 + rank, 2.0 - 0.5 * rank, 100 + rank, world, "cpu")
        dist.barrier()
        q.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_job_totals_single_rank_passthrough():
    assert bench.job_totals(1.5, 2.5, 7, 1, "cpu") == (1.5, 2.5, 7)


def test_job_totals_over_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        el, ee, tok = out[r]
        assert (el, ee, tok) == (2.0, 2.0, 201), (r, out[r])
