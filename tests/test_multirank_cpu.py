"""bench.py's N > 1 path on the CPU: two ranks over gloo (127.0.0.1), the way
torchrun launches the bench, one process per GPU.  The layer itself runs as
independent replicas (no data-path collective); what the ranks share is the
timing rule: the job's step time is the slowest rank's (all_reduce MAX) and
its throughput every rank's tokens over that time.  Each rank draws its own
inputs.  The reference arm runs on rank 0 alone; other ranks exit without
work or output."""
import contextlib
import io
import os
import socket
import types

import torch.multiprocessing as mp

import bench

TOKENS = 262144


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks([3.0, 5.0][rank], world, device="cpu")
        q.put((rank, ms, bench.job_throughput(TOKENS, world, ms), bench.rank_seed(rank)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_time_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [5.0, 5.0]  # both ranks report the slowest rank's time
    assert all(r[2] == 2 * TOKENS / 5e-3 for r in res)
    assert res[0][3] != res[1][3]  # each replica has its own inputs


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(4.0, 1) == 4.0
    assert bench.job_throughput(TOKENS, 1, 4.0) == TOKENS / 4e-3


def test_reference_arm_runs_on_rank_zero_only():
    args = types.SimpleNamespace(gpus=2, steps=1, warmup=0)
    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        bench.run_reference(args, 1)
    assert out.getvalue() == ""
