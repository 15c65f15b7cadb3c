"""The bench's multi-GPU aggregation (one independent replica per rank,
barrier, max-over-ranks time, whole-job throughput), run as world_size-2
gloo process groups on the CPU; and the source hash that keys its recorded
DRAM traffic."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        # each rank "times" its replica differently; the job time is the max
        dist.barrier()
        t = bench.max_over_ranks(10.0 + 5.0 * rank)
        value = bench.job_throughput(1_000_000_000, world, 4, t)
        dist.barrier()
        q.put((rank, t, value))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_throughput_gloo():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, t, value in out:
        assert t == 15.0                       # the slower rank's time
        assert abs(value - 1e9 * 2 * 4 / 15e-3 / 1e9) < 1e-9


def test_single_process_identity():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_throughput(10**9, 1, 1, 1000.0) == 1.0


def test_kernel_hash_ignores_comments_only():
    import bench
    src = 'int f(int x) { // add one\n  return x + 1; /* not "this" */\n}\nconst char *s = "a // b";\n'
    same = '// header\nint f(int x) {\n\n  return x + 1;\n}\nconst char *s = "a // b";  // kept\n'
    other = 'int f(int x) { return x + 2; }\nconst char *s = "a // b";\n'
    assert bench.code_only(src) == bench.code_only(same)
    assert bench.code_only(src) != bench.code_only(other)
    assert '"a // b"' in bench.code_only(src)
