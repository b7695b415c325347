"""Multi-process host logic of bench.py on CPU: world size 2 over gloo (127.0.0.1).

Each rank is an independent replica; the whole-job figure is every rank's bytes over the slowest
rank's time, and only rank 0 runs the reference arm."""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        assert bench.dist_setup() == (world, rank, rank)
        bench.barrier(dist)
        # rank r streamed (r + 1) GB in (r + 1) * 10 ms: the job moved 3 GB in the slowest 20 ms
        gbs, ms_max = bench.replica_throughput(dist, (rank + 1) * 1e9, (rank + 1) * 10.0, device="cpu")
        assert ms_max == 20.0
        assert abs(gbs - 3e9 / 0.020 / 1e9) < 1e-6
        assert bench.max_over_ranks(dist, 5.0 - rank, device="cpu") == 5.0
        assert bench.sum_over_ranks(dist, 1.0, device="cpu") == float(world)
        if rank != 0:
            # the reference arm: only rank 0 runs and prints; the others exit 0 without work
            args = type("A", (), {"seed": 0, "steps": 1, "warmup": 0, "gpus": world})()
            assert bench.run_reference(args, bench.workload_by_name("7b-bf16")) == 0
        out.put((rank, "ok"))
    finally:
        dist.destroy_process_group()


def test_two_replicas_over_gloo():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
    codes = [p.exitcode for p in procs]
    for p in procs:
        if p.is_alive():
            p.kill()
    assert codes == [0, 0], codes
    got = sorted(out.get(timeout=5) for _ in range(2))
    assert got == [(0, "ok"), (1, "ok")]


def test_single_process_helpers_are_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(None, 3.5) == 3.5
    gbs, ms = bench.replica_throughput(None, 13.2e9, 2.0)
    assert ms == 2.0 and abs(gbs - 6600.0) < 1e-9
