"""bench.py's multi-GPU reading is N independent replicas: the whole-job
value is every rank's bytes over the slowest rank's step time.  Checked here
with two gloo ranks on the CPU (the same all-reduces NCCL runs on the GPU
box)."""
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


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r: a step of (1 + r) ms moving 100 (r + 1) MB; e2e 3 + r ms
        res = bench.aggregate_replicas(1.0 + rank, 100e6 * (rank + 1), 3.0 + rank, world)
        bench.barrier(world)
        out.put((rank, res))
    finally:
        dist.destroy_process_group()


def test_two_replicas_aggregate_bytes_over_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        ms, total, gbs, e2e_ms, e2e_gbs = got[r]
        assert ms == pytest.approx(2.0)            # the slower rank's step
        assert total == pytest.approx(300e6)       # both ranks' bytes
        assert gbs == pytest.approx(300e6 / 2e-3 / 1e9)
        assert e2e_ms == pytest.approx(4.0)
        assert e2e_gbs == pytest.approx(300e6 / 4e-3 / 1e9)


def test_one_replica_is_its_own_number():
    sys.path.insert(0, ROOT)
    import bench
    ms, total, gbs, e2e_ms, e2e_gbs = bench.aggregate_replicas(2.0, 1e9, 4.0, 1)
    assert (ms, total, e2e_ms) == (2.0, 1e9, 4.0)
    assert gbs == pytest.approx(500.0) and e2e_gbs == pytest.approx(250.0)
