"""The N > 1 path of bench.py on CPU: two gloo ranks, replicas reduced to the slowest rank.

bench.py runs one independent replica per GPU (the method does not shard a frame);
rank 0 reports all ranks' frames over the slowest rank's time.  This checks that
reduction and the whole-job aggregate with world_size 2 over gloo on 127.0.0.1.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ws, r, local = bench.dist_env()
    # rank r pretends its device loop took 1 + r seconds and its e2e loop 5 - r seconds
    dev_s, e2e_s = bench.reduce_max(dist, [1.0 + r, 5.0 - r], torch.device("cpu"))
    value = bench.aggregate([3] * ws, [dev_s])
    q.put((r, ws, local, dev_s, e2e_s, value))
    dist.destroy_process_group()


def test_two_gloo_ranks_report_slowest_rank_and_all_frames():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r, (rank, ws, local, dev_s, e2e_s, value) in enumerate(res):
        assert (rank, ws, local) == (r, 2, r)
        assert dev_s == 2.0 and e2e_s == 5.0          # max over ranks
        assert value == pytest.approx(6 / 2.0)        # 2 ranks x 3 frames over the slowest 2 s


def test_single_rank_needs_no_process_group():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(None, [1.5, 2.5], None) == [1.5, 2.5]
    assert bench.aggregate([4], [2.0]) == 2.0
