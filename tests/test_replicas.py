"""The N>1 bench path: independent replicas, slowest-rank time, whole-job
value — exercised with two gloo ranks on CPU (no GPU, no data-path
collective)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, ws, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(ws), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench
    w, r, local = bench.dist_setup()
    assert (w, r, local) == (ws, rank, rank)
    ms = 100.0 + 50.0 * rank                    # rank 1 is the slower one
    total = bench.max_over_ranks(ms, ws)
    val = bench.whole_job_value(1000, 10, ws, total)
    out.put((rank, total, val, bench.replica_seed_offset(rank)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_replicas_take_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [t for _, t, _, _ in res] == [150.0, 150.0]
    # 2 ranks x 1000 tokens x 10 steps over the slowest rank's 150 ms
    assert all(abs(v - 2 * 1000 * 10 / 0.150) < 1e-6 for _, _, v, _ in res)
    assert [s for _, _, _, s in res] == [0, 1]          # distinct replica seeds


def test_single_rank_is_identity():
    import bench
    assert bench.max_over_ranks(12.5, 1) == 12.5
    assert bench.whole_job_value(100, 2, 1, 1000.0) == 200.0
