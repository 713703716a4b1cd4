"""KV-head sharding: the host mapping (CPU), and its use by two gloo ranks
that each take their share of every head-indexed tensor and gather the
shares back (no GPU; the kernels of the shards are checked on a GPU in
tests/test_gpu_shard.py)."""
import os
import socket

import numpy as np
import pytest

from paper_2609_38386_gb300 import shard


@pytest.mark.parametrize("hq,hkv,world", [(16, 8, 2), (64, 8, 2), (64, 8, 8), (32, 8, 4), (24, 3, 2), (8, 8, 3)])
def test_shards_cover_every_head_once_with_whole_groups(hq, hkv, world):
    seen_kv, seen_q = [], []
    for r in range(world):
        (qa, qb), (a, b) = shard.shard_geometry(hq, hkv, r, world)
        assert b > a
        seen_kv += list(range(a, b))
        seen_q += list(range(qa, qb))
        # every query head of the shard reads a KV head of the shard
        for h in range(qa, qb):
            assert a <= h // (hq // hkv) < b
    assert seen_kv == list(range(hkv)) and seen_q == list(range(hq))


def test_shard_rejects_bad_arguments():
    with pytest.raises(ValueError):
        shard.kv_head_range(8, 2, 2)
    with pytest.raises(ValueError):
        shard.kv_head_range(2, 0, 4)
    with pytest.raises(ValueError):
        shard.shard_geometry(12, 8, 0, 2)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, ws, port, out):
    import torch
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws))
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    hq, hkv, n = 16, 8, 5
    q = torch.arange(n * hq * 128, dtype=torch.float32).reshape(n, hq, 128)
    pool = torch.arange(3 * hkv * 16 * 128, dtype=torch.float32).reshape(3, hkv, 16, 128)
    qh, kvh = shard.shard_geometry(hq, hkv, rank, ws)
    mine_q = shard.take_heads(q, qh, 1)
    mine_pool = shard.take_heads(pool, kvh, 1)
    parts_q = [torch.empty_like(mine_q) for _ in range(ws)]
    parts_p = [torch.empty_like(mine_pool) for _ in range(ws)]
    dist.all_gather(parts_q, mine_q)
    dist.all_gather(parts_p, mine_pool)
    out.put((rank, bool(torch.equal(torch.cat(parts_q, 1), q)), bool(torch.equal(torch.cat(parts_p, 1), pool))))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_take_and_rejoin_their_heads():
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in ps)
    for p in ps:
        p.join(timeout=60)
    assert [r[0] for r in res] == [0, 1]
    assert all(r[1] and r[2] for r in res)
