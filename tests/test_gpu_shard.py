"""GPU: KV-head sharding.  The shards of a mixed iteration (each a context
with its KV heads and their query groups, its slice of the pools and of
q/k/v/out) run one after the other on this GPU, as each would on its own
GPU, and their outputs and pages, joined by head, equal the unsharded
launch's bit for bit (split length and piece size fixed in both, so that
every head's work is cut the same way)."""
import numpy as np
import pytest

from paper_2609_38386_gb300 import shard
from tests.harness import Case

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.mark.parametrize("hq,world", [(16, 2), (64, 2), (64, 4), (32, 8)])
def test_kv_head_shards_join_to_the_unsharded_result(hq, world):
    import paper_2609_38386_gb300 as pkg
    case = Case(hq, [700, 12, 2300, 64, 65], chunk_start=384, p_t=300, seed=hq + world)
    opts = {pkg.MX_OPT_SPLIT_KEYS: 1024, pkg.MX_OPT_PREFILL_PIECE_TILES: 65535}
    full = case.run_gpu(options=opts)
    d = case.device_inputs()
    hkv = case.geom.hkv
    lay = case.layout
    outs, kps, vps = [], [], []
    for r in range(world):
        qh, kvh = shard.shard_geometry(hq, hkv, r, world)
        ctx = pkg.Context(num_q_heads=qh[1] - qh[0], num_kv_heads=kvh[1] - kvh[0], num_pages=lay.num_pages,
                          num_seqs=lay.num_seqs, max_pages_per_seq=lay.max_pages, max_tokens=case.n_tokens,
                          max_decodes=case.it.n_decodes)
        for k_, v_ in opts.items():
            ctx.set_option(k_, v_)
        q = shard.take_heads(d["q"], qh, 1)
        k, v = shard.take_heads(d["k"], kvh, 1), shard.take_heads(d["v"], kvh, 1)
        kp, vp = shard.take_heads(d["k_pool"], kvh, 1), shard.take_heads(d["v_pool"], kvh, 1)
        out = torch.empty_like(q)
        ctx.mixed_attention(case.desc(ctx, d), ctx.make_bufs(q, k, v, kp, vp, out))
        ctx.sync_status()
        torch.cuda.synchronize()
        outs.append(out.cpu().numpy())
        kps.append(kp.cpu().numpy())
        vps.append(vp.cpu().numpy())
        ctx.close()
    np.testing.assert_array_equal(np.concatenate(outs, axis=1).view(np.uint16), full["out"])
    np.testing.assert_array_equal(np.concatenate(kps, axis=1).view(np.uint16), full["k_pool"])
    np.testing.assert_array_equal(np.concatenate(vps, axis=1).view(np.uint16), full["v_pool"])
