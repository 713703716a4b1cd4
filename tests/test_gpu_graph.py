"""GPU: iterations replayed from a captured CUDA graph (mx_iteration_graph).

A sequence of different iterations (decode-only, chunks of two sizes through
one prompt, decode contexts growing) runs through one captured graph per
value-ring depth and through mx_iteration on a copy of the same state: the
outputs of every iteration and the KV pages at the end must be bit-identical.
Rows of q/k/v past each iteration's tokens hold NaN: the replayed launches
read the buffers up to their capacity and must not let those rows reach a
result.  mx_iteration is checked against the float64 oracle elsewhere.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

NAN16 = 0x7FC1


def _bf16_nan(a):
    u = a.view(np.uint16)
    return ((u & 0x7F80) == 0x7F80) & ((u & 0x7F) != 0)


def _setup(cfg, cap, n_layers):
    import synth
    from synth import device as sdev
    from synth import workload as wl
    lay = cfg.layout()
    g = cfg.geom
    dev = torch.device("cuda")
    layers = []
    for l in range(n_layers):
        kp = torch.empty(lay.pool_shape(), dtype=torch.int16, device=dev)
        vp = torch.empty_like(kp)
        sdev.fill_(kp, wl.pool_base(cfg.seed, l, synth.STREAM_KPOOL))
        sdev.fill_(vp, wl.pool_base(cfg.seed, l, synth.STREAM_VPOOL))
        q = torch.full((cap, g.hq, 128), NAN16, dtype=torch.int16, device=dev)
        k = torch.full((cap, g.hkv, 128), NAN16, dtype=torch.int16, device=dev)
        v = torch.full((cap, g.hkv, 128), NAN16, dtype=torch.int16, device=dev)
        out = torch.full((cap, g.hq, 128), NAN16, dtype=torch.int16, device=dev)
        layers.append({"q": q, "k": k, "v": v, "k_pool": kp, "v_pool": vp, "out": out})
    return lay, layers


def _load_iteration(cfg, it, layers):
    import synth
    from synth import device as sdev
    n = it.n_tokens
    for l, t in enumerate(layers):
        for name, stream in (("q", synth.STREAM_Q), ("k", synth.STREAM_K), ("v", synth.STREAM_V)):
            t[name][n:] = NAN16
            sdev.fill_tokens_(t[name][:n], cfg.seed, l, stream, it)


def _run(cfg, its, graph, v_stages):
    import paper_2609_38386_gb300 as pkg
    cap = max(it.n_tokens for it in its)
    n_layers = 3
    lay, layers = _setup(cfg, cap, n_layers)
    g = cfg.geom
    ctx = pkg.Context(num_q_heads=g.hq, num_kv_heads=g.hkv, num_pages=lay.num_pages, num_seqs=lay.num_seqs,
                      max_pages_per_seq=lay.max_pages, max_tokens=cap, max_decodes=max(len(it.decode_ctx_lens)
                                                                                         for it in its))
    if v_stages:
        ctx.set_option(pkg.MX_OPT_V_STAGES, v_stages)
    pt = torch.from_numpy(lay.page_table).cuda()
    slots = torch.full((cap,), -1, dtype=torch.int32, device="cuda")
    bufs = [ctx.make_bufs(t["q"], t["k"], t["v"], t["k_pool"], t["v_pool"], t["out"]) for t in layers]
    arr = ctx.layer_array(bufs)
    outs = []
    for it in its:
        n = it.n_tokens
        slots[:n] = torch.from_numpy(it.slots(lay)).cuda()
        _load_iteration(cfg, it, layers)
        desc = ctx.make_desc(decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
                             prefill_seq_id=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t,
                             page_table=pt, slots=slots)
        us = ctx.iteration_graph(desc, arr) if graph else ctx.iteration(desc, arr)
        assert us > 0
        outs.append([t["out"][:n].cpu().numpy() for t in layers])
    pools = [(t["k_pool"].cpu().numpy(), t["v_pool"].cpu().numpy()) for t in layers]
    ctx.close()
    return outs, pools


def _sweep():
    from synth import workload as wl
    return wl.SweepConfig("graph-replay-test", hq=16, n_layers=3, n_decodes=12, ctx_lo=40, ctx_hi=700,
                          ctx_dist="uniform", prompt_len=600, chunk_sizes=(0, 256, 128), seed=11)


@pytest.mark.parametrize("v_stages", [0, 2, 3])
def test_graph_replays_equal_iteration(v_stages):
    cfg = _sweep()
    its = cfg.iterations()
    assert len(its) >= 8 and any(it.p_t == 0 for it in its) and any(it.p_t % 128 for it in its)
    ref_outs, ref_pools = _run(cfg, its, graph=False, v_stages=v_stages)
    g_outs, g_pools = _run(cfg, its, graph=True, v_stages=v_stages)
    for i, (a, b) in enumerate(zip(ref_outs, g_outs)):
        for l, (x, y) in enumerate(zip(a, b)):
            assert not _bf16_nan(x).any(), f"NaN in iteration {i} layer {l}"
            np.testing.assert_array_equal(x, y, err_msg=f"iteration {i} layer {l}")
    for (k1, v1), (k2, v2) in zip(ref_pools, g_pools):
        np.testing.assert_array_equal(k1, k2)
        np.testing.assert_array_equal(v1, v2)


def test_graph_recaptures_on_new_page_table():
    """A new page-table tensor (another pointer, the same contents) makes the
    next call capture again; the results stay those of mx_iteration."""
    import paper_2609_38386_gb300 as pkg
    cfg = _sweep()
    its = cfg.iterations()[:4]
    cap = max(it.n_tokens for it in its)
    lay, layers = _setup(cfg, cap, 2)
    g = cfg.geom
    ctx = pkg.Context(num_q_heads=g.hq, num_kv_heads=g.hkv, num_pages=lay.num_pages, num_seqs=lay.num_seqs,
                      max_pages_per_seq=lay.max_pages, max_tokens=cap, max_decodes=12)
    bufs = [ctx.make_bufs(t["q"], t["k"], t["v"], t["k_pool"], t["v_pool"], t["out"]) for t in layers]
    arr = ctx.layer_array(bufs)
    slots = torch.full((cap,), -1, dtype=torch.int32, device="cuda")
    res, tables = [], []
    for i, it in enumerate(its):
        pt = torch.from_numpy(lay.page_table).cuda()   # a new tensor (and pointer) every call
        tables.append(pt)
        n = it.n_tokens
        slots[:n] = torch.from_numpy(it.slots(lay)).cuda()
        _load_iteration(cfg, it, layers)
        desc = ctx.make_desc(decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
                             prefill_seq_id=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t,
                             page_table=pt, slots=slots)
        ctx.iteration_graph(desc, arr)
        res.append([t["out"][:n].cpu().numpy() for t in layers])
    ctx.close()
    ref, _ = _run(cfg, its, graph=False, v_stages=0)
    for a, b in zip(ref, res):
        for x, y in zip(a[:2], b):
            np.testing.assert_array_equal(x, y)
