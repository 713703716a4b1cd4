"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle.

Tolerance for attention outputs (bf16 vs float64): max abs <= 1e-2, mean abs
<= 1e-3.  KV pages: bit-exact.  Sizes span several tiles, ragged tails,
multi-split decodes and the degenerate cases (ctx = 0, p = 1, no decodes,
no prefill).
"""
import numpy as np
import pytest

from tests import harness
from tests.harness import MAX_ABS, MEAN_ABS, Case

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _ok(err):
    assert err["finite"], "non-finite outputs"
    assert err["max_abs"] <= MAX_ABS, err
    assert err["mean_abs"] <= MEAN_ABS, err
    assert err["pools_exact"], "KV pages differ from the oracle"


def test_small_config_full_parity():
    case = harness.config_case("qwen3-0.6b-attn-1layer-small")
    res = case.run_gpu()
    _ok(case.check(res))


@pytest.mark.parametrize("ctx", [[0], [1, 15, 16, 17], list(range(16)), [20, 33, 47, 62, 63, 64, 65],
                                 [5, 300, 1023, 1024, 2049], [4095, 4096, 7000]])
@pytest.mark.parametrize("hq", [16, 64])
def test_decode_only(ctx, hq):
    case = Case(hq, ctx, seed=len(ctx) + hq)
    res = case.run_gpu()
    _ok(case.check(res))


@pytest.mark.parametrize("hq", [8, 16, 32, 64])
def test_decode_n_rep(hq):
    case = Case(hq, [33, 700, 129], seed=hq)
    _ok(case.check(case.run_gpu()))


@pytest.mark.parametrize("split", [128, 256, 4096])
def test_decode_split_sizes(split):
    from paper_2609_38386_gb300 import MX_OPT_SPLIT_KEYS
    case = Case(32, [3000, 129, 128, 4500], seed=split)
    res = case.run_gpu(options={MX_OPT_SPLIT_KEYS: split})
    assert res["plan"]["split_keys"] == split
    _ok(case.check(res))


@pytest.mark.parametrize("cs,p", [(0, 1), (0, 7), (0, 128), (0, 129), (5, 60), (128, 128),
                                  (200, 300), (1000, 384), (16, 255)])
def test_prefill_only(cs, p):
    case = Case(16, [], chunk_start=cs, p_t=p, prompt_len=cs + p + 9, seed=cs + p)
    _ok(case.check(case.run_gpu()))


@pytest.mark.parametrize("hq", [8, 32, 64])
def test_prefill_n_rep(hq):
    case = Case(hq, [], chunk_start=130, p_t=200, seed=hq)
    _ok(case.check(case.run_gpu()))


@pytest.mark.parametrize("hq,ctx,cs,p", [(16, [64, 256, 100, 200], 128, 128),
                                         (32, [0, 17, 1500, 3333, 64], 77, 257),
                                         (64, [2000, 9], 512, 640)])
def test_mixed(hq, ctx, cs, p):
    case = Case(hq, ctx, chunk_start=cs, p_t=p, seed=hq + p)
    _ok(case.check(case.run_gpu()))


def test_paging_invariance_bit_identical():
    a = Case(16, [100, 37, 900], chunk_start=50, p_t=150, seed=3)
    b = Case(16, [100, 37, 900], chunk_start=50, p_t=150, seed=3)
    # b: same logical contents, different physical pages
    from synth import workload as wl
    lay_b = wl.make_layout(b.geom, b.layout.capacities, seed=999, spare_pages=5)
    ka, va = a.pools0()
    perm_a = a.layout.page_table
    kb = np.zeros(lay_b.pool_shape(), np.uint16)
    vb = np.zeros(lay_b.pool_shape(), np.uint16)
    for s in range(perm_a.shape[0]):
        for lp in range(perm_a.shape[1]):
            if perm_a[s, lp] >= 0:
                kb[lay_b.page_table[s, lp]] = ka[perm_a[s, lp]]
                vb[lay_b.page_table[s, lp]] = va[perm_a[s, lp]]
    b.layout = lay_b
    b.slots = b.it.slots(lay_b)
    b._k_pool0, b._v_pool0 = kb, vb
    ra, rb = a.run_gpu(), b.run_gpu()
    np.testing.assert_array_equal(ra["out"], rb["out"])


def test_run_to_run_deterministic():
    case = Case(32, [1200, 50, 4000], chunk_start=300, p_t=260, seed=5)
    r1, r2 = case.run_gpu(), case.run_gpu()
    np.testing.assert_array_equal(r1["out"], r2["out"])
    np.testing.assert_array_equal(r1["k_pool"], r2["k_pool"])


def test_chunked_equals_unchunked_within_tolerance():
    """Prefilling a prompt in chunks gives the one-shot outputs (the paper's
    exact-output agreement, §5.1), here within the bf16 tolerance."""
    L = 640
    base = Case(16, [], chunk_start=0, p_t=L, seed=11)
    full = base.run_gpu()["out"]
    from paper_2609_38386_gb300 import Context  # noqa: F401
    outs = []
    k0, v0 = base.pools0()
    kp = torch.from_numpy(k0.view(np.int16)).cuda()
    vp = torch.from_numpy(v0.view(np.int16)).cuda()
    ctx = base.make_context()
    pt = torch.from_numpy(base.layout.page_table).cuda()
    for cs in range(0, L, 192):
        p = min(192, L - cs)
        sl = torch.from_numpy(base.slots[cs:cs + p].copy()).cuda()
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a[cs:cs + p]).view(np.int16)).cuda()
        q, k, v = t(base.q), t(base.k), t(base.v)
        out = torch.empty((p, 16, 128), dtype=torch.int16, device="cuda")
        desc = ctx.make_desc(decode_seq_ids=[], decode_ctx_lens=[], prefill_seq_id=0,
                             chunk_start=cs, p_t=p, page_table=pt, slots=sl)
        ctx.mixed_attention(desc, ctx.make_bufs(q, k, v, kp, vp, out))
        ctx.sync_status()
        outs.append(out.cpu().numpy().view(np.uint16))
    ctx.close()
    chunked = np.concatenate(outs)
    diff = np.abs(harness._bf16_to_f64(chunked) - harness._bf16_to_f64(full))
    assert diff.max() <= MAX_ABS and diff.mean() <= MEAN_ABS


def test_kv_append_standalone_bit_exact():
    from paper_2609_38386_gb300 import Context
    rng = np.random.default_rng(0)
    num_pages, n = 40, 37
    ctx = Context(num_q_heads=16, num_pages=num_pages, num_seqs=1, max_pages_per_seq=num_pages,
                  max_tokens=64, max_decodes=1)
    kp = torch.full((num_pages, 8, 16, 128), 0x1234, dtype=torch.int16, device="cuda")
    vp = torch.full((num_pages, 8, 16, 128), 0x4321, dtype=torch.int16, device="cuda")
    slots = rng.choice(num_pages * 16, size=n, replace=False).astype(np.int32)
    slots[[3, 9]] = -1
    k = torch.randint(-30000, 30000, (n, 8, 128), dtype=torch.int16, device="cuda")
    v = torch.randint(-30000, 30000, (n, 8, 128), dtype=torch.int16, device="cuda")
    ctx.kv_append(torch.from_numpy(slots).cuda(), k, v, kp, vp)
    ctx.sync_status()
    want_k = np.full((num_pages, 8, 16, 128), 0x1234, np.int16)
    want_v = np.full((num_pages, 8, 16, 128), 0x4321, np.int16)
    kh, vh = k.cpu().numpy(), v.cpu().numpy()
    for t, s in enumerate(slots):
        if s >= 0:
            want_k[s // 16, :, s % 16] = kh[t]
            want_v[s // 16, :, s % 16] = vh[t]
    np.testing.assert_array_equal(kp.cpu().numpy(), want_k)
    np.testing.assert_array_equal(vp.cpu().numpy(), want_v)
    ctx.close()


def test_bad_page_id_reported_not_trapped():
    from paper_2609_38386_gb300 import MxError
    case = Case(16, [40, 70], seed=1)
    case.layout.page_table = case.layout.page_table.copy()
    case.layout.page_table[1, 1] = case.layout.num_pages + 5   # outside the pool
    with pytest.raises(MxError) as ei:
        case.run_gpu()
    assert "ERANGE_PAGE" in str(ei.value)
    # the context and device stay usable
    ok = Case(16, [40, 70], seed=1)
    _ok(ok.check(ok.run_gpu()))


def test_host_validation_rejects_before_launch():
    from paper_2609_38386_gb300 import MxError
    case = Case(16, [40], chunk_start=10, p_t=20, seed=2)
    ctx = case.make_context()
    d = case.device_inputs()
    bufs = ctx.make_bufs(d["q"], d["k"], d["v"], d["k_pool"], d["v_pool"], d["out"])
    bad = ctx.make_desc(decode_seq_ids=[0], decode_ctx_lens=[10**6], prefill_seq_id=1,
                        chunk_start=10, p_t=20, page_table=d["page_table"], slots=d["slots"])
    with pytest.raises(MxError) as ei:
        ctx.mixed_attention(bad, bufs)
    assert "ECAPACITY" in str(ei.value)
    bad2 = ctx.make_desc(decode_seq_ids=[7], decode_ctx_lens=[10], prefill_seq_id=1,
                         chunk_start=10, p_t=20, page_table=d["page_table"], slots=d["slots"])
    with pytest.raises(MxError):
        ctx.mixed_attention(bad2, bufs)
    ctx.close()


def test_iteration_returns_device_time():
    case = Case(16, [300, 500, 1000], chunk_start=256, p_t=256, seed=4)
    ctx = case.make_context()
    layers = []
    devs = []
    for _ in range(3):
        d = case.device_inputs()
        devs.append(d)
        layers.append(ctx.make_bufs(d["q"], d["k"], d["v"], d["k_pool"], d["v_pool"], d["out"]))
    desc = case.desc(ctx, devs[0])
    us = ctx.iteration(desc, layers)
    assert 0.0 < us < 1e6
    # each layer produced the one-layer result
    ref = case.check({"out": devs[0]["out"].cpu().numpy().view(np.uint16),
                      "k_pool": devs[0]["k_pool"].cpu().numpy().view(np.uint16),
                      "v_pool": devs[0]["v_pool"].cpu().numpy().view(np.uint16)})
    _ok(ref)
    np.testing.assert_array_equal(devs[1]["out"].cpu().numpy(), devs[0]["out"].cpu().numpy())
    ctx.close()


@pytest.mark.parametrize("piece", [1, 2, 3, 5])
@pytest.mark.parametrize("cs,p", [(0, 384), (1000, 300), (77, 200), (9, 120)])
def test_prefill_key_pieces(piece, cs, p):
    """Prefill tiles split along keys into pieces merged by log-sum-exp (a
    prompt's first tile at chunk_start < 16 stays whole, so that its rows of
    few keys keep their exact recomputation)."""
    from paper_2609_38386_gb300 import MX_OPT_PREFILL_PIECE_TILES
    case = Case(32, [900, 3], chunk_start=cs, p_t=p, seed=piece * 7 + cs)
    res = case.run_gpu(options={MX_OPT_PREFILL_PIECE_TILES: piece})
    _ok(case.check(res))


@pytest.mark.parametrize("v_stages", [2, 3])
@pytest.mark.parametrize("hq,ctx,cs,p", [(16, [900, 3, 64], 0, 300), (64, [2000, 17], 1000, 260),
                                         (32, [], 77, 700), (8, [40], 4100, 129)])
def test_value_ring_depths(v_stages, hq, ctx, cs, p):
    """Both value-ring depths give results within tolerance of the oracle and
    identical to each other (the ring depth changes no arithmetic)."""
    from paper_2609_38386_gb300 import MX_OPT_V_STAGES
    case = Case(hq, ctx, chunk_start=cs, p_t=p, seed=v_stages + cs + p)
    res = case.run_gpu(options={MX_OPT_V_STAGES: v_stages})
    _ok(case.check(res))
    other = case.run_gpu(options={MX_OPT_V_STAGES: 5 - v_stages})
    np.testing.assert_array_equal(res["out"], other["out"])


def test_value_ring_option_rejects_other_depths():
    import paper_2609_38386_gb300 as pkg
    from paper_2609_38386_gb300 import MX_OPT_V_STAGES
    ctx = pkg.Context(num_q_heads=16, num_kv_heads=8, num_pages=64, num_seqs=4, max_pages_per_seq=16,
                      max_tokens=256, max_decodes=4)
    for bad in (1, 4, -1):
        with pytest.raises(pkg.MxError):
            ctx.set_option(MX_OPT_V_STAGES, bad)
    ctx.set_option(MX_OPT_V_STAGES, 0)
    ctx.close()


@pytest.mark.parametrize("hq,ctx,cs,p", [(16, [900, 3, 64, 5000, 17], 0, 300), (64, [2000, 17, 12000], 1000, 260),
                                         (8, [40, 700, 700], 4100, 129)])
def test_decode_first_ctas(hq, ctx, cs, p):
    """However many CTAs start on the decode queue (none, one, some, all),
    the results are those of the oracle and identical to each other: the
    claim order changes which SM runs an item, not its arithmetic."""
    from paper_2609_38386_gb300 import MX_OPT_DECODE_CTAS
    case = Case(hq, ctx, chunk_start=cs, p_t=p, seed=hq + cs + p)
    base = case.run_gpu(options={MX_OPT_DECODE_CTAS: -1})
    _ok(case.check(base))
    for d in (0, 1, 37, 65535):
        res = case.run_gpu(options={MX_OPT_DECODE_CTAS: d})
        np.testing.assert_array_equal(res["out"], base["out"])
        np.testing.assert_array_equal(res["k_pool"], base["k_pool"])
        np.testing.assert_array_equal(res["v_pool"], base["v_pool"])


def test_decode_ctas_option_range():
    import paper_2609_38386_gb300 as pkg
    from paper_2609_38386_gb300 import MX_OPT_DECODE_CTAS
    ctx = pkg.Context(num_q_heads=16, num_kv_heads=8, num_pages=64, num_seqs=4, max_pages_per_seq=16,
                      max_tokens=256, max_decodes=4)
    for bad in (-2, 65536):
        with pytest.raises(pkg.MxError):
            ctx.set_option(MX_OPT_DECODE_CTAS, bad)
    for good in (-1, 0, 152):
        ctx.set_option(MX_OPT_DECODE_CTAS, good)
    ctx.close()


def test_prefill_auto_pieces_long_context():
    # a short chunk deep into a long prompt: the planner splits its tiles
    case = Case(16, [2000, 40], chunk_start=6000, p_t=200, seed=8)
    res = case.run_gpu()
    # unsplit: 2 query tiles x 8 pairs of query heads
    assert res["plan"]["n_prefill_items"] > 2 * 8
    _ok(case.check(res))


def test_prefill_pieces_deterministic_and_reusable():
    from paper_2609_38386_gb300 import MX_OPT_PREFILL_PIECE_TILES
    case = Case(16, [], chunk_start=700, p_t=256, seed=9)
    ctx = case.make_context()
    ctx.set_option(MX_OPT_PREFILL_PIECE_TILES, 2)
    r1 = case.run_gpu(ctx=ctx)
    r2 = case.run_gpu(ctx=ctx)        # counters reset by the previous launch
    np.testing.assert_array_equal(r1["out"], r2["out"])
    _ok(case.check(r2))
    ctx.close()


@pytest.mark.parametrize("mode", [2])
def test_iteration_launch_mode_matches(mode):
    """MX_OPT_PDL=2 (layer l+1 starts on the SMs layer l frees) gives the
    bit-identical outputs and KV pages of the default mode, on a plan large
    enough for a grid of every SM, over several layers."""
    from paper_2609_38386_gb300 import MX_OPT_PDL, MX_OPT_SPLIT_KEYS
    rng = np.random.default_rng(12)
    ctxs = [int(c) for c in rng.integers(1500, 4000, size=48)]
    case = Case(16, ctxs, chunk_start=512, p_t=384, seed=21)
    results = {}
    for mode in (1, mode):
        ctx = case.make_context()
        ctx.set_option(MX_OPT_PDL, mode)
        ctx.set_option(MX_OPT_SPLIT_KEYS, 1024)   # the same plan in both modes
        devs = [case.device_inputs() for _ in range(5)]
        layers = [ctx.make_bufs(d["q"], d["k"], d["v"], d["k_pool"], d["v_pool"], d["out"]) for d in devs]
        desc = case.desc(ctx, devs[0])
        for _ in range(3):
            ctx.iteration(desc, layers)
        assert ctx.last_plan()["n_items"] >= torch.cuda.get_device_properties(0).multi_processor_count
        results[mode] = [(d["out"].cpu().numpy(), d["k_pool"].cpu().numpy()) for d in devs]
        ctx.close()
    for (o1, k1), (o2, k2) in zip(results[1], results[mode]):
        np.testing.assert_array_equal(o1, o2)
        np.testing.assert_array_equal(k1, k2)
    ref = case.check({"out": results[mode][0][0].view(np.uint16), "k_pool": results[mode][0][1].view(np.uint16),
                      "v_pool": devs[0]["v_pool"].cpu().numpy().view(np.uint16)})
    _ok(ref)


@pytest.mark.parametrize("mode", [1])
def test_dependent_mode_chains_layers(mode):
    """Dependent order: layer l+1's queries are layer l's output (the same
    buffer), as in a model.  The default launch mode (programmatic dependent
    launch) must give the bit-identical chain of ordinary stream order
    (MX_OPT_PDL=0): a layer that read its queries before the previous layer
    finished would differ."""
    from paper_2609_38386_gb300 import MX_OPT_PDL, MX_OPT_SPLIT_KEYS
    rng = np.random.default_rng(5)
    ctxs = [int(c) for c in rng.integers(1000, 3000, size=40)]
    case = Case(16, ctxs, chunk_start=256, p_t=512, seed=31)
    n_layers = 6
    results = {}
    for m in (0, mode):
        ctx = case.make_context()
        ctx.set_option(MX_OPT_PDL, m)
        ctx.set_option(MX_OPT_SPLIT_KEYS, 1024)
        devs = [case.device_inputs() for _ in range(n_layers)]
        outs = [torch.zeros_like(devs[0]["out"]) for _ in range(n_layers)]
        # layer l+1 reads layer l's output as its q
        qs = [devs[0]["q"]] + outs[:-1]
        layers = [ctx.make_bufs(qs[l], devs[l]["k"], devs[l]["v"], devs[l]["k_pool"], devs[l]["v_pool"], outs[l])
                  for l in range(n_layers)]
        desc = case.desc(ctx, devs[0])
        ctx.iteration(desc, layers)
        assert ctx.last_plan()["n_items"] >= torch.cuda.get_device_properties(0).multi_processor_count
        results[m] = [o.cpu().numpy() for o in outs] + [d["k_pool"].cpu().numpy() for d in devs]
        ctx.close()
    for a, b in zip(results[0], results[mode]):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("split", [0, 512])
def test_decode_long_contexts_equal_parts(split):
    """Decodes long enough to be cut into many equal page-aligned parts
    (65 parts at a 512-key split), merged by log-sum-exp, beside short ones."""
    from paper_2609_38386_gb300 import MX_OPT_SPLIT_KEYS
    case = Case(32, [33000, 17, 4100, 513], seed=40 + split)
    res = case.run_gpu(options={MX_OPT_SPLIT_KEYS: split} if split else None)
    _ok(case.check(res))


def test_prefix_cache_hit_shared_pages():
    """A prefix-cache hit: the chunk's cached prefix is another sequence's
    pages (its page-table row points at the decoding sequence's first 16
    pages, chunk_start = 256), read by both while each appends to its own
    pages.  Outputs within tolerance of the oracle, pages bit-exact."""
    from synth import workload as wl
    geom = wl.Geometry(16)
    ctx = [300, 40]
    layout = wl.make_layout(geom, [c + 1 for c in ctx] + [256 + 200], seed=77, spare_pages=1)
    layout.page_table[2, :16] = layout.page_table[0, :16]
    case = Case(16, ctx, chunk_start=256, p_t=200, seed=9, layout=layout)
    _ok(case.check(case.run_gpu()))


@pytest.mark.parametrize("kind", ["decode_splits", "prefill_pieces"])
def test_bounded_wait_times_out_and_context_recovers(kind):
    """Fault injection for the bounded waits: block 0 claims its first work
    item, then waits on a barrier that nothing arrives at.  The wait gives up
    at the wait limit, the launch reports MX_ETIMEOUT instead of hanging, and
    the next call on the same context is correct although the lost item left
    its arrival counter set (a decode split's merge counter, or a prefill
    piece's)."""
    from paper_2609_38386_gb300 import (MX_OPT_PREFILL_PIECE_TILES, MX_OPT_SPLIT_KEYS,
                                        MX_OPT_TEST_STALL_BLOCK, MX_OPT_WAIT_LIMIT_US, MxError)
    if kind == "decode_splits":
        case = Case(16, [3000, 2500, 1700, 40], seed=31)
        opts = {MX_OPT_SPLIT_KEYS: 512}
    else:
        case = Case(16, [900, 40], chunk_start=700, p_t=256, seed=32)
        opts = {MX_OPT_PREFILL_PIECE_TILES: 2}
    ctx = case.make_context()
    for k_, v_ in opts.items():
        ctx.set_option(k_, v_)
    ctx.set_option(MX_OPT_WAIT_LIMIT_US, 2000)
    ctx.set_option(MX_OPT_TEST_STALL_BLOCK, 1)
    with pytest.raises(MxError) as ei:
        case.run_gpu(ctx=ctx)
    assert "ETIMEOUT" in str(ei.value)
    ctx.set_option(MX_OPT_TEST_STALL_BLOCK, 0)
    ctx.set_option(MX_OPT_WAIT_LIMIT_US, 0)
    r1 = case.run_gpu(ctx=ctx)
    _ok(case.check(r1))
    r2 = case.run_gpu(ctx=ctx)
    np.testing.assert_array_equal(r1["out"], r2["out"])
    ctx.close()


@pytest.mark.parametrize("mode", [1, 2])
def test_bounded_wait_timeout_in_iteration(mode):
    """The same injected stall in every layer launch of an iteration, in both
    launch orders: the iteration reports MX_ETIMEOUT, and the next iteration
    on the context matches a fresh context bit for bit."""
    from paper_2609_38386_gb300 import (MX_OPT_PDL, MX_OPT_SPLIT_KEYS, MX_OPT_TEST_STALL_BLOCK,
                                        MX_OPT_WAIT_LIMIT_US, MxError)
    rng = np.random.default_rng(33)
    ctxs = [int(c) for c in rng.integers(1500, 4000, size=48)]
    case = Case(16, ctxs, chunk_start=512, p_t=384, seed=34)

    def run(ctx):
        devs = [case.device_inputs() for _ in range(3)]
        layers = [ctx.make_bufs(d["q"], d["k"], d["v"], d["k_pool"], d["v_pool"], d["out"]) for d in devs]
        ctx.iteration(case.desc(ctx, devs[0]), layers)
        torch.cuda.synchronize()
        return [d["out"].cpu().numpy() for d in devs]

    ctx = case.make_context()
    ctx.set_option(MX_OPT_PDL, mode)
    ctx.set_option(MX_OPT_SPLIT_KEYS, 1024)
    ctx.set_option(MX_OPT_WAIT_LIMIT_US, 2000)
    ctx.set_option(MX_OPT_TEST_STALL_BLOCK, 1)
    with pytest.raises(MxError) as ei:
        run(ctx)
    assert "ETIMEOUT" in str(ei.value)
    ctx.set_option(MX_OPT_TEST_STALL_BLOCK, 0)
    ctx.set_option(MX_OPT_WAIT_LIMIT_US, 0)
    got = run(ctx)
    ctx.close()
    fresh = case.make_context()
    fresh.set_option(MX_OPT_PDL, mode)
    fresh.set_option(MX_OPT_SPLIT_KEYS, 1024)
    want = run(fresh)
    fresh.close()
    for g, w in zip(got, want):
        np.testing.assert_array_equal(g, w)


def _several_chunks_case(hq, ctxs, chunks, seed):
    """Decodes plus several prompts' chunks (each its own sequence), seeded
    host inputs: returns the layout, tokens, slots and initial pools."""
    import synth
    from synth import workload as wl
    geom = wl.Geometry(hq)
    nd = len(ctxs)
    caps = [c + 1 for c in ctxs] + [cs + p for cs, p in chunks]
    lay = wl.make_layout(geom, caps, seed=seed, spare_pages=1)
    ps = geom.page_size
    slots = [lay.page_table[i, c // ps] * ps + c % ps for i, c in enumerate(ctxs)]
    for f, (cs, p) in enumerate(chunks):
        slots += [lay.page_table[nd + f, (cs + j) // ps] * ps + (cs + j) % ps for j in range(p)]
    n_tok = len(slots)
    base = lambda s: synth.stream_base(seed, s)
    q = synth.fill(base(1), (n_tok, hq, 128))
    k = synth.fill(base(2), (n_tok, 8, 128))
    v = synth.fill(base(3), (n_tok, 8, 128))
    kp = synth.fill(base(4), lay.pool_shape())
    vp = synth.fill(base(5), lay.pool_shape())
    return geom, lay, np.asarray(slots, np.int32), q, k, v, kp, vp


@pytest.mark.parametrize("hq,ctxs,chunks", [
    (16, [300, 40], [(0, 100), (256, 200), (7000, 1)]),
    (32, [], [(128, 128), (77, 300)]),
    (64, [700, 3, 1500], [(1000, 300), (0, 640), (3000, 200), (10, 10)]),
])
def test_several_prefill_chunks(hq, ctxs, chunks):
    """Several prompts' chunks in one launch (each a chunk of its own
    sequence, rows after the decodes chunk by chunk), with ragged lengths,
    a chunk at position 0 and a one-row chunk deep into its prompt (split
    into key pieces): every row against the oracle, KV pages bit-exact."""
    import oracle
    from paper_2609_38386_gb300 import Context
    geom, lay, slots, q, k, v, kp0, vp0 = _several_chunks_case(hq, ctxs, chunks, seed=hq + len(chunks))
    nd = len(ctxs)
    prefills = [(nd + f, cs, p) for f, (cs, p) in enumerate(chunks)]
    ctx = Context(num_q_heads=hq, num_kv_heads=8, num_pages=lay.num_pages, num_seqs=lay.num_seqs,
                  max_pages_per_seq=lay.max_pages, max_tokens=len(slots), max_decodes=max(nd, 1))
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()
    d_q, d_k, d_v, d_kp, d_vp = t(q), t(k), t(v), t(kp0), t(vp0)
    d_out = torch.full((len(slots), hq, 128), 0x7FC1, dtype=torch.int16, device="cuda")
    d_pt, d_sl = torch.from_numpy(lay.page_table).cuda(), torch.from_numpy(slots).cuda()
    desc = ctx.make_desc(decode_seq_ids=list(range(nd)), decode_ctx_lens=ctxs, page_table=d_pt,
                         slots=d_sl, prefills=prefills)
    ctx.mixed_attention(desc, ctx.make_bufs(d_q, d_k, d_v, d_kp, d_vp, d_out))
    ctx.sync_status()
    torch.cuda.synchronize()
    kp, vp = kp0.copy(), vp0.copy()
    want, _ = oracle.mixed_attention(q=q, k=k, v=v, k_pool=kp, v_pool=vp, page_table=lay.page_table,
                                     slots=slots, decode_seq_ids=np.arange(nd), decode_ctx_lens=ctxs,
                                     prefills=prefills)
    got = harness._bf16_to_f64(d_out.cpu().numpy())
    err = np.abs(got - want)
    assert np.all(np.isfinite(got))
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())
    np.testing.assert_array_equal(d_kp.cpu().numpy().view(np.uint16), kp)
    np.testing.assert_array_equal(d_vp.cpu().numpy().view(np.uint16), vp)
    # the same chunks through the multi-layer iteration call
    d_out2 = torch.zeros_like(d_out)
    d_kp2, d_vp2 = t(kp0), t(vp0)
    ctx.iteration(desc, [ctx.make_bufs(d_q, d_k, d_v, d_kp2, d_vp2, d_out2)])
    np.testing.assert_array_equal(d_out2.cpu().numpy(), d_out.cpu().numpy())
    ctx.close()


def test_two_chunks_of_one_sequence_rejected():
    from paper_2609_38386_gb300 import MxError
    case = Case(16, [40], chunk_start=10, p_t=20, seed=2)
    ctx = case.make_context()
    d = case.device_inputs()
    bad = ctx.make_desc(decode_seq_ids=[0], decode_ctx_lens=[40], page_table=d["page_table"],
                        slots=d["slots"], prefills=[(1, 10, 20), (1, 30, 5)])   # one sequence twice
    with pytest.raises(MxError, match="EINVAL"):
        ctx.mixed_attention(bad, ctx.make_bufs(d["q"], d["k"], d["v"], d["k_pool"], d["v_pool"], d["out"]))
    ctx.close()


def test_several_chunks_key_pieces_repeated_calls():
    """Two prompts' short chunks deep into long prompts (positions 6200 and
    7000), so that the tiles of chunk 0 AND of chunk 1 are split into key
    pieces merged by log-sum-exp, beside decodes.  The per-tile arrival
    counters of the pieces live in the context's workspace sets, which
    consecutive launches use in turn (three sets) and each launch resets as
    it merges: six single-layer calls and one four-layer iteration on one
    context reuse every set at least twice, and every row of every call must
    match the oracle (a counter left set would leave a tile unmerged)."""
    import oracle
    from paper_2609_38386_gb300 import Context
    hq, ctxs, chunks = 16, [900, 40, 2500], [(6200, 100), (7000, 100)]
    geom, lay, slots, q, k, v, kp0, vp0 = _several_chunks_case(hq, ctxs, chunks, seed=77)
    nd = len(ctxs)
    prefills = [(nd + f, cs, p) for f, (cs, p) in enumerate(chunks)]
    ctx = Context(num_q_heads=hq, num_kv_heads=8, num_pages=lay.num_pages, num_seqs=lay.num_seqs,
                  max_pages_per_seq=lay.max_pages, max_tokens=len(slots), max_decodes=nd)
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()
    d_q, d_k, d_v, d_kp, d_vp = t(q), t(k), t(v), t(kp0), t(vp0)
    d_pt, d_sl = torch.from_numpy(lay.page_table).cuda(), torch.from_numpy(slots).cuda()
    desc = ctx.make_desc(decode_seq_ids=list(range(nd)), decode_ctx_lens=ctxs, page_table=d_pt,
                         slots=d_sl, prefills=prefills)
    kp, vp = kp0.copy(), vp0.copy()
    want, _ = oracle.mixed_attention(q=q, k=k, v=v, k_pool=kp, v_pool=vp, page_table=lay.page_table,
                                     slots=slots, decode_seq_ids=np.arange(nd), decode_ctx_lens=ctxs,
                                     prefills=prefills)

    def check(out, what):
        got = harness._bf16_to_f64(out.cpu().numpy())
        assert np.all(np.isfinite(got)), what
        err = np.abs(got - want)
        assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (what, err.max(), err.mean())

    for call in range(6):
        d_out = torch.full((len(slots), hq, 128), 0x7FC1, dtype=torch.int16, device="cuda")
        ctx.mixed_attention(desc, ctx.make_bufs(d_q, d_k, d_v, d_kp, d_vp, d_out))
        ctx.sync_status()
        if call == 0:
            # both chunks' tiles (one item per pair of query heads) were cut
            # into key pieces
            n_tiles = sum(-(-p // 128) for _, p in chunks) * (hq // 2)
            assert ctx.last_plan()["n_prefill_items"] >= 2 * n_tiles, ctx.last_plan()
        check(d_out, f"call {call}")
    outs = [torch.full((len(slots), hq, 128), 0x7FC1, dtype=torch.int16, device="cuda") for _ in range(4)]
    ctx.iteration(desc, [ctx.make_bufs(d_q, d_k, d_v, d_kp, d_vp, o) for o in outs])
    for l, o in enumerate(outs):
        check(o, f"iteration layer {l}")
    np.testing.assert_array_equal(d_kp.cpu().numpy().view(np.uint16), kp)
    np.testing.assert_array_equal(d_vp.cpu().numpy().view(np.uint16), vp)
    ctx.close()


@pytest.mark.parametrize("hq", [16, 64])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_short_rows_chunk_start_1_to_15(hq, seed):
    """Chunks starting at positions 1..15 of a prompt: their first rows see
    a few keys, some cached (read from a page) and some the chunk's own.
    With so few keys the bf16 rounding of one weight of P would show, so
    rows of at most 64 keys are computed exactly; every row of every chunk
    length is checked against the oracle."""
    from synth import workload as wl
    geom = wl.Geometry(hq)
    lay = wl.make_layout(geom, [15 + 130 + 9], seed=seed + 100)
    ctx = None
    for cs in range(1, 16):
        for p in (1, 7, 40, 130):
            case = Case(hq, [], chunk_start=cs, p_t=p, seed=1000 * seed + 10 * cs + p, layout=lay)
            if ctx is None:
                from paper_2609_38386_gb300 import Context
                ctx = Context(num_q_heads=hq, num_kv_heads=8, num_pages=lay.num_pages,
                              num_seqs=lay.num_seqs, max_pages_per_seq=lay.max_pages,
                              max_tokens=130, max_decodes=1)
            err = case.check(case.run_gpu(ctx=ctx))
            assert err["finite"] and err["pools_exact"], (cs, p, err)
            assert err["max_abs"] <= MAX_ABS and err["mean_abs"] <= MEAN_ABS, (cs, p, err)
    ctx.close()


@pytest.mark.parametrize("cs", [1, 9, 200])
def test_rescale_in_some_rows_of_a_warp(cs):
    """Rows of one warp disagree on the lazy O rescale: one key of the
    chunk's own tile (row 60, KV head 0) aligns with the queries of every
    even row from 60 on (query heads 0 and 1), so their running max jumps
    far beyond the rescale threshold at that tile while odd rows' does not.
    The rescale reads and writes TMEM with warp-collective instructions,
    which the whole warp must execute together."""
    case = Case(16, [40], chunk_start=cs, p_t=128, seed=71 + cs)
    two = np.uint16(0x4000)                 # bf16 2.0
    nd = case.it.n_decodes
    case.k[nd + 60, 0, :] = two
    rows = np.arange(nd + 60, nd + 128, 2)
    case.q[rows, 0:2, :] = two
    res = case.run_gpu()
    _ok(case.check(res))
