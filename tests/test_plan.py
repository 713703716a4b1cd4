"""The per-iteration work list (host planning, no GPU): every key of every
decode row and every key tile of every chunk query tile is covered exactly
once, in the claim order and record layout that include/mixattn.h documents
for mx_plan_work.  The GPU parity tests check that the kernel computes the
right result from these lists; these tests check the lists themselves over
many more shapes than a GPU run can afford."""
import numpy as np
import pytest

from paper_2609_38386_gb300 import MxError, plan_work

PAGE, TILE = 16, 128
SHORT_KEYS = 64             # rows of at most this many keys take the exact path
PART_SLOTS = 16384          # decode split partials of a context
PRE_PART_SLOTS = 1024       # prefill piece partials of a context


def _decode_items(items):
    """Decode the records of the header's layout into dicts."""
    pre, dec = [], []
    for x, y, z, w in items.astype(np.int64):
        ux = int(x) & 0xFFFFFFFF
        if ux & 0xF == 0:
            pre.append(dict(f=(ux >> 4) & 0xF, heads=((ux >> 8) & 1) + 1, t=y & 0xFFFF, hq=y >> 16,
                            s=z & 0xFFFF, ns=z >> 16, base=int(w)))
        else:
            # 1: a split; 2: a decode of at most 64 keys (exact short path)
            assert ux & 0xF in (1, 2), hex(ux)
            assert ux & 0xF == 1 or int(w) + 1 <= SHORT_KEYS
            dec.append(dict(kind=ux & 0xF, h=(ux >> 4) & 0x7F, s=(ux >> 11) & 0xFFF, len=(ux >> 23) * 16,
                            i=int(y), row=int(z), ctx=int(w)))
    return pre, dec


def _plan(hq, ctxs, cs=0, p=0, sms=152, **kw):
    nd = len(ctxs)
    max_pages = (max([c + 1 for c in ctxs] + [cs + p, 1]) + PAGE - 1) // PAGE
    return plan_work(num_q_heads=hq, num_kv_heads=8, num_pages=100000, num_seqs=nd + 1,
                     max_pages_per_seq=max_pages, max_tokens=nd + p, max_decodes=max(nd, 1),
                     decode_seq_ids=list(range(nd)), decode_ctx_lens=ctxs,
                     prefill_seq_id=nd if p else -1, chunk_start=cs, p_t=p, num_sms=sms, **kw)


def _check(plan, hq, ctxs, cs, p, chunks=None):
    """chunks: [(chunk_start, p_t), ...] for several prefill chunks (else
    the single chunk cs, p)."""
    hkv = 8
    if chunks is None:
        chunks = [(cs, p)] if p else []
    items = plan["items"]
    assert plan["n_items"] == len(items)
    pre, dec = _decode_items(items)
    assert len(pre) == plan["n_prefill_items"]
    # claim order: every prefill item first, heaviest first; then decode
    # splits (and exact short decodes), longest first
    kinds = [(int(x) & 0xF) for x in items[:, 0]]
    n_pre = kinds.count(0)
    assert kinds[:n_pre] == [0] * n_pre
    n_a = [-(-c // TILE) for c, _ in chunks]
    tiles = [(n_a[d["f"]] + d["t"] + 1) * (d["s"] + 1) // d["ns"] -
             (n_a[d["f"]] + d["t"] + 1) * d["s"] // d["ns"] for d in pre]
    assert all(a >= b for a, b in zip(tiles, tiles[1:]))

    # prefill: each (chunk, tile, pair of query heads of one KV head; one head
    # when Hq = Hkv) split into pieces that partition its key tiles
    nh = 2 if hq // hkv >= 2 else 1
    assert all(d["heads"] == nh and d["hq"] % nh == 0 for d in pre)
    seen = {}
    for d in pre:
        seen.setdefault((d["f"], d["t"], d["hq"]), []).append(d)
    assert set(seen) == {(f, t, h) for f, (_, p_) in enumerate(chunks)
                         for t in range(-(-p_ // TILE)) for h in range(0, hq, nh)}
    bases = []
    for (f, t, h), ps in seen.items():
        cs, p = chunks[f]
        ns = ps[0]["ns"]
        assert sorted(x["s"] for x in ps) == list(range(ns))
        assert len({x["base"] for x in ps}) == 1
        n_t = n_a[f] + t + 1
        # the key tiles reach the tile's last row (absolute position); one
        # more, fully masked, only for a ragged last tile whose rows end in
        # the key tile before
        last_pos = cs + min(TILE * t + TILE - 1, p - 1)
        need = last_pos // TILE + 1
        assert n_t == need or (n_t == need + 1 and TILE * t + TILE > p)
        cover = []
        for x in ps:
            cover += range(n_t * x["s"] // ns, n_t * (x["s"] + 1) // ns)
        assert sorted(cover) == list(range(n_t))
        if ns > 1:   # head e of piece s writes partial base + e * ns + s
            bases.append((ps[0]["base"], ps[0]["base"] + nh * ns))
    bases.sort()
    assert all(a[1] <= b[0] for a, b in zip(bases, bases[1:]))
    assert not bases or bases[-1][1] <= PRE_PART_SLOTS

    # decode: each (decode, head) split into page-aligned parts that partition
    # its ctx + 1 keys
    lens = [min(d["len"], ctxs[d["i"]] + 1 - d["s"] * d["len"]) for d in dec]
    assert all(a >= b for a, b in zip(lens, lens[1:]))
    decs = plan["decodes"]
    seen = {}
    for d in dec:
        assert d["row"] == d["i"] and d["ctx"] == ctxs[d["i"]]
        assert d["kind"] == (2 if ctxs[d["i"]] + 1 <= SHORT_KEYS else 1)   # the exact short path
        assert d["len"] % PAGE == 0 and 0 < d["len"] <= 4096
        seen.setdefault((d["i"], d["h"]), []).append(d)
    assert set(seen) == {(i, h) for i in range(len(ctxs)) for h in range(hkv)}
    parts = []
    for (i, h), ss in seen.items():
        ns = int(decs[i][2])
        assert decs[i][0] == i and decs[i][1] == ctxs[i]
        assert sorted(x["s"] for x in ss) == list(range(ns))
        assert len({x["len"] for x in ss}) == 1
        n = ctxs[i] + 1
        cover = []
        for x in ss:
            lo, hi = x["s"] * x["len"], min((x["s"] + 1) * x["len"], n)
            assert lo < hi
            cover += range(lo, hi)
        assert sorted(cover) == list(range(n))
        if ns > 1 and h == 0:
            parts.append((int(decs[i][3]), int(decs[i][3]) + hkv * ns))
    parts.sort()
    assert all(a[1] <= b[0] for a, b in zip(parts, parts[1:]))
    assert not parts or parts[-1][1] <= PART_SLOTS
    return pre, dec


CASES = [
    # hq, decode contexts, chunk_start, p_t
    (16, [0], 0, 0),
    (16, [1, 15, 16, 17, 4095, 4096, 7000], 0, 0),
    (16, [], 0, 1),
    (16, [], 77, 200),
    (32, [900, 3], 1000, 300),
    (16, [2000, 40], 6000, 200),
    (64, [33000, 17, 4100, 513], 0, 0),
    (16, list(range(500, 4100, 113)), 7936, 256),
    (32, [8191] * 64, 4096, 4096),
    (64, [16383] * 128, 0, 8192),
    (8, [100, 3000], 500, 300),          # Hq = Hkv: one query head per prefill item
    (8, [7], 6000, 100),                 # ... and its key pieces
]


@pytest.mark.parametrize("hq,ctxs,cs,p", CASES)
@pytest.mark.parametrize("sms", [152, 20])
def test_work_list_covers_every_key_once(hq, ctxs, cs, p, sms):
    _check(_plan(hq, ctxs, cs, p, sms=sms), hq, ctxs, cs, p)


@pytest.mark.parametrize("seed", range(12))
def test_random_iterations(seed):
    rng = np.random.default_rng(seed)
    hq = int(rng.choice([16, 32, 64]))
    nd = int(rng.integers(0, 40))
    ctxs = [int(c) for c in rng.integers(0, 20000, size=nd)]
    p = int(rng.choice([0, 1, 100, 256, 1000, 2048]))
    cs = int(rng.integers(0, 9000)) if p else 0
    if nd + p == 0:
        p = 1
    kw = dict(split_keys=int(rng.choice([0, 128, 512, 2048])), piece_tiles=int(rng.choice([0, 1, 3, 48])),
              pdl=int(rng.choice([0, 1, 2])))
    _check(_plan(hq, ctxs, cs, p, sms=int(rng.choice([152, 148, 8])), **kw), hq, ctxs, cs, p)


MULTI = [
    # hq, decode contexts, [(chunk_start, p_t), ...]
    (16, [300, 40], [(0, 100), (256, 200), (7000, 1)]),
    (32, [], [(128, 128), (77, 300)]),
    (64, [5000] * 4, [(1000, 300), (0, 4096), (6000, 200), (10, 10)]),
    (16, [1, 2, 3], [(4096, 256)] + [(c, 17) for c in range(0, 15 * 500, 500)]),
]


def _plan_multi(hq, ctxs, chunks, sms=152, **kw):
    nd, npf = len(ctxs), len(chunks)
    n_tok = nd + sum(p for _, p in chunks)
    max_pages = (max([c + 1 for c in ctxs] + [c + p for c, p in chunks] + [1]) + PAGE - 1) // PAGE
    return plan_work(num_q_heads=hq, num_kv_heads=8, num_pages=100000, num_seqs=nd + npf,
                     max_pages_per_seq=max_pages, max_tokens=n_tok, max_decodes=max(nd, 1),
                     decode_seq_ids=list(range(nd)), decode_ctx_lens=ctxs,
                     prefills=[(nd + f, c, p) for f, (c, p) in enumerate(chunks)], num_sms=sms, **kw)


@pytest.mark.parametrize("hq,ctxs,chunks", MULTI)
@pytest.mark.parametrize("piece", [0, 3])
def test_several_chunks_cover_every_key_tile_once(hq, ctxs, chunks, piece):
    _check(_plan_multi(hq, ctxs, chunks, piece_tiles=piece), hq, ctxs, 0, 0, chunks=chunks)


def test_several_chunks_rejections():
    base = dict(num_q_heads=16, num_pages=1000, num_seqs=4, max_pages_per_seq=64, max_tokens=600,
                max_decodes=1, decode_seq_ids=[0], decode_ctx_lens=[5])
    with pytest.raises(MxError, match="EINVAL"):         # two chunks of one sequence
        plan_work(prefills=[(1, 0, 10), (1, 10, 10)], **base)
    with pytest.raises(MxError, match="EINVAL"):         # an empty chunk
        plan_work(prefills=[(1, 0, 0)], **base)
    with pytest.raises(MxError, match="EINVAL"):         # both forms at once
        plan_work(prefills=[(1, 0, 10)], prefill_seq_id=2, p_t=5, **base)
    with pytest.raises(MxError, match="ECAPACITY"):      # more tokens than max_tokens
        plan_work(prefills=[(1, 0, 300), (2, 0, 300)], **base)
    with pytest.raises(MxError, match="EINVAL"):         # more than 16 chunks
        plan_work(**dict(base, num_seqs=40), prefills=[(1 + f, 0, 1) for f in range(17)])


def test_options_are_honoured():
    ctxs = [3000, 2500, 40]
    pl = _plan(16, ctxs, split_keys=512)
    assert pl["split_keys"] == 512
    _, dec = _check(pl, 16, ctxs, 0, 0)
    assert max(d["len"] for d in dec) <= 512
    pl = _plan(16, [10], 700, 256, piece_tiles=2)
    assert pl["piece_tiles"] == 2
    pre, _ = _check(pl, 16, [10], 700, 256)
    assert all(-(-(-(-700 // TILE) + d["t"] + 1) // d["ns"]) <= 2 for d in pre)


def test_automatic_splits_and_pieces():
    # decode-only: splits of [512, 4096] keys, enough of them to fill the SMs
    ctxs = [int(c) for c in np.random.default_rng(3).integers(512, 4096, size=32)]
    pl = _plan(16, ctxs)
    assert 512 <= pl["split_keys"] <= 4096 and pl["split_keys"] % 128 == 0
    assert pl["n_items"] >= 152
    # a short chunk deep into a long prompt is cut into key pieces
    pl = _plan(16, [100], 6000, 200)
    assert pl["n_prefill_items"] > 2 * 8
    # a chunk with enough query tiles to fill the GPU is not (16 tiles x 8
    # pairs of heads)
    pl = _plan(16, [100], 6000, 2048)
    assert pl["n_prefill_items"] == 16 * 8


def _makespan(tiles, m, start=2):
    """List schedule of items (key tiles, claim order) on m SMs, each item
    paying `start` tiles of start-up: the latest finish."""
    import heapq
    h = [0] * m
    for t in tiles:
        heapq.heapreplace(h, h[0] + t + start)
    return max(h)


def test_decode_first_ctas():
    """CTAs that start on the decode queue: none when the prefill items fit
    in one round on the SMs, without decodes, or when the decode is a small
    share of the launch; otherwise at most 24, chosen so that the prefill
    items' schedule on the remaining SMs is within 3 % of theirs on all SMs."""
    rng = np.random.default_rng(5)
    ctxs = [int(c) for c in np.exp(rng.uniform(np.log(1024), np.log(16384), 128))]
    # 1024 rows at 16384, 64 query heads: 8 tiles x 32 head pairs = 256 items
    # of 129..136 key tiles, two rounds on 152 SMs and on 128
    pl = _plan(64, ctxs, 16384, 1024)
    assert pl["decode_first_ctas"] == 24
    assert _plan(64, ctxs, 16384, 1024, sms=100)["decode_first_ctas"] <= 24
    # one round of prefill items (64 on 152 SMs), no decodes, a long chunk
    # beside a few decodes: none
    assert _plan(16, ctxs[:32], 4096, 1024)["decode_first_ctas"] == 0
    assert _plan(64, [], 16384, 1024)["decode_first_ctas"] == 0
    assert _plan(64, ctxs[:8], 24576, 8192)["decode_first_ctas"] == 0
    # the defining property over random iterations
    seen = 0
    for seed in range(12):
        r = np.random.default_rng(100 + seed)
        hq = int(r.choice([16, 32, 64]))
        nd = int(r.integers(1, 129))
        cx = [int(c) for c in r.integers(100, 16384, nd)]
        cs, p = int(r.integers(0, 24576)), int(r.choice([256, 1024, 2048, 4096]))
        pl = _plan(hq, cx, cs, p)
        pre, _ = _check(pl, hq, cx, cs, p)
        n_a = -(-cs // TILE)
        tiles = [(n_a + d["t"] + 1) * (d["s"] + 1) // d["ns"] - (n_a + d["t"] + 1) * d["s"] // d["ns"]
                 for d in pre]
        dq = pl["decode_first_ctas"]
        assert 0 <= dq <= 24
        if dq:
            seen += 1
            assert len(tiles) > 152
            assert _makespan(tiles, 152 - dq) <= 1.03 * _makespan(tiles, 152)
    assert seen > 0


def test_partial_workspace_bounds_the_split_count():
    # 128 decodes x 8 heads at 128-key splits would need 128k partial slots:
    # the planner lengthens the splits until they fit
    ctxs = [16000] * 128
    pl = _plan(64, ctxs, split_keys=128)
    assert pl["split_keys"] > 128
    _check(pl, 64, ctxs, 0, 0)


def test_deterministic():
    a = _plan(32, [900, 3, 5000], 1000, 300)
    b = _plan(32, [900, 3, 5000], 1000, 300)
    np.testing.assert_array_equal(a["items"], b["items"])
    np.testing.assert_array_equal(a["decodes"], b["decodes"])


def test_rejections():
    with pytest.raises(MxError, match="ECAPACITY"):      # more items than the array holds
        _plan(16, [5000] * 8, max_items=4)
    with pytest.raises(MxError, match="EINVAL"):         # seq id outside the page table
        plan_work(num_q_heads=16, num_pages=10, num_seqs=1, max_pages_per_seq=4, max_tokens=4,
                  max_decodes=1, decode_seq_ids=[3], decode_ctx_lens=[5])
    with pytest.raises(MxError, match="ECAPACITY"):      # ctx + 1 beyond the page-table row
        plan_work(num_q_heads=16, num_pages=10, num_seqs=1, max_pages_per_seq=4, max_tokens=4,
                  max_decodes=1, decode_seq_ids=[0], decode_ctx_lens=[64])
    with pytest.raises(MxError, match="EINVAL"):         # n_rep 3 is not supported
        plan_work(num_q_heads=24, num_pages=10, num_seqs=1, max_pages_per_seq=4, max_tokens=4,
                  max_decodes=1, decode_seq_ids=[0], decode_ctx_lens=[5])
    with pytest.raises(MxError, match="EINVAL"):         # split option not a multiple of 128
        _plan(16, [100], split_keys=100)


def test_a_sequence_takes_part_once():
    """A sequence is one decode or one prefill chunk of an iteration, not
    two entries: those would append to and read the same pages in one
    launch.  Each repetition is rejected on the host before any launch."""
    base = dict(num_q_heads=16, num_pages=1000, num_seqs=4, max_pages_per_seq=64, max_tokens=600,
                max_decodes=3)
    with pytest.raises(MxError, match="appears twice"):      # two decodes of sequence 1
        plan_work(decode_seq_ids=[1, 0, 1], decode_ctx_lens=[5, 6, 7], **base)
    with pytest.raises(MxError, match="appears twice"):      # a decode and the chunk
        plan_work(decode_seq_ids=[0, 2], decode_ctx_lens=[5, 6], prefill_seq_id=2, chunk_start=0, p_t=20,
                  **base)
    with pytest.raises(MxError, match="appears twice"):      # a decode and one of several chunks
        plan_work(decode_seq_ids=[0, 3], decode_ctx_lens=[5, 6], prefills=[(1, 0, 10), (3, 0, 10)], **base)
    # distinct sequences plan; a decode-only descriptor's prefill row is ignored
    plan_work(decode_seq_ids=[0, 3], decode_ctx_lens=[5, 6], prefills=[(1, 0, 10), (2, 0, 10)], **base)
    plan_work(decode_seq_ids=[0, 3], decode_ctx_lens=[5, 6], prefill_seq_id=3, p_t=0, **base)



@pytest.mark.parametrize("cs", [0, 5, 15, 16, 200])
def test_first_tile_of_a_prompt_stays_whole(cs):
    """A prompt's first query tile at chunk_start < 16 is never cut into key
    pieces, even with the smallest piece option: its rows of at most 16 keys
    are recomputed exactly from the key tiles the item holds.  Other tiles
    are cut as the option says."""
    pl = _plan(16, [], cs, 300, piece_tiles=1)
    pre, _ = _decode_items(pl["items"])
    n_a = -(-cs // TILE)
    for d in pre:
        n_t = n_a + d["t"] + 1
        want = 1 if (d["t"] == 0 and cs < 16) else n_t
        assert d["ns"] == want, (cs, d)
    _check(pl, 16, [], cs, 300)
