"""Pins for the float64 oracle, independent of the oracle's own code.

Each check fixes the oracle against something the mathematics or the paper
determines: brute-force dense attention over contiguous (unpaged) keys with an
explicit mask, closed forms, invariances (paging, chunking, GQA grouping,
causality) and the paper's worked controller example.  A plausible mistake in
the oracle — a dropped scale, a wrong GQA index, a shifted causal window, a
transposed operand, a missed append — fails at least one of them.
"""
import os

import numpy as np
import pytest
import scipy.special

import oracle
import synth
from oracle import controller as ctl
from synth import workload as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- helpers
def _randn_bf16(rng, shape, scale=1.0):
    return synth.f32_to_bf16_bits(rng.standard_normal(shape) * scale)


def _f(b):
    return synth.bf16_bits_to_f32(b).astype(np.float64)


class Case:
    """Dense ground truth for a few sequences, scattered into a paged pool.

    Each sequence s has dense K/V [cap][hkv][d] (its logical contents after
    this iteration's append).  The pool gets the dense contents at cached
    positions and *garbage* at the positions this iteration appends, so the
    oracle is right only if it applies the append before attending.
    """

    def __init__(self, rng, hq, hkv, d, ps, ctx, chunk_start=0, p_t=0,
                 prompt_len=None, spare=3, perm_seed=7, q_zero=False, prefills=None):
        # prefills: [(chunk_start, p_t, prompt_len or None), ...], one
        # sequence each (rows nd, nd + 1, ... of the page table); the
        # chunk_start / p_t / prompt_len arguments give a single one
        self.hq, self.hkv, self.d, self.ps = hq, hkv, d, ps
        nd = len(ctx)
        caps = [c + 1 for c in ctx]
        self.multi = prefills is not None
        if prefills is None:
            prefills = [(chunk_start, p_t, prompt_len)] if p_t > 0 else []
        self.prefills = [(cs_, p_, pl_ or cs_ + p_) for cs_, p_, pl_ in prefills]
        self.prefill = len(self.prefills) > 0
        caps += [pl_ for _, _, pl_ in self.prefills]
        self.caps = caps
        self.dense_k = [_randn_bf16(rng, (c, hkv, d)) for c in caps]
        self.dense_v = [_randn_bf16(rng, (c, hkv, d)) for c in caps]
        npg = [-(-c // ps) for c in caps]
        self.num_pages = sum(npg) + spare
        prng = np.random.default_rng(perm_seed)
        perm = prng.permutation(self.num_pages).astype(np.int32)
        self.max_pages = max(npg)
        self.pt = np.full((len(caps), self.max_pages), -1, np.int32)
        at = 0
        for s, n in enumerate(npg):
            self.pt[s, :n] = perm[at:at + n]
            at += n
        self.k_pool = _randn_bf16(rng, (self.num_pages, hkv, ps, d), 3.0)
        self.v_pool = _randn_bf16(rng, (self.num_pages, hkv, ps, d), 3.0)
        # cached positions: scatter dense contents; appended ones stay garbage
        for s, cap in enumerate(caps):
            cached = ctx[s] if s < nd else self.prefills[s - nd][0]
            for pos in range(cached):
                pg, off = self.pt[s, pos // ps], pos % ps
                self.k_pool[pg, :, off, :] = self.dense_k[s][pos]
                self.v_pool[pg, :, off, :] = self.dense_v[s][pos]
        self.ctx = np.asarray(ctx, np.int32)
        self.dids = np.arange(nd, dtype=np.int32)
        self.pseq = nd if self.prefill else -1
        self.cs, self.p = chunk_start, p_t
        rows_k, rows_v, slots, pos_of = [], [], [], []
        for i in range(nd):
            rows_k.append(self.dense_k[i][ctx[i]])
            rows_v.append(self.dense_v[i][ctx[i]])
            slots.append(self.pt[i, ctx[i] // ps] * ps + ctx[i] % ps)
            pos_of.append((i, ctx[i]))
        for f, (cs_, p_, _) in enumerate(self.prefills):
            for j in range(p_):
                pos = cs_ + j
                rows_k.append(self.dense_k[nd + f][pos])
                rows_v.append(self.dense_v[nd + f][pos])
                slots.append(self.pt[nd + f, pos // ps] * ps + pos % ps)
                pos_of.append((nd + f, pos))
        n_tok = len(pos_of)
        self.k = np.array(rows_k, np.uint16).reshape(n_tok, hkv, d)
        self.v = np.array(rows_v, np.uint16).reshape(n_tok, hkv, d)
        self.slots = np.array(slots, np.int32)
        self.pos_of = pos_of
        self.q = (np.zeros((n_tok, hq, d), np.uint16) if q_zero
                  else _randn_bf16(rng, (n_tok, hq, d)))

    def run(self, rows=None, k_pool=None, v_pool=None, pt=None):
        kp = (self.k_pool if k_pool is None else k_pool).copy()
        vp = (self.v_pool if v_pool is None else v_pool).copy()
        if self.multi:
            nd = len(self.ctx)
            return oracle.mixed_attention(
                q=self.q, k=self.k, v=self.v, k_pool=kp, v_pool=vp,
                page_table=self.pt if pt is None else pt, slots=self.slots,
                decode_seq_ids=self.dids, decode_ctx_lens=self.ctx,
                prefills=[(nd + f, cs_, p_) for f, (cs_, p_, _) in enumerate(self.prefills)],
                rows=rows)
        return oracle.mixed_attention(
            q=self.q, k=self.k, v=self.v, k_pool=kp, v_pool=vp,
            page_table=self.pt if pt is None else pt, slots=self.slots,
            decode_seq_ids=self.dids, decode_ctx_lens=self.ctx,
            prefill_seq=self.pseq, chunk_start=self.cs, p_t=self.p, rows=rows)

    def brute(self):
        """Dense contiguous attention with an explicit causal mask (numpy)."""
        n_tok = len(self.pos_of)
        out = np.zeros((n_tok, self.hq, self.d))
        rep = self.hq // self.hkv
        for r, (s, pos) in enumerate(self.pos_of):
            K = _f(self.dense_k[s])           # [cap][hkv][d]
            V = _f(self.dense_v[s])
            cap = K.shape[0]
            mask = np.arange(cap) <= pos      # explicit, bottom-right aligned
            for h in range(self.hq):
                qv = _f(self.q[r, h])
                sc = K[:, h // rep, :] @ qv / np.sqrt(self.d)
                sc = np.where(mask, sc, -np.inf)
                w = scipy.special.softmax(sc)
                out[r, h] = w @ V[:, h // rep, :]
        return out


# ---------------------------------------------------------------- bf16
def test_bf16_bits_decode_to_exact_values():
    # bf16 is the high half of an IEEE binary32: fixed values.
    bits = np.array([0x3F80, 0xC000, 0x3F81, 0x0000, 0x4049], np.uint16)
    want = [1.0, -2.0, 1.0078125, 0.0, 3.140625]
    np.testing.assert_array_equal(_f(bits), want)
    # the oracle sees those exact values: q=1 (bits 0x3F80) on d=1 heads
    c = Case(np.random.default_rng(0), 1, 1, 8, 4, [0], q_zero=True)
    c.k[:] = 0
    c.v[:] = 0x4049
    out, _ = c.run()
    np.testing.assert_array_equal(out[0, 0], np.full(8, 3.140625))


# ------------------------------------------------------- brute force pins
@pytest.mark.parametrize("hq,hkv,d,ps", [(2, 1, 8, 4), (4, 2, 8, 16),
                                         (4, 1, 128, 16), (2, 2, 128, 4)])
def test_oracle_equals_dense_bruteforce(hq, hkv, d, ps):
    rng = np.random.default_rng(hq * 100 + hkv * 10 + d + ps)
    c = Case(rng, hq, hkv, d, ps, ctx=[0, 5, 17, 40], chunk_start=13, p_t=11,
             prompt_len=30)
    out, lse = c.run()
    want = c.brute()
    np.testing.assert_allclose(out, want, rtol=0, atol=1e-12)
    assert np.all(np.isfinite(lse))


@pytest.mark.parametrize("hq,hkv,d,ps", [(2, 1, 8, 4), (4, 2, 128, 16)])
def test_several_prefill_chunks_equal_dense_bruteforce(hq, hkv, d, ps):
    """Several prompts' chunks in one iteration (each a chunk of its own
    sequence, rows laid out one chunk after another): every row against
    dense attention over its own sequence's keys, including a chunk at
    position 0 and ragged lengths."""
    rng = np.random.default_rng(hq * 7 + d + ps)
    c = Case(rng, hq, hkv, d, ps, ctx=[0, 21],
             prefills=[(13, 11, 30), (0, 5, None), (40, 1, 41), (3, 9, 20)])
    out, lse = c.run()
    np.testing.assert_allclose(out, c.brute(), rtol=0, atol=1e-12)
    assert np.all(np.isfinite(lse))


def test_several_prefill_chunks_one_at_a_time_bit_identical():
    """Each chunk's rows equal, bit for bit, the rows of an iteration that
    carries that chunk alone: chunks of different sequences do not interact
    (a wrong row-to-chunk mapping or token offset would break this)."""
    rng = np.random.default_rng(11)
    pfs = [(5, 7, 20), (0, 3, None), (17, 6, 23)]
    c = Case(rng, 4, 2, 16, 4, ctx=[3, 9], prefills=pfs)
    full, lse_full = c.run()
    nd = 2
    base = nd
    for f, (cs_, p_, _) in enumerate(pfs):
        rows = list(range(base, base + p_))
        kp, vp = c.k_pool.copy(), c.v_pool.copy()
        sel = list(range(nd)) + rows
        one, lse_one = oracle.mixed_attention(
            q=c.q[sel], k=c.k[sel], v=c.v[sel], k_pool=kp, v_pool=vp, page_table=c.pt,
            slots=c.slots[sel], decode_seq_ids=c.dids, decode_ctx_lens=c.ctx,
            prefill_seq=nd + f, chunk_start=cs_, p_t=p_)
        np.testing.assert_array_equal(full[rows], one[nd:])
        np.testing.assert_array_equal(lse_full[rows], lse_one[nd:])
        np.testing.assert_array_equal(full[:nd], one[:nd])
        base += p_


def test_oracle_rows_subset_equals_full():
    rng = np.random.default_rng(3)
    c = Case(rng, 4, 2, 16, 4, ctx=[3, 9], chunk_start=5, p_t=7)
    full, lse_full = c.run()
    rows = [8, 0, 4, 2]
    sub, lse_sub = c.run(rows=rows)
    np.testing.assert_array_equal(sub, full[rows])
    np.testing.assert_array_equal(lse_sub, lse_full[rows])


# ---------------------------------------------------------- closed forms
def test_single_key_returns_its_value():
    # ctx = 0: the decode sees only its own new key, weight 1.
    rng = np.random.default_rng(11)
    c = Case(rng, 4, 2, 128, 16, ctx=[0, 0])
    out, lse = c.run()
    for r in range(2):
        for h in range(4):
            np.testing.assert_array_equal(out[r, h], _f(c.v[r, h // 2]))
            s = _f(c.q[r, h]) @ _f(c.k[r, h // 2]) / np.sqrt(128)
            assert abs(lse[r, h] - s) < 1e-12


def test_zero_query_gives_mean_of_visible_values():
    rng = np.random.default_rng(12)
    c = Case(rng, 2, 1, 16, 4, ctx=[6, 21], chunk_start=9, p_t=5, q_zero=True)
    out, lse = c.run()
    for r, (s, pos) in enumerate(c.pos_of):
        V = _f(c.dense_v[s][:pos + 1, 0, :])
        for h in range(2):
            np.testing.assert_allclose(out[r, h], V.mean(axis=0), atol=1e-12)
            assert abs(lse[r, h] - np.log(pos + 1)) < 1e-12


def test_identical_value_rows_and_weights_sum_to_one():
    rng = np.random.default_rng(13)
    c = Case(rng, 4, 2, 32, 4, ctx=[2, 30], chunk_start=4, p_t=6)
    row = _randn_bf16(rng, (32,))
    # set every value row (pool and new tokens) to the same vector
    c.v_pool[:] = row
    c.v[:] = row
    out, _ = c.run()
    np.testing.assert_allclose(out, np.broadcast_to(_f(row), out.shape), atol=1e-12)
    # all-ones values: the output equals the sum of the softmax weights
    c.v_pool[:] = 0x3F80
    c.v[:] = 0x3F80
    out, _ = c.run()
    np.testing.assert_allclose(out, 1.0, atol=1e-12)


def test_two_key_closed_form_pins_the_scale():
    # q = a e0, k0 = b e0, k1 = 0: weights exp(ab/sqrt(d)) : 1.
    d = 128
    c = Case(np.random.default_rng(14), 1, 1, d, 16, ctx=[1], q_zero=True)
    a, b = 3.0, 2.0
    c.q[0, 0, 0] = synth.f32_to_bf16_bits(np.float32(a))
    pg = c.pt[0, 0]
    c.k_pool[pg, 0, 0, :] = 0
    c.k_pool[pg, 0, 0, 0] = synth.f32_to_bf16_bits(np.float32(b))
    c.k[0, 0, :] = 0                              # the new key (position 1)
    v0, v1 = _f(c.v_pool[pg, 0, 0]), _f(c.v[0, 0])
    out, lse = c.run()
    e = np.exp(a * b / np.sqrt(d))
    np.testing.assert_allclose(out[0, 0], (e * v0 + v1) / (e + 1), atol=1e-12)
    assert abs(lse[0, 0] - np.log(e + 1)) < 1e-12


# ------------------------------------------------------------ invariances
def test_paging_invariance_bit_identical():
    rng = np.random.default_rng(21)
    c = Case(rng, 4, 2, 32, 4, ctx=[7, 19, 33], chunk_start=10, p_t=9)
    base, lse = c.run()
    # renumber physical pages: pool page x moves to perm[x]
    perm = np.random.default_rng(99).permutation(c.num_pages)
    kp = np.empty_like(c.k_pool)
    vp = np.empty_like(c.v_pool)
    kp[perm] = c.k_pool
    vp[perm] = c.v_pool
    pt = np.where(c.pt >= 0, perm[np.maximum(c.pt, 0)], -1).astype(np.int32)
    saved = c.slots.copy()
    c.slots = (perm[c.slots // c.ps] * c.ps + c.slots % c.ps).astype(np.int32)
    out2, lse2 = c.run(k_pool=kp, v_pool=vp, pt=pt)
    c.slots = saved
    np.testing.assert_array_equal(out2, base)
    np.testing.assert_array_equal(lse2, lse)


@pytest.mark.parametrize("chunk", [1, 3, 16, 17, 128])
def test_chunking_invariance_bit_identical(chunk):
    """Prefilling a prompt in chunks of any size gives the same outputs as
    one unchunked prefill (the paper's exact-output agreement, §4.3/§5.1)."""
    L, hq, hkv, d, ps = 40, 4, 2, 16, 4
    rng = np.random.default_rng(31)
    q = _randn_bf16(rng, (L, hq, d))
    kk = _randn_bf16(rng, (L, hkv, d))
    vv = _randn_bf16(rng, (L, hkv, d))
    npg = -(-L // ps)
    pt = np.random.default_rng(5).permutation(npg + 2)[:npg].astype(np.int32)[None]
    pool_shape = (npg + 2, hkv, ps, d)

    def prefill(chunk_size):
        kp = _randn_bf16(np.random.default_rng(6), pool_shape)
        vp = _randn_bf16(np.random.default_rng(7), pool_shape)
        outs = []
        for cs in range(0, L, chunk_size):
            p = min(chunk_size, L - cs)
            pos = np.arange(cs, cs + p)
            slots = (pt[0, pos // ps] * ps + pos % ps).astype(np.int32)
            o, _ = oracle.mixed_attention(
                q=q[cs:cs + p], k=kk[cs:cs + p], v=vv[cs:cs + p], k_pool=kp,
                v_pool=vp, page_table=pt, slots=slots, decode_seq_ids=[],
                decode_ctx_lens=[], prefill_seq=0, chunk_start=cs, p_t=p)
            outs.append(o)
        return np.concatenate(outs)

    np.testing.assert_array_equal(prefill(chunk), prefill(L))


def test_causal_mask_future_keys_do_not_matter():
    rng = np.random.default_rng(41)
    c = Case(rng, 2, 1, 16, 4, ctx=[], chunk_start=6, p_t=10)
    base, _ = c.run()
    j = 4                                  # row j sits at position 6 + 4 = 10
    # perturb the new key/value of position 11..15: rows <= j unchanged
    c.k[j + 1:] ^= np.uint16(0x0040)
    c.v[j + 1:] ^= np.uint16(0x0040)
    pert, _ = c.run()
    np.testing.assert_array_equal(pert[:j + 1], base[:j + 1])
    assert not np.array_equal(pert[j + 1:], base[j + 1:])
    # perturbing the row's own key changes it: the window is inclusive
    c.k[j] ^= np.uint16(0x0040)
    pert2, _ = c.run()
    assert not np.array_equal(pert2[j], base[j])
    np.testing.assert_array_equal(pert2[:j], base[:j])


def test_gqa_grouping_matches_replicated_kv_heads():
    # Hq=4 over Hkv=2 equals Hq=4 over Hkv=4 with KV heads [0,0,1,1].
    rng = np.random.default_rng(51)
    c = Case(rng, 4, 2, 16, 4, ctx=[5, 12], chunk_start=3, p_t=4)
    out, _ = c.run()
    rep = [0, 0, 1, 1]
    kp4 = np.ascontiguousarray(c.k_pool[:, rep])
    vp4 = np.ascontiguousarray(c.v_pool[:, rep])
    o4, _ = oracle.mixed_attention(
        q=c.q, k=np.ascontiguousarray(c.k[:, rep]),
        v=np.ascontiguousarray(c.v[:, rep]), k_pool=kp4, v_pool=vp4,
        page_table=c.pt, slots=c.slots, decode_seq_ids=c.dids,
        decode_ctx_lens=c.ctx, prefill_seq=c.pseq, chunk_start=c.cs, p_t=c.p)
    np.testing.assert_array_equal(out, o4)
    # and differs from the interleaved mapping h % Hkv
    rep_bad = [0, 1, 0, 1]
    ob, _ = oracle.mixed_attention(
        q=c.q, k=np.ascontiguousarray(c.k[:, rep_bad]),
        v=np.ascontiguousarray(c.v[:, rep_bad]),
        k_pool=np.ascontiguousarray(c.k_pool[:, rep_bad]),
        v_pool=np.ascontiguousarray(c.v_pool[:, rep_bad]),
        page_table=c.pt, slots=c.slots, decode_seq_ids=c.dids,
        decode_ctx_lens=c.ctx, prefill_seq=c.pseq, chunk_start=c.cs, p_t=c.p)
    assert not np.array_equal(out, ob)


def test_append_is_required_for_new_keys():
    # If the oracle read new keys before writing them it would see garbage.
    rng = np.random.default_rng(61)
    c = Case(rng, 2, 1, 16, 4, ctx=[8], chunk_start=4, p_t=3)
    out, _ = c.run()
    np.testing.assert_allclose(out, c.brute(), atol=1e-12)
    kp, vp = c.k_pool.copy(), c.v_pool.copy()
    oracle.kv_append(kp, vp, c.slots, c.k, c.v, page_size=4)
    assert not np.array_equal(kp, c.k_pool)


# ------------------------------------------------------------- KV append
def test_kv_append_bytes_exact_and_untouched_unchanged():
    rng = np.random.default_rng(71)
    num_pages, hkv, ps, d = 9, 2, 4, 8
    kp = np.full((num_pages, hkv, ps, d), 0xA5A5, np.uint16)
    vp = np.full((num_pages, hkv, ps, d), 0x5A5A, np.uint16)
    n = 7
    k = _randn_bf16(rng, (n, hkv, d))
    v = _randn_bf16(rng, (n, hkv, d))
    slots = np.array([0, 35, -1, 17, 3, -5, 22], np.int32)
    kp2, vp2 = kp.copy(), vp.copy()
    oracle.kv_append(kp2, vp2, slots, k, v, page_size=ps)
    want_k, want_v = kp.copy(), vp.copy()
    for t, s in enumerate(slots):
        if s < 0:
            continue
        want_k[s // ps, :, s % ps, :] = k[t]
        want_v[s // ps, :, s % ps, :] = v[t]
    np.testing.assert_array_equal(kp2, want_k)
    np.testing.assert_array_equal(vp2, want_v)
    changed = (kp2 != kp).any(axis=(1, 3))        # [page][offset]
    touched = np.zeros_like(changed)
    for s in slots[slots >= 0]:
        touched[s // ps, s % ps] = True
    assert not (changed & ~touched).any()


def test_kv_append_rejects_out_of_range_slot():
    kp = np.zeros((2, 1, 4, 8), np.uint16)
    with pytest.raises(ValueError):
        oracle.kv_append(kp, kp.copy(), np.array([8], np.int32),
                         np.zeros((1, 1, 8), np.uint16),
                         np.zeros((1, 1, 8), np.uint16), page_size=4)


# -------------------------------------------------------------- controller
def _golden_controller():
    with open(os.path.join(GOLDEN, "dlfp_controller_example.txt")) as f:
        line = [l for l in f if l.strip() and not l.startswith("#")][0]
    return {k: float(v) for k, v in (tok.split("=") for tok in line.split())}


def test_controller_paper_worked_example():
    g = _golden_controller()
    got = ctl.eq2_next_cap(int(g["c_t"]), g["T_ms"], g["observed_ms"],
                           int(g["c_min"]), int(g["c_max"]))
    assert got == int(g["c_next"]) == 4224


def test_controller_clamps_and_quantum():
    assert ctl.eq2_next_cap(3072, 80.0, 1000.0) == 1024        # c_min
    assert ctl.eq2_next_cap(3072, 80.0, 10.0) == 6144          # c_max
    assert ctl.eq2_next_cap(3072, 80.0, 80.0) == 3072          # fixed point
    # 3072 * 80 / 81 = 3034.07 -> largest multiple of 128 below: 2944
    assert ctl.eq2_next_cap(3072, 80.0, 81.0) == 2944
    # an exact multiple stays put: 3072 * 80 / 60 = 4096
    assert ctl.eq2_next_cap(3072, 80.0, 60.0) == 4096


def test_controller_activation_and_reset():
    # no decoder active: reset to c_initial, prefill uncapped
    assert ctl.cycle(4224, 0, True, 50.0) == (None, 3072)
    # decoders but no prefill sharing the cycle: no cap, no update
    assert ctl.cycle(4224, 5, False, 50.0) == (None, 4224)
    # guarded cycle: the current cap applies, Eq. 2 updates it
    assert ctl.cycle(3072, 5, True, 57.51) == (3072, 4224)
