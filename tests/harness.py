"""Parity harness: one layer call on the GPU (through the C ABI) against the
float64 oracle on the same seeded inputs.

Inputs come from the counter-based generator in ``synth``: small tensors are
generated on the host and uploaded; large pools are filled on the device by
the same formula, and the oracle regenerates on the host exactly the pages it
needs.  No oracle input is read back from the GPU.

Tolerance (attention outputs, bf16, against float64): max abs <= 1e-2 and
mean abs <= 1e-3.  KV pages: bit-exact.
"""
from __future__ import annotations

import numpy as np

import oracle
import synth
from synth import workload as wl

MAX_ABS = 1e-2
MEAN_ABS = 1e-3


def _bf16_to_f64(x):
    return synth.bf16_bits_to_f32(np.asarray(x).view(np.uint16)).astype(np.float64)


class Case:
    """One layer call: decodes (seq ids + cached lengths) and one chunk."""

    def __init__(self, hq, ctx_lens, chunk_start=0, p_t=0, prompt_len=None, seed=0,
                 layer=0, salt=0, layout=None, spare_pages=1, device_pools=False):
        self.geom = wl.Geometry(hq)
        ctx = np.asarray(ctx_lens, dtype=np.int32)
        nd = len(ctx)
        if layout is None:
            caps = [int(c) + 1 for c in ctx]
            if p_t > 0:
                caps.append(prompt_len or chunk_start + p_t)
            layout = wl.make_layout(self.geom, caps, seed=seed + 17, spare_pages=spare_pages)
        self.layout = layout
        self.it = wl.IterSpec(0, np.arange(nd, dtype=np.int32), ctx,
                              nd if p_t > 0 else -1, chunk_start, p_t, p_t)
        self.seed, self.layer, self.salt = seed, layer, salt
        self.device_pools = device_pools
        self.slots = self.it.slots(layout)
        self._gen_tokens()

    @classmethod
    def from_config(cls, cfg: wl.SweepConfig, it_index: int, layer=0, device_pools=True):
        it = cfg.iterations()[it_index]
        c = cls.__new__(cls)
        c.geom = cfg.geom
        c.layout = cfg.layout()
        c.it = it
        c.seed, c.layer, c.salt = cfg.seed, layer, 0
        c.device_pools = device_pools
        c.slots = it.slots(c.layout)
        c._gen_tokens()
        return c

    def _gen_tokens(self):
        g, it = self.geom, self.it
        self.q = wl.host_tokens(self.seed, self.layer, synth.STREAM_Q, it, g.hq)
        self.k = wl.host_tokens(self.seed, self.layer, synth.STREAM_K, it, g.hkv)
        self.v = wl.host_tokens(self.seed, self.layer, synth.STREAM_V, it, g.hkv)
        self._k_pool0 = self._v_pool0 = None

    # ---------------------------------------------------------------- inputs
    def _base(self, kind):
        return wl.pool_base(self.seed, self.layer, kind)

    @property
    def n_tokens(self):
        return self.it.n_tokens

    @property
    def pool_shape(self):
        return self.layout.pool_shape()

    def pools0(self):
        """Initial pool contents on the host (small cases only)."""
        if self._k_pool0 is None:
            self._k_pool0 = synth.fill(self._base(synth.STREAM_KPOOL), self.pool_shape)
            self._v_pool0 = synth.fill(self._base(synth.STREAM_VPOOL), self.pool_shape)
        return self._k_pool0, self._v_pool0

    def page_elems(self):
        g = self.geom
        return g.hkv * g.page_size * g.head_dim

    def pages0(self, pages):
        """Initial contents of the listed physical pages, regenerated on the host."""
        pe = self.page_elems()
        shp = (len(pages),) + self.pool_shape[1:]
        kp = synth.values_pages(self._base(synth.STREAM_KPOOL), pages, pe).reshape(shp)
        vp = synth.values_pages(self._base(synth.STREAM_VPOOL), pages, pe).reshape(shp)
        return kp, vp

    # ------------------------------------------------------------------ GPU
    def make_context(self, **kw):
        from paper_2609_38386_gb300 import Context
        lay = self.layout
        return Context(num_q_heads=self.geom.hq, num_kv_heads=self.geom.hkv,
                       num_pages=lay.num_pages, num_seqs=lay.num_seqs,
                       max_pages_per_seq=lay.max_pages, max_tokens=max(self.n_tokens, 1),
                       max_decodes=max(self.it.n_decodes, 1), **kw)

    def device_inputs(self, device="cuda"):
        import torch
        from synth import device as sdev
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(device)
        d = {"q": t(self.q), "k": t(self.k), "v": t(self.v),
             "page_table": torch.from_numpy(self.layout.page_table).to(device),
             "slots": torch.from_numpy(self.slots).to(device)}
        if self.device_pools:
            kp = torch.empty(self.pool_shape, dtype=torch.int16, device=device)
            vp = torch.empty(self.pool_shape, dtype=torch.int16, device=device)
            sdev.fill_(kp, self._base(synth.STREAM_KPOOL))
            sdev.fill_(vp, self._base(synth.STREAM_VPOOL))
        else:
            k0, v0 = self.pools0()
            kp, vp = t(k0), t(v0)
        d["k_pool"], d["v_pool"] = kp, vp
        d["out"] = torch.full((self.n_tokens, self.geom.hq, self.geom.head_dim), 0x7FC1,
                              dtype=torch.int16, device=device)
        return d

    def desc(self, ctx, d):
        it = self.it
        return ctx.make_desc(decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
                             prefill_seq_id=it.prefill_seq, chunk_start=it.chunk_start,
                             p_t=it.p_t, page_table=d["page_table"], slots=d["slots"])

    def run_gpu(self, ctx=None, options=None, d=None, keep=False):
        import torch
        own = ctx is None
        if own:
            ctx = self.make_context()
        for k_, v_ in (options or {}).items():
            ctx.set_option(k_, v_)
        if d is None:
            d = self.device_inputs()
        desc = self.desc(ctx, d)
        bufs = ctx.make_bufs(d["q"], d["k"], d["v"], d["k_pool"], d["v_pool"], d["out"])
        ctx.mixed_attention(desc, bufs)
        ctx.sync_status()
        torch.cuda.synchronize()
        res = {"out": d["out"].cpu().numpy().view(np.uint16), "plan": ctx.last_plan()}
        if not self.device_pools:
            res["k_pool"] = d["k_pool"].cpu().numpy().view(np.uint16)
            res["v_pool"] = d["v_pool"].cpu().numpy().view(np.uint16)
        if keep:
            res["dev"] = d
            res["ctx"] = ctx
        elif own:
            ctx.close()
        return res

    # --------------------------------------------------------------- oracle
    def oracle_full(self):
        k0, v0 = self.pools0()
        kp, vp = k0.copy(), v0.copy()
        it = self.it
        out, lse = oracle.mixed_attention(
            q=self.q, k=self.k, v=self.v, k_pool=kp, v_pool=vp,
            page_table=self.layout.page_table, slots=self.slots,
            decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
            prefill_seq=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t)
        return out, lse, kp, vp

    def needed_pages(self, rows):
        it, lay, ps = self.it, self.layout, self.geom.page_size
        pages = set()
        for r in rows:
            if r < it.n_decodes:
                seq, nk = int(it.decode_seq_ids[r]), int(it.decode_ctx_lens[r]) + 1
            else:
                seq, nk = it.prefill_seq, it.chunk_start + (r - it.n_decodes) + 1
            pages.update(int(x) for x in lay.page_table[seq, :-(-nk // ps)])
        return np.array(sorted(pages), dtype=np.int64)

    def oracle_sampled(self, rows):
        """Oracle on a compact pool holding only the pages the rows read."""
        it, ps = self.it, self.geom.page_size
        pages = self.needed_pages(rows)
        remap = {int(p): i for i, p in enumerate(pages)}
        kp, vp = self.pages0(pages)
        pt = np.vectorize(lambda x: remap.get(int(x), -1), otypes=[np.int32])(self.layout.page_table)
        sl = np.array([remap[int(s) // ps] * ps + int(s) % ps if int(s) // ps in remap else -1
                       for s in self.slots], dtype=np.int32)
        out, lse = oracle.mixed_attention(
            q=self.q, k=self.k, v=self.v, k_pool=kp, v_pool=vp, page_table=pt, slots=sl,
            decode_seq_ids=it.decode_seq_ids, decode_ctx_lens=it.decode_ctx_lens,
            prefill_seq=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t, rows=rows)
        return out, lse, pages, kp, vp

    # ---------------------------------------------------------------- check
    def check(self, res):
        out_ref, _, kp, vp = self.oracle_full()
        got = _bf16_to_f64(res["out"])
        err = np.abs(got - out_ref)
        r = {"max_abs": float(np.nanmax(err)) if err.size else 0.0,
             "mean_abs": float(np.mean(err)) if err.size else 0.0,
             "finite": bool(np.all(np.isfinite(got)))}
        if not r["finite"]:
            r["max_abs"] = float("inf")
        r["pools_exact"] = bool(np.array_equal(res["k_pool"], kp) and np.array_equal(res["v_pool"], vp))
        return r

    def sample_rows(self, n_random=62, seed=0):
        """All decode rows; first, last and random rows of the chunk."""
        it = self.it
        rows = list(range(it.n_decodes))
        if it.p_t:
            rng = np.random.default_rng(seed)
            ch = {it.n_decodes, it.n_decodes + it.p_t - 1}
            ch.update(int(x) for x in rng.integers(it.n_decodes, it.n_tokens,
                                                   size=min(n_random, it.p_t)))
            rows += sorted(ch)
        return rows


def config_case(name, it_index=0, layer=0, device_pools=None):
    cfg = wl.CONFIGS[name]
    small = cfg.single_chunk is not None
    return Case.from_config(cfg, it_index, layer,
                            device_pools=(not small) if device_pools is None else device_pools)


def compare_rows(case, res, rows):
    out_ref, _, _, _, _ = case.oracle_sampled(rows)
    got = _bf16_to_f64(res["out"][rows])
    err = np.abs(got - out_ref)
    if not np.all(np.isfinite(got)):
        return {"max_abs": float("inf"), "mean_abs": float("inf")}
    return {"max_abs": float(err.max()), "mean_abs": float(err.mean())}


def check_pages(case, d, n_untouched=32, seed=0):
    """KV pages after the call: every page the append touched equals its
    initial contents with the new rows written at their slots; a random
    sample of untouched pages is unchanged.  Returns the number of pages
    compared."""
    import torch
    ps = case.geom.page_size
    valid = case.slots >= 0
    toks = np.nonzero(valid)[0]
    sl = case.slots[valid].astype(np.int64)
    touched = np.unique(sl // ps)
    rng = np.random.default_rng(seed)
    others = np.setdiff1d(np.arange(case.layout.num_pages), touched)
    untouched = rng.choice(others, size=min(n_untouched, len(others)), replace=False)
    pages = np.concatenate([touched, untouched])
    kp, vp = case.pages0(pages)
    where = np.searchsorted(touched, sl // ps)
    kp[where, :, sl % ps, :] = case.k[toks]
    vp[where, :, sl % ps, :] = case.v[toks]
    sel = torch.from_numpy(pages).to(d["k_pool"].device)
    got_k = d["k_pool"][sel].cpu().numpy().view(np.uint16)
    got_v = d["v_pool"][sel].cpu().numpy().view(np.uint16)
    assert np.array_equal(got_k, kp) and np.array_equal(got_v, vp), "KV pages differ"
    return len(pages)
