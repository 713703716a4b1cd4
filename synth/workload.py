"""Seeded workload shapes: page layouts, decode contexts and chunk sweeps.

Shapes follow the paper's setting: Qwen3-0.6B/8B/32B attention geometry
(§4.1: 16/32/64 query heads, 8 KV heads, head dim 128, BF16), continuous
batching of |D_t| decodes beside one chunked prefill (§2.1), vLLM's 16-token
pages and an 8192-token batch budget with at most 64 sequences (§4.1).  The
paper's prompts are synthetic token sequences; here every tensor is drawn
from the counter-based generator in ``synth`` instead.

Nothing here computes attention.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

import synth

PAGE = 16
HKV = 8
HEAD_DIM = 128


@dataclasses.dataclass(frozen=True)
class Geometry:
    hq: int
    hkv: int = HKV
    head_dim: int = HEAD_DIM
    page_size: int = PAGE

    @property
    def n_rep(self) -> int:
        return self.hq // self.hkv


@dataclasses.dataclass
class Layout:
    """Physical page assignment of a set of sequences (one per layer pool).

    Sequence s owns pages page_table[s, :n_pages(s)]; physical ids are a
    seeded random permutation of [0, num_pages), so logically adjacent pages
    are scattered through the pool.  Unused table entries hold -1.
    """
    geom: Geometry
    capacities: np.ndarray          # tokens each sequence may hold
    page_table: np.ndarray          # int32 [num_seqs][max_pages]
    num_pages: int

    @property
    def max_pages(self) -> int:
        return int(self.page_table.shape[1])

    @property
    def num_seqs(self) -> int:
        return int(self.page_table.shape[0])

    def slot(self, seq: int, pos) -> np.ndarray:
        """Physical slot page*16+offset of logical positions of a sequence."""
        pos = np.asarray(pos, dtype=np.int64)
        ps = self.geom.page_size
        return (self.page_table[seq, pos // ps].astype(np.int64) * ps
                + pos % ps).astype(np.int32)

    def pool_shape(self):
        g = self.geom
        return (self.num_pages, g.hkv, g.page_size, g.head_dim)


def make_layout(geom: Geometry, capacities, seed: int, spare_pages: int = 0) -> Layout:
    caps = np.asarray(capacities, dtype=np.int64)
    ps = geom.page_size
    n_pages = [max(1, -(-int(c) // ps)) for c in caps]
    total = sum(n_pages) + spare_pages
    rng = np.random.default_rng(seed)
    perm = rng.permutation(total).astype(np.int32)
    max_pages = max(n_pages)
    pt = np.full((len(caps), max_pages), -1, dtype=np.int32)
    at = 0
    for s, n in enumerate(n_pages):
        pt[s, :n] = perm[at:at + n]
        at += n
    return Layout(geom, caps, pt, total)


@dataclasses.dataclass
class IterSpec:
    """One mixed iteration: decodes (seq ids, cached lengths) + one chunk."""
    index: int
    decode_seq_ids: np.ndarray
    decode_ctx_lens: np.ndarray
    prefill_seq: int
    chunk_start: int
    p_t: int
    chunk_size: int                  # the sweep's nominal chunk (0: decode only)

    @property
    def n_decodes(self) -> int:
        return len(self.decode_ctx_lens)

    @property
    def n_tokens(self) -> int:
        return self.n_decodes + self.p_t

    def slots(self, layout: Layout) -> np.ndarray:
        """Slot mapping: decode i writes position ctx_i, chunk row j writes
        chunk_start + j, each through its sequence's page-table row."""
        parts = [layout.slot(int(s), int(c))[None]
                 for s, c in zip(self.decode_seq_ids, self.decode_ctx_lens)]
        if self.p_t:
            parts.append(layout.slot(self.prefill_seq,
                                     np.arange(self.chunk_start,
                                               self.chunk_start + self.p_t)))
        if not parts:
            return np.zeros(0, dtype=np.int32)
        return np.concatenate(parts).astype(np.int32)


@dataclasses.dataclass
class SweepConfig:
    """A chunk-size sweep: decodes beside every chunk of one prompt, in order.

    For each chunk size p (p = 0: one decode-only iteration) the prompt is
    prefilled chunk by chunk from position 0; decode contexts grow by one per
    iteration over the whole sweep.
    """
    name: str
    hq: int
    n_layers: int
    n_decodes: int
    ctx_lo: int
    ctx_hi: int
    ctx_dist: str                    # "uniform" or "loguniform"
    prompt_len: int
    chunk_sizes: tuple
    seed: int = 0
    first_chunk_start: int | None = None   # single-iteration configs
    single_chunk: int | None = None
    hkv: int = HKV                          # KV heads (fewer on a rank of a KV-head-sharded run)

    @property
    def geom(self) -> Geometry:
        return Geometry(self.hq, self.hkv)

    def decode_ctx0(self) -> np.ndarray:
        rng = np.random.default_rng(self.seed)
        if self.ctx_dist == "uniform":
            c = rng.integers(self.ctx_lo, self.ctx_hi + 1, size=self.n_decodes)
        else:
            c = np.exp(rng.uniform(math.log(self.ctx_lo), math.log(self.ctx_hi),
                                   size=self.n_decodes))
            c = np.clip(np.floor(c), self.ctx_lo, self.ctx_hi)
        return c.astype(np.int32)

    def iterations(self):
        ctx0 = self.decode_ctx0()
        dids = np.arange(self.n_decodes, dtype=np.int32)
        pseq = self.n_decodes
        its = []
        if self.single_chunk is not None:
            its.append(IterSpec(0, dids, ctx0.copy(), pseq,
                                self.first_chunk_start, self.single_chunk,
                                self.single_chunk))
            return its
        for p in self.chunk_sizes:
            if p == 0:
                its.append(IterSpec(len(its), dids, ctx0 + len(its), -1, 0, 0, 0))
                continue
            for cs in range(0, self.prompt_len, p):
                pt = min(p, self.prompt_len - cs)
                its.append(IterSpec(len(its), dids, ctx0 + len(its), pseq, cs, pt, p))
        return its

    def layout(self) -> Layout:
        its = self.iterations()
        ctx0 = self.decode_ctx0()
        growth = len(its) + 1
        caps = list(ctx0 + growth) + [self.prompt_len]
        return make_layout(self.geom, caps, seed=self.seed + 1000)


# Workload shapes (attention geometry of the Qwen3 family, §4.1 and §4.2).
SMALL = SweepConfig("qwen3-0.6b-attn-1layer-small", hq=16, n_layers=1,
                    n_decodes=4, ctx_lo=64, ctx_hi=256, ctx_dist="uniform",
                    prompt_len=256, chunk_sizes=(128,), seed=0,
                    first_chunk_start=128, single_chunk=128)
QWEN06B = SweepConfig("qwen3-0.6b-attn-28L-chunk-sweep", hq=16, n_layers=28,
                      n_decodes=32, ctx_lo=512, ctx_hi=4096, ctx_dist="uniform",
                      prompt_len=8192, chunk_sizes=(0, 256, 512, 1024, 2048, 4096),
                      seed=0)
QWEN8B = SweepConfig("qwen3-8b-attn-36L-chunk-sweep", hq=32, n_layers=36,
                     n_decodes=64, ctx_lo=1024, ctx_hi=8192, ctx_dist="loguniform",
                     prompt_len=16384, chunk_sizes=(0, 512, 1024, 2048, 4096),
                     seed=0)
QWEN32B = SweepConfig("qwen3-32b-attn-64L-chunk-sweep", hq=64, n_layers=64,
                      n_decodes=128, ctx_lo=1024, ctx_hi=16384,
                      ctx_dist="loguniform", prompt_len=32768,
                      chunk_sizes=(0, 1024, 2048, 4096, 8192), seed=0)

CONFIGS = {c.name: c for c in (SMALL, QWEN06B, QWEN8B, QWEN32B)}


def algorithmic_work(geom: Geometry, it: IterSpec):
    """Algorithmic bytes and flops of one layer call of an iteration.

    Only unmasked (query, key) pairs and only bytes that must move: each
    cached key/value read once, each new K/V read once and written once, q
    read and out written once, plus the page-table entries.  Split partials
    (workspace) are excluded.
    """
    kv_tok = 2 * geom.hkv * geom.head_dim * 2        # K+V bytes per token
    qo_tok = 2 * geom.hq * geom.head_dim * 2         # q read + out written
    B = 0
    F = 0
    for n in it.decode_ctx_lens.astype(np.int64):
        B += n * kv_tok + 2 * kv_tok + qo_tok + 4 * (-(-(n + 1) // geom.page_size))
        F += 4 * geom.hq * geom.head_dim * (n + 1)
    if it.p_t:
        s, p = it.chunk_start, it.p_t
        B += s * kv_tok + 2 * p * kv_tok + p * qo_tok + 4 * (-(-(s + p) // geom.page_size))
        F += 4 * geom.hq * geom.head_dim * (p * s + p * (p + 1) // 2)
    return int(B), int(F)


def token_parts(seed: int, layer: int, kind: int, it: IterSpec):
    """Where the rows of a per-token input ([n_tokens][heads][128]) come from.

    Returns (row0, n_rows, base, start_row) parts: decode rows come from the
    iteration's own stream, chunk rows from the prompt's stream at the chunk's
    positions, so a prompt's tokens have the same q/k/v however it is chunked.
    """
    parts = []
    if it.n_decodes:
        parts.append((0, it.n_decodes,
                      synth.stream_base(seed, synth.stream_id(layer, kind, it.index + 1)), 0))
    if it.p_t:
        parts.append((it.n_decodes, it.p_t,
                      synth.stream_base(seed, synth.stream_id(layer, kind, 0)), it.chunk_start))
    return parts


def host_tokens(seed: int, layer: int, kind: int, it: IterSpec, heads: int,
                head_dim: int = HEAD_DIM) -> np.ndarray:
    """Host copy of a per-token input, bit-identical to the device fill."""
    w = heads * head_dim
    out = np.empty((it.n_tokens, heads, head_dim), dtype=np.uint16)
    for row0, n, base, start in token_parts(seed, layer, kind, it):
        out[row0:row0 + n] = synth.values_range(base, start * w, n * w).reshape(n, heads, head_dim)
    return out


def pool_base(seed: int, layer: int, kind: int) -> int:
    return synth.stream_base(seed, synth.stream_id(layer, kind, 0))
