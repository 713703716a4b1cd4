"""Reference oracle — TEST INFRASTRUCTURE ONLY.

A plain, slow, float64 CPU restatement of what one layer of the mixed
prefill/decode iteration computes (paper §2.1 Eq. 1 setting, §3.2 unchanged
attention and KV layout), plus the DLFP controller of §3.1 Eq. 2 in
``oracle.controller``.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline leg may import this package.  It shares no code
with the CUDA library under ``paper_2609_38386_gb300/`` and never imports it.

The C part (``mx_oracle.c``) is compiled with the host C compiler into
``liboracle.so`` next to this file, on demand or by ``__graft_entry__.build()``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mx_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile mx_oracle.c into liboracle.so (gcc, OpenMP, -O2, no -march)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC",
                           "-shared", "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32, i64 = ctypes.c_int32, ctypes.c_int64
        lib.oracle_kv_append.restype = ctypes.c_int
        lib.oracle_kv_append.argtypes = [P, P, i64, i32, i32, i32, P, i32, P, P]
        lib.oracle_mixed_attention.restype = ctypes.c_int
        lib.oracle_mixed_attention.argtypes = (
            [i32, i32, i32, i32, i64, i32, P, P, i32, P, P, P, i32]
            + [P] * 7 + [P, i32, P, P, P, i64])
        lib.oracle_max_threads.restype = ctypes.c_int
        _lib = lib
    return _lib


def max_threads() -> int:
    """OpenMP threads the oracle uses (OMP_NUM_THREADS or all host cores)."""
    return int(_load().oracle_max_threads())


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("bf16 tensors are passed as their uint16 bit patterns")
    return a


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def kv_append(k_pool, v_pool, slots, k, v, page_size=16):
    """Apply the KV append in place to host pool copies (a byte copy).

    k_pool/v_pool: uint16 [num_pages][hkv][page_size][head_dim];
    k/v: uint16 [n_tokens][hkv][head_dim]; slots: int32 [n_tokens], <0 skips.
    """
    assert k_pool.flags.c_contiguous and v_pool.flags.c_contiguous
    num_pages, hkv, ps, hd = k_pool.shape
    assert ps == page_size
    slots, k, v = _i32(slots), _u16(k), _u16(v)
    rc = _load().oracle_kv_append(_p(k_pool), _p(v_pool), num_pages, hkv, ps,
                                  hd, _p(slots), len(slots), _p(k), _p(v))
    if rc != 0:
        raise ValueError(f"oracle_kv_append failed: {rc}")


def mixed_attention(*, q, k, v, k_pool, v_pool, page_table, slots,
                    decode_seq_ids, decode_ctx_lens, prefill_seq=-1,
                    chunk_start=0, p_t=0, prefills=None, rows=None):
    """One layer of the mixed iteration in float64 (pools are modified).

    One prefill chunk (prefill_seq, chunk_start, p_t), or several given as
    ``prefills`` = [(seq, chunk_start, p_t), ...] (then p_t must be 0).
    q: uint16 [n_tokens][hq][head_dim]; k, v: uint16
    [n_tokens][hkv][head_dim] with n_tokens = n_decodes + the chunk rows;
    pools: uint16 [num_pages][hkv][page_size][head_dim]; page_table: int32
    [num_seqs][max_pages]; slots: int32 [n_tokens].
    Returns (out float64 [n_rows][hq][head_dim], lse float64 [n_rows][hq])
    for the requested token rows (all rows when ``rows`` is None).
    """
    assert k_pool.flags.c_contiguous and v_pool.flags.c_contiguous
    q, k, v = _u16(q), _u16(k), _u16(v)
    num_pages, hkv, ps, hd = k_pool.shape
    n_tok, hq, hd2 = q.shape
    assert hd2 == hd and k.shape == (n_tok, hkv, hd) and v.shape == k.shape
    nd = len(decode_ctx_lens)
    if prefills is None:
        prefills = [(prefill_seq, chunk_start, p_t)] if p_t > 0 else []
    else:
        assert p_t == 0
    pf_seq = _i32([pf[0] for pf in prefills] or [0])
    pf_cs = _i32([pf[1] for pf in prefills] or [0])
    pf_p = _i32([pf[2] for pf in prefills] or [0])
    assert n_tok == nd + sum(pf[2] for pf in prefills)
    page_table = _i32(page_table)
    slots = _i32(slots)
    dids, dlens = _i32(decode_seq_ids), _i32(decode_ctx_lens)
    rows_a = None if rows is None else _i32(rows)
    n_rows = n_tok if rows_a is None else len(rows_a)
    out = np.zeros((n_rows, hq, hd), dtype=np.float64)
    lse = np.zeros((n_rows, hq), dtype=np.float64)
    max_keys = max([int(x) + 1 for x in dlens] + [pf[1] + pf[2] for pf in prefills] + [1])
    nthr = max_threads()
    scratch = np.zeros(nthr * max_keys, dtype=np.float64)
    rc = _load().oracle_mixed_attention(
        hq, hkv, hd, ps, num_pages, page_table.shape[1], _p(dids), _p(dlens),
        nd, _p(pf_seq), _p(pf_cs), _p(pf_p), len(prefills), _p(page_table), _p(slots), _p(q),
        _p(k), _p(v), _p(k_pool), _p(v_pool), _p(rows_a), n_rows, _p(out),
        _p(lse), _p(scratch), max_keys)
    if rc != 0:
        raise ValueError(f"oracle_mixed_attention failed: {rc}")
    return out, lse
