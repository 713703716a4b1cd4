"""ctypes binding of libmixattn.so: argument marshalling only.

Every step of the mixed iteration runs in the library's CUDA kernels; this
module converts torch tensors / numpy arrays to pointers and return codes to
exceptions.  If the library is missing the import fails loudly: there is no
CPU path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmixattn.so")

MX_OK = 0
ERRORS = {-1: "MX_EINVAL", -2: "MX_ERANGE_PAGE", -3: "MX_ERANGE_SLOT", -4: "MX_ECUDA",
          -5: "MX_ETIMEOUT", -6: "MX_EDEVICE", -7: "MX_ECAPACITY"}
MX_OPT_SPLIT_KEYS = 1
MX_OPT_GRID = 2
MX_OPT_PREFILL_PIECE_TILES = 3
MX_OPT_PDL = 4
MX_OPT_WAIT_LIMIT_US = 5
MX_OPT_TEST_STALL_BLOCK = 6
MX_OPT_V_STAGES = 7
MX_OPT_DECODE_CTAS = 8

# Names every C-ABI build must export (the declarations of include/mixattn.h).
EXPORTS = ("mx_create", "mx_destroy", "mx_kv_append", "mx_mixed_attention",
           "mx_iteration", "mx_iteration_graph", "mx_sync_status", "mx_error_detail", "mx_set_option",
           "mx_last_plan", "mx_plan_work", "mx_mixed_attention_noalloc",
           "mx_rms_norm", "mx_qk_norm_rope", "mx_silu_mul", "mx_gemm")


class MxError(RuntimeError):
    def __init__(self, code, detail=""):
        self.code = code
        super().__init__(f"{ERRORS.get(code, code)}: {detail}")


class mx_geom(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "num_q_heads", "num_kv_heads", "head_dim", "page_size", "num_pages",
        "num_seqs", "max_pages_per_seq", "max_tokens", "max_decodes")]


class mx_prefill(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("seq_id", "chunk_start", "p_t")]


class mx_iter_desc(ctypes.Structure):
    _fields_ = [("decode_seq_ids", ctypes.c_void_p), ("decode_ctx_lens", ctypes.c_void_p),
                ("n_decodes", ctypes.c_int32), ("prefill_seq_id", ctypes.c_int32),
                ("chunk_start", ctypes.c_int32), ("p_t", ctypes.c_int32),
                ("page_table", ctypes.c_void_p), ("slots", ctypes.c_void_p),
                ("n_prefills", ctypes.c_int32), ("prefills", ctypes.c_void_p)]


def _prefill_array(prefills):
    """[(seq, chunk_start, p_t), ...] -> (C array or None, count)."""
    if not prefills:
        return None, 0
    arr = (mx_prefill * len(prefills))(*[mx_prefill(int(a), int(b), int(c)) for a, b, c in prefills])
    return arr, len(prefills)


class mx_layer_bufs(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in ("q", "k", "v", "k_pool", "v_pool", "out")]


_lib = None


def load():
    """Load the in-tree library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} not found: build it with "
                              "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(LIB_PATH)
        P, i32, i64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        sig = {
            "mx_create": [ctypes.POINTER(P), ctypes.POINTER(mx_geom), ctypes.c_int],
            "mx_destroy": [P],
            "mx_kv_append": [P, P, i32, P, P, P, P, P],
            "mx_mixed_attention": [P, ctypes.POINTER(mx_iter_desc),
                                   ctypes.POINTER(mx_layer_bufs), P],
            "mx_iteration": [P, ctypes.POINTER(mx_iter_desc), i32,
                             ctypes.POINTER(mx_layer_bufs), ctypes.POINTER(ctypes.c_float), P],
            "mx_iteration_graph": [P, ctypes.POINTER(mx_iter_desc), i32,
                                   ctypes.POINTER(mx_layer_bufs), ctypes.POINTER(ctypes.c_float), P],
            "mx_sync_status": [P, P],
            "mx_error_detail": [P, ctypes.c_char_p, i32],
            "mx_set_option": [P, i32, i64],
            "mx_last_plan": [P, ctypes.POINTER(i32), ctypes.POINTER(i32), ctypes.POINTER(i32)],
            "mx_mixed_attention_noalloc": [ctypes.POINTER(mx_geom), ctypes.POINTER(mx_iter_desc),
                                           ctypes.POINTER(mx_layer_bufs), P, ctypes.c_char_p, i32],
            "mx_plan_work": [ctypes.POINTER(mx_geom), ctypes.POINTER(mx_iter_desc), i32, i32, i32, i32,
                             P, i32, P, P, ctypes.c_char_p, i32],
            "mx_rms_norm": [P, P, P, i32, i32, ctypes.c_float, P],
            "mx_qk_norm_rope": [P, P, P, P, P, P, P, i32, i32, i32, ctypes.c_float, ctypes.c_float, P],
            "mx_silu_mul": [P, P, i32, i32, P],
            "mx_gemm": [P, P, P, i32, i32, i32, i32, P],
        }
        for name, args in sig.items():
            f = getattr(lib, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        _lib = lib
    return _lib


def plan_work(*, num_q_heads, num_kv_heads=8, num_pages, num_seqs, max_pages_per_seq,
              max_tokens, max_decodes, decode_seq_ids, decode_ctx_lens, prefill_seq_id=-1,
              chunk_start=0, p_t=0, prefills=None, num_sms=152, split_keys=0, piece_tiles=0,
              pdl=1, max_items=1 << 16):
    """The work list a launch would run (host only, no device): items
    int32 [n, 4] in claim order, decodes int32 [n_decodes, 4] and the counts
    (n_items, prefill items, split_keys, piece_tiles, CTAs that start on the
    decode queue)."""
    lib = load()
    geom = mx_geom(num_q_heads, num_kv_heads, 128, 16, num_pages, num_seqs, max_pages_per_seq,
                   max_tokens, max_decodes)
    ids = np.ascontiguousarray(np.asarray(decode_seq_ids, dtype=np.int32))
    lens = np.ascontiguousarray(np.asarray(decode_ctx_lens, dtype=np.int32))
    pf_arr, n_pf = _prefill_array(prefills)
    desc = mx_iter_desc(ids.ctypes.data if len(ids) else None, lens.ctypes.data if len(lens) else None,
                        len(lens), int(prefill_seq_id), int(chunk_start), int(p_t), None, None,
                        n_pf, ctypes.cast(pf_arr, ctypes.c_void_p) if pf_arr is not None else None)
    items = np.zeros((max(max_items, 1), 4), np.int32)
    decs = np.zeros((max(len(lens), 1), 4), np.int32)
    counts = np.zeros(5, np.int32)
    err = ctypes.create_string_buffer(512)
    rc = lib.mx_plan_work(ctypes.byref(geom), ctypes.byref(desc), int(num_sms), int(split_keys),
                          int(piece_tiles), int(pdl), items.ctypes.data, int(max_items),
                          decs.ctypes.data, counts.ctypes.data, err, 512)
    if rc != MX_OK:
        raise MxError(rc, err.value.decode(errors="replace"))
    return {"items": items[:counts[0]].copy(), "decodes": decs[:len(lens)].copy(),
            "n_items": int(counts[0]), "n_prefill_items": int(counts[1]),
            "split_keys": int(counts[2]), "piece_tiles": int(counts[3]), "decode_first_ctas": int(counts[4])}


def _ptr(t):
    """Device pointer of a torch tensor (or an int address, or None)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream_handle(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ------------------------------------------------------------- layer ops
# The rest of a decoder layer (context-free C-ABI entry points): torch
# tensors in, argument marshalling only.
def _op(rc, name):
    if rc != 0:
        raise MxError(rc, f"{name} failed ({rc})")


def rms_norm(x, w, y, eps, stream=None):
    """y = x / sqrt(mean(x^2) + eps) * w over the last dim (bf16 as int16)."""
    rows, dim = x.shape[0], x.shape[-1]
    assert x.is_contiguous() and y.is_contiguous() and w.numel() == dim and y.shape == x.shape
    _op(load().mx_rms_norm(x.data_ptr(), w.data_ptr(), y.data_ptr(), rows, dim, float(eps),
                           _stream_handle(stream)), "mx_rms_norm")


def qk_norm_rope(qkv, q_norm, k_norm, positions, q, k, v, num_q_heads, num_kv_heads, theta, eps, stream=None):
    """q/k/v of the attention from the fused projection (see the header)."""
    n = qkv.shape[0]
    assert qkv.is_contiguous() and qkv.numel() == n * (num_q_heads + 2 * num_kv_heads) * 128
    assert q.is_contiguous() and k.is_contiguous() and v.is_contiguous() and positions.numel() >= n
    _op(load().mx_qk_norm_rope(qkv.data_ptr(), q_norm.data_ptr(), k_norm.data_ptr(), positions.data_ptr(),
                               q.data_ptr(), k.data_ptr(), v.data_ptr(), n, num_q_heads, num_kv_heads,
                               float(theta), float(eps), _stream_handle(stream)), "mx_qk_norm_rope")


def silu_mul(gate_up, y, stream=None):
    rows, d = y.shape[0], y.shape[-1]
    assert gate_up.is_contiguous() and y.is_contiguous() and gate_up.shape[-1] == 2 * d
    _op(load().mx_silu_mul(gate_up.data_ptr(), y.data_ptr(), rows, d, _stream_handle(stream)), "mx_silu_mul")


def gemm(a, b, c, accumulate=False, stream=None):
    """c [m][n] (+)= a [m][k] b [k][n], bf16 (as int16), fp32 accumulation."""
    m, k = a.shape[0], a.numel() // a.shape[0]
    n = b.shape[-1]
    assert a.is_contiguous() and b.is_contiguous() and c.is_contiguous()
    assert b.numel() == k * n and c.numel() == m * n
    _op(load().mx_gemm(a.data_ptr(), b.data_ptr(), c.data_ptr(), m, n, k, 1 if accumulate else 0,
                       _stream_handle(stream)), "mx_gemm")


class Context:
    """A mixattn context (fixed geometry and workspace) on one GPU."""

    def __init__(self, *, num_q_heads, num_kv_heads=8, head_dim=128, page_size=16,
                 num_pages, num_seqs, max_pages_per_seq, max_tokens, max_decodes,
                 device=0):
        self._lib = load()
        self.geom = mx_geom(num_q_heads, num_kv_heads, head_dim, page_size, num_pages,
                            num_seqs, max_pages_per_seq, max_tokens, max_decodes)
        self.device = device
        h = ctypes.c_void_p()
        rc = self._lib.mx_create(ctypes.byref(h), ctypes.byref(self.geom), device)
        if rc != MX_OK:
            buf = ctypes.create_string_buffer(512)
            self._lib.mx_error_detail(None, buf, 512)
            raise MxError(rc, "mx_create: " + buf.value.decode(errors="replace"))
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            self._lib.mx_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, rc):
        if rc != MX_OK:
            buf = ctypes.create_string_buffer(512)
            self._lib.mx_error_detail(self._h, buf, 512)
            raise MxError(rc, buf.value.decode(errors="replace"))

    # ------------------------------------------------------------------ calls
    def set_option(self, option, value):
        self._check(self._lib.mx_set_option(self._h, option, int(value)))

    def last_plan(self):
        a, b, c = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
        self._check(self._lib.mx_last_plan(self._h, ctypes.byref(a), ctypes.byref(b),
                                           ctypes.byref(c)))
        return {"n_items": a.value, "split_keys": b.value, "n_prefill_items": c.value}

    def kv_append(self, slots, k, v, k_pool, v_pool, stream=None):
        n = int(slots.shape[0])
        self._check(self._lib.mx_kv_append(self._h, _ptr(slots), n, _ptr(k), _ptr(v),
                                           _ptr(k_pool), _ptr(v_pool), _stream_handle(stream)))

    def make_desc(self, *, decode_seq_ids, decode_ctx_lens, prefill_seq_id=-1,
                  chunk_start=0, p_t=0, page_table, slots, prefills=None):
        """Descriptor with HOST decode arrays and DEVICE page_table/slots;
        several prefill chunks as ``prefills`` = [(seq, chunk_start, p_t),
        ...].  The returned object keeps the host arrays alive."""
        ids = np.ascontiguousarray(np.asarray(decode_seq_ids, dtype=np.int32))
        lens = np.ascontiguousarray(np.asarray(decode_ctx_lens, dtype=np.int32))
        pf_arr, n_pf = _prefill_array(prefills)
        d = mx_iter_desc(ids.ctypes.data if len(ids) else None,
                         lens.ctypes.data if len(lens) else None, len(lens),
                         int(prefill_seq_id), int(chunk_start), int(p_t),
                         _ptr(page_table), _ptr(slots), n_pf,
                         ctypes.cast(pf_arr, ctypes.c_void_p) if pf_arr is not None else None)
        d._keep = (ids, lens, pf_arr)
        return d

    @staticmethod
    def make_bufs(q, k, v, k_pool, v_pool, out):
        return mx_layer_bufs(_ptr(q), _ptr(k), _ptr(v), _ptr(k_pool), _ptr(v_pool), _ptr(out))

    def mixed_attention(self, desc, bufs, stream=None):
        self._check(self._lib.mx_mixed_attention(self._h, ctypes.byref(desc),
                                                 ctypes.byref(bufs), _stream_handle(stream)))

    @staticmethod
    def layer_array(layers):
        """Pack a list of mx_layer_bufs into a C array (reusable across calls)."""
        return (mx_layer_bufs * max(len(layers), 1))(*layers), len(layers)

    def iteration(self, desc, layers, stream=None, wait=True):
        """Run all layers.  wait=True: returns the device-completion time in
        microseconds (CUDA events, synchronised).  wait=False: enqueue only."""
        arr, n = layers if isinstance(layers, tuple) else self.layer_array(layers)
        us = ctypes.c_float()
        self._check(self._lib.mx_iteration(self._h, ctypes.byref(desc), n, arr,
                                           ctypes.byref(us) if wait else None,
                                           _stream_handle(stream)))
        return float(us.value) if wait else None

    def iteration_graph(self, desc, layers, stream=None, wait=True):
        """As iteration(), replayed from the context's captured graph (each
        layer's q/k/v/out must hold max_tokens rows)."""
        arr, n = layers if isinstance(layers, tuple) else self.layer_array(layers)
        us = ctypes.c_float()
        self._check(self._lib.mx_iteration_graph(self._h, ctypes.byref(desc), n, arr,
                                                 ctypes.byref(us) if wait else None,
                                                 _stream_handle(stream)))
        return float(us.value) if wait else None

    def sync_status(self, stream=None):
        self._check(self._lib.mx_sync_status(self._h, _stream_handle(stream)))
