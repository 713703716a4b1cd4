"""Device fill with the counter-based generator of ``synth`` (test/bench input
set-up only).  Every value it writes can be recomputed on the host with
``synth.values`` — the oracle never reads an input back from the GPU."""
from __future__ import annotations

import ctypes
import os

import numpy as np

import synth

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB = os.path.join(_HERE, "libsynth.so")
_lib = None
_tables = {}


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is missing: run __graft_entry__.build() first")
        lib = ctypes.CDLL(LIB)
        lib.synth_fill.restype = ctypes.c_int
        lib.synth_fill.argtypes = [ctypes.c_void_p, ctypes.c_longlong, ctypes.c_ulonglong,
                                   ctypes.c_longlong, ctypes.c_void_p, ctypes.c_void_p]
        _lib = lib
    return _lib


def _table(device):
    import torch
    key = str(device)
    if key not in _tables:
        t = torch.from_numpy(synth.normal_table().view(np.int16).copy())
        _tables[key] = t.to(device)
    return _tables[key]


def fill_(tensor, base: int, start: int = 0, stream=None):
    """Fill a contiguous 16-bit CUDA tensor with elements start.. of a stream."""
    import torch
    assert tensor.is_cuda and tensor.is_contiguous() and tensor.element_size() == 2
    s = torch.cuda.current_stream(tensor.device) if stream is None else stream
    rc = _load().synth_fill(tensor.data_ptr(), tensor.numel(), ctypes.c_ulonglong(base),
                            start, _table(tensor.device).data_ptr(), s.cuda_stream)
    if rc != 0:
        raise RuntimeError(f"synth_fill failed: cuda error {rc}")
    return tensor


def fill_tokens_(tensor, seed, layer, kind, it, stream=None):
    """Device fill of a per-token input with the layout of
    ``synth.workload.token_parts`` (decode rows, then chunk rows)."""
    from synth import workload as wl
    w = tensor.shape[1] * tensor.shape[2]
    for row0, n, base, start in wl.token_parts(seed, layer, kind, it):
        fill_(tensor[row0:row0 + n], base, start * w, stream)
    return tensor
