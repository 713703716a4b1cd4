"""The C-ABI library loads and exports every entry point include/*.h
declares; argument checks that need no GPU return their error codes."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_38386_gb300 import build as b
    if not os.path.exists(b.LIB):
        b.build_library()
    from paper_2609_38386_gb300 import _binding
    return _binding.load()


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        names.update(re.findall(r"^int\s+(mx_\w+)\s*\(", open(h).read(), re.M))
    return names


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("mx_create", "mx_destroy", "mx_kv_append", "mx_mixed_attention",
                 "mx_iteration"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2609_38386_gb300 import _binding
    for name in _declared():
        assert hasattr(lib, name), name
    assert set(_binding.EXPORTS) >= _declared()


def test_null_and_geometry_checks_without_gpu(lib):
    from paper_2609_38386_gb300._binding import mx_geom
    assert lib.mx_destroy(None) == 0
    assert lib.mx_mixed_attention(None, None, None, None) == -1
    assert lib.mx_iteration(None, None, 0, None, None, None) == -1
    assert lib.mx_iteration_graph(None, None, 0, None, None, None) == -1
    assert lib.mx_error_detail(None, None, 0) == -1
    assert lib.mx_set_option(None, 1, 0) == -1
    h = ctypes.c_void_p()
    bad = mx_geom(16, 8, 64, 16, 10, 1, 4, 8, 1)          # head_dim 64 unsupported
    assert lib.mx_create(ctypes.byref(h), ctypes.byref(bad), 0) == -1
    bad = mx_geom(24, 8, 128, 16, 10, 1, 4, 8, 1)         # n_rep 3 unsupported
    assert lib.mx_create(ctypes.byref(h), ctypes.byref(bad), 0) == -1
    # with no context, mx_error_detail reports why this thread's mx_create failed
    buf = ctypes.create_string_buffer(256)
    assert lib.mx_error_detail(None, buf, 256) > 0
    assert b"geometry" in buf.value
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:
        has_gpu = False
    if not has_gpu:
        good = mx_geom(16, 8, 128, 16, 10, 1, 4, 8, 1)
        assert lib.mx_create(ctypes.byref(h), ctypes.byref(good), 0) == -6   # MX_EDEVICE
        assert lib.mx_error_detail(None, buf, 256) > 0 and b"device" in buf.value


def test_noalloc_rejects_a_repeated_sequence_before_any_cuda_call(lib):
    """The allocation-free entry point checks its descriptor on the host
    first: a sequence listed twice (two decodes, or a decode and the chunk)
    returns MX_EINVAL before any CUDA call, so this runs without a GPU.  The
    tensor pointers are never dereferenced."""
    from paper_2609_38386_gb300._binding import mx_geom, mx_iter_desc, mx_layer_bufs
    import numpy as np
    geom = mx_geom(16, 8, 128, 16, 100, 4, 8, 0, 0)
    fake = 1 << 20                                       # aligned, never used
    bufs = mx_layer_bufs(fake, fake, fake, fake, fake, fake)
    err = ctypes.create_string_buffer(256)
    for ids, pseq, p in (([1, 1], -1, 0), ([0, 2], 2, 16)):
        seqs = np.asarray(ids, np.int32)
        lens = np.asarray([5, 6], np.int32)
        desc = mx_iter_desc(seqs.ctypes.data, lens.ctypes.data, 2, pseq, 0, p, fake, fake, 0, None)
        rc = lib.mx_mixed_attention_noalloc(ctypes.byref(geom), ctypes.byref(desc), ctypes.byref(bufs),
                                            None, err, 256)
        assert rc == -1 and b"twice" in err.value, (rc, err.value)
