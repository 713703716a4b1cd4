"""The allocation-free entry point, mx_mixed_attention_noalloc.

It serves callers that cannot call cudaMalloc (a framework whose allocator
owns the GPU, a plug-in with a fixed memory budget, a path that must not risk
an allocation's synchronisation or OOM): it runs one mixed layer call with its
scratch in a fixed device array compiled into the library.  Checked here
through the C ABI, on two calls in a row (the second call reuses the array
the first one left behind):

- against the float64 oracle, within the parity tolerance, with the KV pages
  bit-exact;
- against the context-based mx_mixed_attention on the same inputs: both
  plan the same work list for these cases, so the outputs are bit-identical;
- with decodes of 1 and 6 keys (the exact short path) and long decodes cut
  into several splits merged through the array's partial slots;
- rejections: more decodes than the array holds, and several prefill chunks
  (which need a context), both with nothing enqueued.

This file sorts last so that a run stopping at the first failure has already
run every other test.
"""
import ctypes

import numpy as np
import pytest

from tests import harness
from tests.harness import MAX_ABS, MEAN_ABS, Case

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _call_noalloc(lib, case, d, prefills=None):
    from paper_2609_38386_gb300._binding import _prefill_array, mx_geom, mx_iter_desc, mx_layer_bufs
    lay = case.layout
    geom = mx_geom(case.geom.hq, case.geom.hkv, 128, 16, lay.num_pages, lay.num_seqs,
                   lay.max_pages, 0, 0)
    it = case.it
    ids = np.ascontiguousarray(it.decode_seq_ids, dtype=np.int32)
    lens = np.ascontiguousarray(it.decode_ctx_lens, dtype=np.int32)
    pf_arr, n_pf = _prefill_array(prefills)
    desc = mx_iter_desc(ids.ctypes.data if len(ids) else None,
                        lens.ctypes.data if len(lens) else None, len(lens), it.prefill_seq,
                        it.chunk_start, it.p_t, d["page_table"].data_ptr(), d["slots"].data_ptr(),
                        n_pf, ctypes.cast(pf_arr, ctypes.c_void_p) if pf_arr is not None else None)
    bufs = mx_layer_bufs(d["q"].data_ptr(), d["k"].data_ptr(), d["v"].data_ptr(),
                         d["k_pool"].data_ptr(), d["v_pool"].data_ptr(), d["out"].data_ptr())
    err = ctypes.create_string_buffer(256)
    rc = lib.mx_mixed_attention_noalloc(ctypes.byref(geom), ctypes.byref(desc), ctypes.byref(bufs),
                                        torch.cuda.current_stream().cuda_stream, err, 256)
    return rc, err.value.decode()


@pytest.mark.parametrize("ctxs,cs,p,hq", [
    ([5000, 17, 1500, 3333, 64, 9000], 300, 260, 32),     # split partials + a chunk
    ([0, 5, 700, 12000, 15, 16], 0, 37, 16),              # 1- and 6-key decodes, chunk at 0
    ([30000, 25000, 4097], 0, 0, 64),                     # long decodes, decode-only
])
def test_noalloc_matches_oracle_and_context_entry_point_twice(ctxs, cs, p, hq):
    from paper_2609_38386_gb300 import load
    lib = load()
    case = Case(hq, ctxs, chunk_start=cs, p_t=p, seed=21 + hq)
    ref = case.run_gpu()                       # context-based entry point
    _, _, kp_want, vp_want = case.oracle_full()
    for call in range(2):
        d = case.device_inputs()
        rc, msg = _call_noalloc(lib, case, d)
        assert rc == 0, (call, rc, msg)
        out = d["out"].cpu().numpy().view(np.uint16)
        res = {"out": out, "k_pool": d["k_pool"].cpu().numpy().view(np.uint16),
               "v_pool": d["v_pool"].cpu().numpy().view(np.uint16)}
        err = case.check(res)                  # the float64 oracle
        assert err["finite"] and err["pools_exact"], (call, err)
        assert err["max_abs"] <= MAX_ABS and err["mean_abs"] <= MEAN_ABS, (call, err)
        diff = np.abs(harness._bf16_to_f64(out) - harness._bf16_to_f64(ref["out"]))
        assert diff.max() <= MAX_ABS and diff.mean() <= MEAN_ABS, (call, diff.max(), diff.mean())
        # the same work list as the context path: the same bits
        np.testing.assert_array_equal(out, ref["out"])
        np.testing.assert_array_equal(res["k_pool"], kp_want)
        np.testing.assert_array_equal(res["v_pool"], vp_want)


def test_noalloc_rejects_sizes_beyond_its_limits():
    from paper_2609_38386_gb300 import load
    lib = load()
    case = Case(16, [10] * 257, seed=3)        # 257 decodes > 256
    d = case.device_inputs()
    rc, msg = _call_noalloc(lib, case, d)
    assert rc == -7 and "256" in msg, (rc, msg)
    assert np.all(d["out"].cpu().numpy() == 0x7FC1)   # nothing was enqueued


def test_noalloc_rejects_several_chunks():
    from paper_2609_38386_gb300 import load
    lib = load()
    case = Case(16, [40, 90], seed=4)
    d = case.device_inputs()
    case.it.prefill_seq = -1
    rc, msg = _call_noalloc(lib, case, d, prefills=[(0, 10, 20), (1, 30, 5)])
    assert rc == -1 and "context" in msg, (rc, msg)
    assert np.all(d["out"].cpu().numpy() == 0x7FC1)   # nothing was enqueued
