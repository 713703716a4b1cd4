"""Host-side checks of the seeded input generator and workload layouts."""
import numpy as np

import synth
from synth import workload as wl


def test_splitmix64_published_outputs():
    # SplitMix64 seeded with 0: first two outputs of the reference generator.
    assert int(synth.splitmix64(np.uint64(0))) == 0xE220A8397B1DCDAF
    g = np.uint64(0x9E3779B97F4A7C15)
    assert int(synth.splitmix64(g)) == 0x6E789E6AA1B965F4


def test_bf16_round_to_nearest_even():
    f = np.array([1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, 1.0 + 2**-9, -0.0],
                 np.float32)
    # 1+2^-8 is a tie -> even (1.0); 1+3*2^-8 is a tie -> even (1+2^-6)
    np.testing.assert_array_equal(synth.f32_to_bf16_bits(f),
                                  [0x3F80, 0x3F80, 0x3F82, 0x3F80, 0x8000])


def test_table_is_normal_and_fill_matches_values():
    t = synth.normal_table()
    x = synth.bf16_bits_to_f32(t).astype(np.float64)
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    base = synth.stream_base(0, synth.stream_id(3, synth.STREAM_K))
    a = synth.fill(base, (5, 7))
    b = synth.values(base, np.arange(35, dtype=np.uint64)).reshape(5, 7)
    np.testing.assert_array_equal(a, b)
    # offsets address the same stream: elements 10.. equal a sub-range
    np.testing.assert_array_equal(
        synth.values(base, np.arange(10, 35, dtype=np.uint64)), a.ravel()[10:])
    assert synth.stream_base(0, 1) != synth.stream_base(0, 2)


def test_layout_pages_are_a_permutation_and_slots_consistent():
    lay = wl.make_layout(wl.Geometry(16), [33, 1, 16, 100], seed=4, spare_pages=2)
    used = lay.page_table[lay.page_table >= 0]
    assert len(np.unique(used)) == len(used)
    assert used.max() < lay.num_pages
    s = lay.slot(0, np.arange(33))
    assert len(np.unique(s)) == 33
    np.testing.assert_array_equal(s // 16, lay.page_table[0, np.arange(33) // 16])


def test_sweep_iterations_cover_every_chunk_in_order():
    its = wl.QWEN06B.iterations()
    assert its[0].p_t == 0 and its[0].n_decodes == 32
    for p in (256, 4096):
        chunks = [(i.chunk_start, i.p_t) for i in its if i.chunk_size == p]
        assert chunks == [(cs, p) for cs in range(0, 8192, p)]
    # decode contexts grow by one per iteration
    assert np.all(its[5].decode_ctx_lens == its[0].decode_ctx_lens + 5)
    ctx = its[0].decode_ctx_lens
    assert ctx.min() >= 512 and ctx.max() <= 4096
    small = wl.SMALL.iterations()
    assert len(small) == 1 and small[0].chunk_start == 128 and small[0].p_t == 128
    lay = wl.SMALL.layout()
    sl = small[0].slots(lay)
    assert len(sl) == 4 + 128 and len(np.unique(sl)) == len(sl)


def test_c_fast_path_matches_numpy_definition():
    base = synth.stream_base(7, synth.stream_id(2, synth.STREAM_V, 3))
    idx = np.arange(1000, 5000, dtype=np.uint64)
    np.testing.assert_array_equal(synth.values_range(base, 1000, 4000), synth.values(base, idx))
    pages = np.array([5, 0, 17], np.int64)
    pe = 64
    want = synth.values(base, (pages.astype(np.uint64)[:, None] * np.uint64(pe)
                               + np.arange(pe, dtype=np.uint64)[None]).ravel())
    np.testing.assert_array_equal(synth.values_pages(base, pages, pe), want)
