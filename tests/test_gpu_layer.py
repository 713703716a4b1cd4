"""GPU parity of the decoder-layer steps around the mixed attention (RMSNorm,
QK norm with RoPE, SwiGLU gate, bf16 GEMM) and of one whole Qwen3 layer,
against the float64 oracle of oracle/layer.py (pinned in
tests/test_oracle_layer.py).

Tolerances: every step stores bf16, so a single step may differ from the
oracle (float64, the same bf16 rounding points) by the rounding of its own
output, one bf16 ulp (at most 2^-7 relative) plus the float32 arithmetic's
error; the GEMM that adds into its output (a residual) rounds the product
and then the sum, a bound on the terms' magnitudes (they may cancel);
the whole layer compounds such differences through its GEMMs (relative RMS
below 1e-2, max abs below 4 % of the largest output).
"""
import numpy as np
import pytest

from oracle import layer as OL
from tests.harness import Case

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _bf16(rng, *shape, scale=1.0):
    return OL.f64_to_bf16(rng.standard_normal(shape) * scale)


def _dev(u16):
    return torch.from_numpy(np.ascontiguousarray(u16).view(np.int16)).cuda()


def _host(t):
    return OL.bf16_to_f64(t.cpu().numpy().view(np.uint16))


def _within_ulp(got, ref, ulps=1.0, floor=1e-6):
    err = np.abs(got - ref)
    bound = ulps * np.maximum(np.abs(ref), floor) * 2.0 ** -7 + floor
    assert np.all(err <= bound), f"max err {err.max():.3e}, worst ratio {(err / bound).max():.2f}"


@pytest.mark.parametrize("rows,dim", [(37, 1024), (5, 5120), (1, 8)])
def test_rms_norm(rows, dim):
    from paper_2609_38386_gb300 import _binding as B
    rng = np.random.default_rng(rows + dim)
    x, w = _bf16(rng, rows, dim, scale=3.0), OL.f64_to_bf16(1 + 0.1 * rng.standard_normal(dim))
    y = torch.empty((rows, dim), dtype=torch.int16, device="cuda")
    B.rms_norm(_dev(x), _dev(w), y, 1e-6)
    ref = OL.round_bf16(OL.rms_norm(OL.bf16_to_f64(x), OL.bf16_to_f64(w), 1e-6))
    _within_ulp(_host(y), ref)


@pytest.mark.parametrize("hq,hkv", [(16, 8), (64, 8), (8, 8)])
def test_qk_norm_rope(hq, hkv):
    from paper_2609_38386_gb300 import _binding as B
    rng = np.random.default_rng(hq)
    n = 50
    qkv = _bf16(rng, n, (hq + 2 * hkv) * 128, scale=2.0)
    qn, kn = (OL.f64_to_bf16(1 + 0.1 * rng.standard_normal(128)) for _ in range(2))
    pos = np.concatenate([[0, 1, 2, 63, 64, 4095, 16384, 32767], rng.integers(0, 32768, n - 8)]).astype(np.int32)
    q = torch.empty((n, hq, 128), dtype=torch.int16, device="cuda")
    k = torch.empty((n, hkv, 128), dtype=torch.int16, device="cuda")
    v = torch.empty_like(k)
    B.qk_norm_rope(_dev(qkv), _dev(qn), _dev(kn), torch.from_numpy(pos).cuda(), q, k, v, hq, hkv, 1e6, 1e-6)
    rq, rk, rv = OL.qk_norm_rope(OL.bf16_to_f64(qkv), OL.bf16_to_f64(qn), OL.bf16_to_f64(kn), pos, hq, hkv,
                                 1e6, 1e-6)
    # the rotation mixes two values of a pair: one ulp of the pair's magnitude
    for got, ref in ((_host(q), rq), (_host(k), rk)):
        pair = np.sqrt(ref[..., :64] ** 2 + ref[..., 64:] ** 2)
        err = np.abs(got - OL.round_bf16(ref))
        assert np.all(err <= np.concatenate([pair, pair], axis=-1) * 2.0 ** -7 + 1e-6), err.max()
    np.testing.assert_array_equal(v.cpu().numpy().view(np.uint16),
                                  qkv.reshape(n, hq + 2 * hkv, 128)[:, hq + hkv:])


def test_silu_mul():
    from paper_2609_38386_gb300 import _binding as B
    rng = np.random.default_rng(7)
    rows, d = 33, 3072
    gu = _bf16(rng, rows, 2 * d, scale=2.0)
    y = torch.empty((rows, d), dtype=torch.int16, device="cuda")
    B.silu_mul(_dev(gu), y)
    ref = OL.round_bf16(OL.silu_mul(OL.bf16_to_f64(gu), d))
    _within_ulp(_host(y), ref, floor=1e-4)


@pytest.mark.parametrize("m,n,k,acc", [(70, 384, 1024, False), (3, 1024, 2048, True), (257, 96, 64, True)])
def test_gemm(m, n, k, acc):
    from paper_2609_38386_gb300 import _binding as B
    rng = np.random.default_rng(m + n + k)
    a, b = _bf16(rng, m, k), _bf16(rng, k, n, scale=k ** -0.5)
    c0 = _bf16(rng, m, n)
    c = _dev(c0)
    B.gemm(_dev(a), _dev(b), c, accumulate=acc)
    ab = OL.bf16_to_f64(a) @ OL.bf16_to_f64(b)
    ref = ab + (OL.bf16_to_f64(c0) if acc else 0.0)
    # float32 accumulation over k terms, then one bf16 rounding of the
    # product; with accumulate the sum may be rounded again, so the bound
    # follows the terms' magnitudes (they may cancel in the sum)
    got = _host(c)
    scale = np.sqrt(k) * np.abs(OL.bf16_to_f64(a)).max() * np.abs(OL.bf16_to_f64(b)).max()
    terms = np.abs(ab) + (np.abs(OL.bf16_to_f64(c0)) if acc else 0.0)
    assert np.all(np.abs(got - ref) <= 2.0 ** -7 * (terms + np.abs(ref)) + scale * 1e-5), np.abs(got - ref).max()


def test_ops_reject_bad_arguments():
    from paper_2609_38386_gb300 import _binding as B
    lib = B.load()
    assert lib.mx_rms_norm(None, None, None, 4, 12, 1e-6, None) == -1      # dim not a multiple of 8
    assert lib.mx_silu_mul(None, None, 4, 12, None) == -1
    assert lib.mx_gemm(None, None, None, 4, 0, 8, 0, None) == -1
    assert lib.mx_qk_norm_rope(None, None, None, None, None, None, None, 4, 16, 8, 0.5, 1e-6, None) == -1


@pytest.mark.parametrize("hq,d,f", [(16, 1024, 3072), (32, 1536, 4096)])
def test_decoder_layer_vs_oracle(hq, d, f):
    import oracle
    from paper_2609_38386_gb300.layer import Qwen3Layer, positions_of
    case = Case(hq, [300, 17, 1200, 5], chunk_start=640, p_t=200, seed=hq, device_pools=False)
    n, hkv = case.n_tokens, case.geom.hkv
    layer = Qwen3Layer(d, f, hq, hkv, seed=5, device="cuda")
    ctx = case.make_context()
    dinp = case.device_inputs()
    attn = {"q": torch.empty((n, hq, 128), dtype=torch.int16, device="cuda"),
            "k": torch.empty((n, hkv, 128), dtype=torch.int16, device="cuda"),
            "v": torch.empty((n, hkv, 128), dtype=torch.int16, device="cuda"),
            "k_pool": dinp["k_pool"], "v_pool": dinp["v_pool"],
            "out": torch.empty((n, hq, 128), dtype=torch.int16, device="cuda")}
    rng = np.random.default_rng(9)
    x0 = _bf16(rng, n, d)
    x = _dev(x0)
    pos = positions_of(case.it)
    layer.forward(ctx, case.desc(ctx, dinp), x, torch.from_numpy(pos).cuda(), attn)
    torch.cuda.synchronize()
    ctx.sync_status()
    got = _host(x)
    ctx.close()

    w = {k_: OL.bf16_to_f64(t.cpu().numpy().view(np.uint16)) for k_, t in layer.weights().items()}
    k0, v0 = case.pools0()
    it = case.it

    def attention(q, k, v):
        out, _ = oracle.mixed_attention(
            q=OL.f64_to_bf16(q), k=OL.f64_to_bf16(k), v=OL.f64_to_bf16(v), k_pool=k0.copy(), v_pool=v0.copy(),
            page_table=case.layout.page_table, slots=case.slots, decode_seq_ids=it.decode_seq_ids,
            decode_ctx_lens=it.decode_ctx_lens, prefill_seq=it.prefill_seq, chunk_start=it.chunk_start, p_t=it.p_t)
        return out

    ref = OL.decoder_layer(OL.bf16_to_f64(x0), w, attention, pos, hq, hkv, 1e6, 1e-6)
    err = got - ref
    rel_rms = np.sqrt(np.mean(err ** 2) / np.mean(ref ** 2))
    print(f"layer: rel rms {rel_rms:.3e}, max abs {np.abs(err).max():.3e}, max |ref| {np.abs(ref).max():.3e}")
    assert np.isfinite(got).all()
    assert rel_rms < 1e-2
    assert np.abs(err).max() < 0.04 * np.abs(ref).max()
