"""The rest of a Qwen3 decoder layer around the mixed attention, float64 —
TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may use it).

The whole-model setting of the paper's measurements (§4.1: Qwen3 models in
vLLM) puts these steps around attention in every layer; their cost is part
of the iteration time L_t of Eq. 1.  A pre-norm decoder layer:

    h  = RMSNorm(x) * g_in
    q, k, v = split(h W_qkv)                          (q: Hq heads, k, v: Hkv)
    q, k = RoPE(RMSNorm_head(q) * g_q), RoPE(RMSNorm_head(k) * g_k)
    x  = x + Attention(q, k, v) W_o
    h  = RMSNorm(x) * g_post
    x  = x + (silu(h W_gate) * (h W_up)) W_down

RMSNorm(x) = x / sqrt(mean(x^2) + eps).  RoPE pairs element i of a head
with element i + 64 (rotate-half) and turns the pair by the angle
pos * theta^(-i/64).  All arithmetic is float64; ``rounded=True`` rounds to
bf16 exactly where the GPU path stores a bf16 tensor (after each norm, GEMM,
the q/k/v and the attention output, and x after each residual add), so that
the two differ only by fp32-versus-fp64 arithmetic.
"""
from __future__ import annotations

import numpy as np

HEAD_DIM = 128


def bf16_to_f64(u):
    """uint16 bf16 bits -> float64."""
    u = np.asarray(u, dtype=np.uint16)
    return (u.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def f64_to_bf16(x):
    """float64 -> uint16 bf16 bits, round to nearest even (via float32)."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    nan = np.isnan(f)
    if nan.any():
        r = np.where(nan, np.uint16(0x7FC0), r)
    return r


def round_bf16(x):
    return bf16_to_f64(f64_to_bf16(x))


def rms_norm(x, w, eps):
    """x [rows][dim], w [dim] (float64)."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(w, dtype=np.float64)


def rope_angles(positions, theta):
    """angle[t][f] = pos_t * theta^(-f/64), f = 0..63."""
    f = np.arange(HEAD_DIM // 2, dtype=np.float64)
    return np.asarray(positions, dtype=np.float64)[:, None] * theta ** (-f / (HEAD_DIM // 2))


def rope(x, positions, theta):
    """x [tokens][heads][128]: element i and i + 64 turned by angle[t][i]."""
    a = rope_angles(positions, theta)[:, None, :]
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., :HEAD_DIM // 2], x[..., HEAD_DIM // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def qk_norm_rope(qkv, q_norm, k_norm, positions, hq, hkv, theta, eps):
    """qkv [tokens][(hq + 2 hkv) * 128] (float64) -> q, k, v (float64)."""
    n = qkv.shape[0]
    heads = np.asarray(qkv, dtype=np.float64).reshape(n, hq + 2 * hkv, HEAD_DIM)
    q, k, v = heads[:, :hq], heads[:, hq:hq + hkv], heads[:, hq + hkv:]
    q = rope(rms_norm(q, q_norm, eps), positions, theta)
    k = rope(rms_norm(k, k_norm, eps), positions, theta)
    return q, k, v.copy()


def silu_mul(gate_up, d_ffn):
    g, u = gate_up[:, :d_ffn], gate_up[:, d_ffn:]
    return g / (1.0 + np.exp(-g)) * u


def decoder_layer(x, w, attention, positions, hq, hkv, theta, eps, rounded=True):
    """One layer.  x [tokens][d] float64; w: dict of float64 arrays
    (norm_in, w_qkv [d][(hq+2hkv)128], q_norm, k_norm, w_o [hq 128][d],
    norm_post, w_gate_up [d][2 f], w_down [f][d]); attention(q, k, v) ->
    out [tokens][hq][128] float64 for bf16-valued q/k/v (the mixed
    attention of one layer, KV append included).  Returns the new x."""
    rb = round_bf16 if rounded else (lambda a: a)
    n = x.shape[0]
    h = rb(rms_norm(x, w["norm_in"], eps))
    qkv = rb(h @ w["w_qkv"])
    q, k, v = qk_norm_rope(qkv, w["q_norm"], w["k_norm"], positions, hq, hkv, theta, eps)
    o = rb(attention(rb(q), rb(k), rb(v)))
    x = rb(x + o.reshape(n, hq * HEAD_DIM) @ w["w_o"])
    h = rb(rms_norm(x, w["norm_post"], eps))
    d_ffn = w["w_down"].shape[0]
    a = rb(silu_mul(rb(h @ w["w_gate_up"]), d_ffn))
    return rb(x + a @ w["w_down"])
