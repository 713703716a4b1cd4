"""A Qwen3 decoder layer around the mixed attention, with random weights.

The paper measures whole models (§4.1: Qwen3 in vLLM), so the iteration time
L_t of Eq. 1 holds, besides attention, the projections and the MLP of every
token of the batch: the prefill share grows with p_t through them too.  One
layer, pre-norm:

    h = RMSNorm(x) g_in;  q, k, v = h W_qkv
    q, k = RoPE(RMSNorm_head(q) g_q), RoPE(RMSNorm_head(k) g_k)   (positions)
    x += MixedAttention(q, k, v) W_o                              (KV append included)
    h = RMSNorm(x) g_post;  x += (silu(h W_gate) * h W_up) W_down

Every step runs in this package's library: RMSNorm, the QK norm with RoPE
and the SwiGLU gate in its own kernels, the projections as cuBLAS GEMMs
(`mx_gemm`, the residual adds folded into the GEMM's accumulate), attention
in `mx_mixed_attention`.  This module holds the weights and calls the steps
in order.
"""
from __future__ import annotations

from . import _binding as B

HEAD_DIM = 128


class Qwen3Layer:
    """Weights of one decoder layer (bf16 stored as int16 tensors), seeded:
    projections N(0, 1 / fan_in), norm gains 1 + N(0, 0.1^2)."""

    def __init__(self, d_model, d_ffn, num_q_heads, num_kv_heads, seed, device, theta=1.0e6, eps=1.0e-6):
        import torch
        self.d, self.f, self.hq, self.hkv = d_model, d_ffn, num_q_heads, num_kv_heads
        self.theta, self.eps = theta, eps
        gen = torch.Generator(device="cpu").manual_seed(int(seed))

        def rnd(*shape, std):
            t = torch.randn(*shape, generator=gen, dtype=torch.float32) * std
            return t.to(torch.bfloat16).view(torch.int16).to(device).contiguous()

        def gain(n):
            t = 1.0 + 0.1 * torch.randn(n, generator=gen, dtype=torch.float32)
            return t.to(torch.bfloat16).view(torch.int16).to(device).contiguous()

        qkv_w = (num_q_heads + 2 * num_kv_heads) * HEAD_DIM
        self.norm_in = gain(d_model)
        self.w_qkv = rnd(d_model, qkv_w, std=d_model ** -0.5)
        self.q_norm = gain(HEAD_DIM)
        self.k_norm = gain(HEAD_DIM)
        self.w_o = rnd(num_q_heads * HEAD_DIM, d_model, std=(num_q_heads * HEAD_DIM) ** -0.5)
        self.norm_post = gain(d_model)
        self.w_gate_up = rnd(d_model, 2 * d_ffn, std=d_model ** -0.5)
        self.w_down = rnd(d_ffn, d_model, std=d_ffn ** -0.5)

    def weights(self):
        return {n: getattr(self, n) for n in ("norm_in", "w_qkv", "q_norm", "k_norm", "w_o", "norm_post",
                                              "w_gate_up", "w_down")}

    def forward(self, ctx, desc, x, positions, attn, stream=None):
        """x [n][d] (the layer input, updated in place); positions int32 [n]
        (decode i: its cached tokens; chunk row j: chunk_start + j); attn:
        dict of the layer's attention tensors q, k, v, k_pool, v_pool, out
        (at least n rows).  Asynchronous on `stream`."""
        import torch
        n = x.shape[0]
        if n == 0:
            return x
        dev = x.device
        h = torch.empty((n, self.d), dtype=torch.int16, device=dev)
        qkv = torch.empty((n, (self.hq + 2 * self.hkv) * HEAD_DIM), dtype=torch.int16, device=dev)
        q, k, v, out = attn["q"][:n], attn["k"][:n], attn["v"][:n], attn["out"][:n]
        B.rms_norm(x, self.norm_in, h, self.eps, stream)
        B.gemm(h, self.w_qkv, qkv, stream=stream)
        B.qk_norm_rope(qkv, self.q_norm, self.k_norm, positions, q, k, v, self.hq, self.hkv, self.theta,
                       self.eps, stream)
        bufs = ctx.make_bufs(attn["q"], attn["k"], attn["v"], attn["k_pool"], attn["v_pool"], attn["out"])
        ctx.mixed_attention(desc, bufs, stream)
        B.gemm(out, self.w_o, x, accumulate=True, stream=stream)
        B.rms_norm(x, self.norm_post, h, self.eps, stream)
        gu = torch.empty((n, 2 * self.f), dtype=torch.int16, device=dev)
        a = torch.empty((n, self.f), dtype=torch.int16, device=dev)
        B.gemm(h, self.w_gate_up, gu, stream=stream)
        B.silu_mul(gu, a, stream)
        B.gemm(a, self.w_down, x, accumulate=True, stream=stream)
        return x


def positions_of(desc_it):
    """Token positions of an iteration (decode i at ctx_i, chunk row j at
    chunk_start + j) as int32, for an object with decode_ctx_lens,
    chunk_start and p_t."""
    import numpy as np
    parts = [np.asarray(desc_it.decode_ctx_lens, dtype=np.int32)]
    if desc_it.p_t:
        parts.append(np.arange(desc_it.chunk_start, desc_it.chunk_start + desc_it.p_t, dtype=np.int32))
    return np.concatenate(parts).astype(np.int32)
