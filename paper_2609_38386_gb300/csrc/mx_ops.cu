// The rest of a Qwen3 decoder layer around the mixed attention (the
// whole-model setting of the paper's measurements, §4.1, whose prefill share
// of L_t is Eq. 1's L_prefill): RMSNorm, the per-head QK RMSNorm with rotary
// position embedding that produces the attention's q/k/v, the SwiGLU gate,
// and a bf16 GEMM (cuBLAS, fp32 accumulation) for the projections.
// Context-free entry points: plain device pointers, row-major bf16 tensors.
#include "../../include/mixattn.h"
#include "mx_internal.h"

#include <cublas_v2.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

namespace mx {
namespace {

__device__ __forceinline__ float bf(uint16_t u) { return __uint_as_float((uint32_t)u << 16); }
__device__ __forceinline__ uint16_t to_bf(float x)
{
    __nv_bfloat16 b = __float2bfloat16_rn(x);
    return *reinterpret_cast<uint16_t *>(&b);
}

__device__ __forceinline__ float warp_sum(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// y = x / sqrt(mean(x^2) + eps) * w, one warp per row, 8 bf16 per 16-byte
// access (dim a multiple of 8); the sum of squares in fp32.
__global__ void rms_norm_kernel(const uint4 *__restrict__ x, const uint4 *__restrict__ w, uint4 *__restrict__ y,
                                int rows, int dim8, float eps)
{
    const int row = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= rows)
        return;
    const uint4 *xr = x + (size_t)row * dim8;
    float ss = 0.f;
    for (int c = lane; c < dim8; c += 32) {
        const uint4 v = __ldg(xr + c);
        const uint32_t u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = bf((uint16_t)(u[e] & 0xFFFFu)), b = bf((uint16_t)(u[e] >> 16));
            ss += a * a + b * b;
        }
    }
    ss = warp_sum(ss);
    const float inv = rsqrtf(ss / (float)(dim8 * 8) + eps);
    uint4 *yr = y + (size_t)row * dim8;
    for (int c = lane; c < dim8; c += 32) {
        const uint4 v = __ldg(xr + c), g = __ldg(w + c);
        const uint32_t u[4] = {v.x, v.y, v.z, v.w}, gw[4] = {g.x, g.y, g.z, g.w};
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float a = bf((uint16_t)(u[e] & 0xFFFFu)) * inv * bf((uint16_t)(gw[e] & 0xFFFFu));
            const float b = bf((uint16_t)(u[e] >> 16)) * inv * bf((uint16_t)(gw[e] >> 16));
            o[e] = (uint32_t)to_bf(a) | ((uint32_t)to_bf(b) << 16);
        }
        yr[c] = make_uint4(o[0], o[1], o[2], o[3]);
    }
}

// One warp per (token, head slot) of a fused QKV row [q heads | k heads | v
// heads] (head_dim 128: four elements per lane).  q and k heads: RMSNorm over
// the head (weight qn / kn), then the rotary embedding of position pos in
// the rotate-half pairing (element i with i + 64, frequency theta^(-i/64)),
// the angle reduced modulo 2 pi in double precision; v heads: copied.
__global__ void qk_norm_rope_kernel(const uint16_t *__restrict__ qkv, const uint16_t *__restrict__ qn,
                                    const uint16_t *__restrict__ kn, const int32_t *__restrict__ pos,
                                    uint16_t *__restrict__ q, uint16_t *__restrict__ k, uint16_t *__restrict__ v,
                                    int n_tok, int hq, int hkv, float theta, float eps)
{
    const int slots = hq + 2 * hkv;
    const long long gw = (long long)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (gw >= (long long)n_tok * slots)
        return;
    const int tok = (int)(gw / slots), h = (int)(gw % slots);
    const uint16_t *src = qkv + ((size_t)tok * slots + h) * kHeadDim + 4 * lane;
    const uint2 raw = *reinterpret_cast<const uint2 *>(src);
    float x[4] = {bf((uint16_t)(raw.x & 0xFFFFu)), bf((uint16_t)(raw.x >> 16)), bf((uint16_t)(raw.y & 0xFFFFu)),
                  bf((uint16_t)(raw.y >> 16))};
    uint16_t *dst;
    if (h >= hq + hkv) {   // v head: as it is
        dst = v + ((size_t)tok * hkv + (h - hq - hkv)) * kHeadDim + 4 * lane;
        *reinterpret_cast<uint2 *>(dst) = raw;
        return;
    }
    const bool is_q = h < hq;
    const uint16_t *nw = (is_q ? qn : kn) + 4 * lane;
    dst = is_q ? q + ((size_t)tok * hq + h) * kHeadDim + 4 * lane
               : k + ((size_t)tok * hkv + (h - hq)) * kHeadDim + 4 * lane;
    const float ss = warp_sum(x[0] * x[0] + x[1] * x[1] + x[2] * x[2] + x[3] * x[3]);
    const float inv = rsqrtf(ss / (float)kHeadDim + eps);
#pragma unroll
    for (int e = 0; e < 4; ++e)
        x[e] = x[e] * inv * bf(nw[e]);
    // partner elements (i <-> i + 64) are 16 lanes apart
    float px[4];
#pragma unroll
    for (int e = 0; e < 4; ++e)
        px[e] = __shfl_xor_sync(0xffffffffu, x[e], 16);
    const bool first = lane < 16;
    const double p = (double)pos[tok];
    const double l2t = log2((double)theta);
    float o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const int f = (4 * lane + e) & 63;                       // frequency index
        double ang = p * exp2(-(double)f / 64.0 * l2t);
        ang = fmod(ang, 6.283185307179586476925286766559);
        float s, c;
        sincosf((float)ang, &s, &c);
        o[e] = first ? x[e] * c - px[e] * s : x[e] * c + px[e] * s;
    }
    uint2 outv;
    outv.x = (uint32_t)to_bf(o[0]) | ((uint32_t)to_bf(o[1]) << 16);
    outv.y = (uint32_t)to_bf(o[2]) | ((uint32_t)to_bf(o[3]) << 16);
    *reinterpret_cast<uint2 *>(dst) = outv;
}

// y[r, j] = silu(g) * u with g = gu[r, j], u = gu[r, d + j]; 8 per thread.
__global__ void silu_mul_kernel(const uint4 *__restrict__ gu, uint4 *__restrict__ y, int rows, int d8)
{
    const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= (long long)rows * d8)
        return;
    const long long r = i / d8, c = i % d8;
    const uint4 g = __ldg(gu + r * 2 * d8 + c), u = __ldg(gu + r * 2 * d8 + d8 + c);
    const uint32_t gw[4] = {g.x, g.y, g.z, g.w}, uw[4] = {u.x, u.y, u.z, u.w};
    uint32_t o[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        const float g0 = bf((uint16_t)(gw[e] & 0xFFFFu)), g1 = bf((uint16_t)(gw[e] >> 16));
        const float u0 = bf((uint16_t)(uw[e] & 0xFFFFu)), u1 = bf((uint16_t)(uw[e] >> 16));
        const float a = g0 / (1.0f + expf(-g0)) * u0, b = g1 / (1.0f + expf(-g1)) * u1;
        o[e] = (uint32_t)to_bf(a) | ((uint32_t)to_bf(b) << 16);
    }
    y[i] = make_uint4(o[0], o[1], o[2], o[3]);
}

bool al16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool al8(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 7u) == 0; }

int launch_status()
{
    return cudaGetLastError() == cudaSuccess ? MX_OK : MX_ECUDA;
}

// One cuBLAS handle per host thread, created on first use.
thread_local cublasHandle_t t_blas = nullptr;

}  // namespace
}  // namespace mx

using namespace mx;

extern "C" {

int mx_rms_norm(const void *x, const void *w, void *y, int32_t rows, int32_t dim, float eps, void *stream)
{
    if (rows < 0 || dim <= 0 || dim % 8 || !(eps >= 0.f))
        return MX_EINVAL;
    if (rows == 0)
        return MX_OK;
    if (!x || !w || !y || !al16(x) || !al16(w) || !al16(y))
        return MX_EINVAL;
    const int warps = 8;
    rms_norm_kernel<<<(rows + warps - 1) / warps, 32 * warps, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(x), static_cast<const uint4 *>(w), static_cast<uint4 *>(y), rows, dim / 8, eps);
    return launch_status();
}

int mx_qk_norm_rope(const void *qkv, const void *q_norm, const void *k_norm, const int32_t *positions, void *q,
                    void *k, void *v, int32_t n_tokens, int32_t num_q_heads, int32_t num_kv_heads, float theta,
                    float eps, void *stream)
{
    if (n_tokens < 0 || num_q_heads <= 0 || num_kv_heads <= 0 || !(theta > 1.f) || !(eps >= 0.f))
        return MX_EINVAL;
    if (n_tokens == 0)
        return MX_OK;
    const void *ps[] = {qkv, q_norm, k_norm, positions, q, k, v};
    for (const void *p : ps)
        if (!p || !al8(p))
            return MX_EINVAL;
    const long long warps = (long long)n_tokens * (num_q_heads + 2 * num_kv_heads);
    const int per_block = 8;
    qk_norm_rope_kernel<<<(unsigned)((warps + per_block - 1) / per_block), 32 * per_block, 0,
                          static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint16_t *>(qkv), static_cast<const uint16_t *>(q_norm),
        static_cast<const uint16_t *>(k_norm), positions, static_cast<uint16_t *>(q), static_cast<uint16_t *>(k),
        static_cast<uint16_t *>(v), n_tokens, num_q_heads, num_kv_heads, theta, eps);
    return launch_status();
}

int mx_silu_mul(const void *gate_up, void *y, int32_t rows, int32_t d_ffn, void *stream)
{
    if (rows < 0 || d_ffn <= 0 || d_ffn % 8)
        return MX_EINVAL;
    if (rows == 0)
        return MX_OK;
    if (!gate_up || !y || !al16(gate_up) || !al16(y))
        return MX_EINVAL;
    const long long n = (long long)rows * (d_ffn / 8);
    silu_mul_kernel<<<(unsigned)((n + 255) / 256), 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(gate_up), static_cast<uint4 *>(y), rows, d_ffn / 8);
    return launch_status();
}

int mx_gemm(const void *a, const void *b, void *c, int32_t m, int32_t n, int32_t k, int32_t accumulate,
            void *stream)
{
    if (m < 0 || n <= 0 || k <= 0 || (accumulate != 0 && accumulate != 1))
        return MX_EINVAL;
    if (m == 0)
        return MX_OK;
    if (!a || !b || !c)
        return MX_EINVAL;
    if (!t_blas && cublasCreate(&t_blas) != CUBLAS_STATUS_SUCCESS) {
        t_blas = nullptr;
        return MX_ECUDA;
    }
    if (cublasSetStream(t_blas, static_cast<cudaStream_t>(stream)) != CUBLAS_STATUS_SUCCESS)
        return MX_ECUDA;
    const float alpha = 1.0f, beta = accumulate ? 1.0f : 0.0f;
    // row-major C[m,n] = A[m,k] B[k,n] is column-major C^T = B^T A^T
    const cublasStatus_t s = cublasGemmEx(t_blas, CUBLAS_OP_N, CUBLAS_OP_N, n, m, k, &alpha, b, CUDA_R_16BF, n, a,
                                          CUDA_R_16BF, k, &beta, c, CUDA_R_16BF, n, CUBLAS_COMPUTE_32F,
                                          CUBLAS_GEMM_DEFAULT);
    return s == CUBLAS_STATUS_SUCCESS ? MX_OK : MX_ECUDA;
}

}  // extern "C"
