// Device side of the seeded input generator (see synth/__init__.py):
//   value(stream, i) = table[splitmix64(base + i) >> (64 - 20)]
// SplitMix64 as published by Steele, Lea and Flood (OOPSLA 2014).  Pure
// integer arithmetic, so host and device produce identical bits.  Holds no
// attention arithmetic; used only to lay down test and benchmark inputs.
#include <cstdint>
#include <cuda_runtime.h>

namespace {

__device__ __forceinline__ uint64_t splitmix64(uint64_t x)
{
    uint64_t z = x + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__global__ void fill_kernel(uint16_t *__restrict__ dst, long long n, unsigned long long base,
                            long long start, const uint16_t *__restrict__ table)
{
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long v = (long long)blockIdx.x * blockDim.x + threadIdx.x; v * 8 < n; v += stride) {
        const long long i0 = v * 8;
        if (i0 + 8 <= n) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const uint32_t lo = table[splitmix64(base + (uint64_t)(start + i0 + 2 * e)) >> 44];
                const uint32_t hi = table[splitmix64(base + (uint64_t)(start + i0 + 2 * e + 1)) >> 44];
                w[e] = lo | (hi << 16);
            }
            if ((reinterpret_cast<uintptr_t>(dst + i0) & 15u) == 0)
                *reinterpret_cast<uint4 *>(dst + i0) = make_uint4(w[0], w[1], w[2], w[3]);
            else
                for (int e = 0; e < 4; ++e) {
                    dst[i0 + 2 * e] = (uint16_t)(w[e] & 0xFFFFu);
                    dst[i0 + 2 * e + 1] = (uint16_t)(w[e] >> 16);
                }
        } else {
            for (long long i = i0; i < n; ++i)
                dst[i] = table[splitmix64(base + (uint64_t)(start + i)) >> 44];
        }
    }
}

}  // namespace

extern "C" int synth_fill(void *dst, long long n, unsigned long long base, long long start,
                          const void *table, void *stream)
{
    if (n <= 0)
        return 0;
    const long long vecs = (n + 7) / 8;
    long long grid = (vecs + 255) / 256;
    if (grid > 152LL * 16)
        grid = 152LL * 16;
    fill_kernel<<<(unsigned)grid, 256, 0, (cudaStream_t)stream>>>(
        (uint16_t *)dst, n, base, start, (const uint16_t *)table);
    return (int)cudaGetLastError();
}
