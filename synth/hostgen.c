/* Host side of the seeded input generator, in C for speed (the numpy code in
 * synth/__init__.py is the readable definition; a test checks they agree bit
 * for bit).  value(i) = table[splitmix64(base + i) >> 44], SplitMix64 as
 * published by Steele, Lea and Flood (OOPSLA 2014).  No attention
 * arithmetic lives here. */
#include <stdint.h>

static inline uint64_t splitmix64(uint64_t x)
{
    uint64_t z = x + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

void synth_range(uint16_t *out, int64_t n, uint64_t base, uint64_t start, const uint16_t *table)
{
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i)
        out[i] = table[splitmix64(base + start + (uint64_t)i) >> 44];
}

void synth_pages(uint16_t *out, const int64_t *pages, int64_t n_pages, int64_t page_elems,
                 uint64_t base, const uint16_t *table)
{
#pragma omp parallel for schedule(static)
    for (int64_t p = 0; p < n_pages; ++p) {
        const uint64_t first = (uint64_t)pages[p] * (uint64_t)page_elems;
        uint16_t *o = out + p * page_elems;
        for (int64_t e = 0; e < page_elems; ++e)
            o[e] = table[splitmix64(base + first + (uint64_t)e) >> 44];
    }
}
