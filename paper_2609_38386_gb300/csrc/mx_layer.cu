// One layer of the mixed prefill/decode iteration in one persistent launch.
//
// Semantics (paper §2.1, Eq. 1 setting; §3.2 attention and KV layout
// unchanged): the |D_t| decode tokens and the p_t chunk tokens of one prompt
// append their K/V to their page slots and attend causally over the paged
// cache.  Query head h reads KV head h / (Hq / Hkv); scores are scaled by
// 1/sqrt(128); a decode with ctx cached tokens sees ctx + 1 keys; chunk row j
// sees keys [0, chunk_start + j].
//
// CTA: 12 warps.  Warpgroup 0 (warps 0-3, few registers) loads tiles and
// issues tensor-core MMAs; warpgroups 1 and 2 (the 256 "consumer" threads,
// many registers) run the softmax and epilogue of prefill items and the whole
// of decode items.  Each role runs its own copy of the persistent item loop;
// the roles meet at a named barrier between items.
//
// Work items (built on the host, fetched with one atomic counter):
//   ITEM_PREFILL {t, hq, heads, piece}: 128 chunk rows [128t, 128t+128) of
//                           query heads hq (and hq + 1 when heads = 2, the
//                           same KV head) against one contiguous range of
//                           their key tiles, on tcgen05 tensor cores (S and O
//                           accumulators of both heads in TMEM, one K/V tile
//                           load for both).  Warp 0 loads Q and K, warp 2 V,
//                           warp 1 issues the MMAs; consumer warpgroup e runs
//                           the softmax of head hq + e.  A tile with several
//                           pieces writes (O, lse) partials; the last-arriving
//                           piece merges them.  Piece 0 of each of the
//                           n_rep / heads items of a KV head appends its share
//                           of the tile's tokens to the KV cache.
//   ITEM_DECODE  {h, s | i | seq | ctx}: split s of decode i's keys for KV
//                           head h, all n_rep query heads of the group at
//                           once: a split-KV flash-decode whose partial
//                           (O, lse) is merged by the last-arriving split (no
//                           waiting).
//   ITEM_DECODE_SHORT: a decode of at most 16 keys, exact on CUDA cores.
// New keys/values are read from the k/v inputs, never from the pages being
// written in the same launch, so the append needs no ordering.
#include "mx_internal.h"
#include "mx_ptx.cuh"

#include <cuda_bf16.h>
#include <cuda_runtime.h>

namespace mx {

struct Misc {
    uint64_t bar_q;                   // Q tiles of the item landed
    uint64_t bar_kfull[kKStages];     // K tile landed
    uint64_t bar_kempty[kKStages];    // both heads' S = Q K^T of that tile done
    uint64_t bar_vfull[kVStagesMax];  // V tile landed
    uint64_t bar_vempty[kVStagesMax]; // both heads' P V of that tile done
    uint64_t bar_sfull[2];            // S_h ready for head h's softmax
    uint64_t bar_pfull[2];            // P_h written by head h's 128 softmax threads
    uint64_t bar_odone;               // every MMA of the item done
    uint64_t bar_never;               // fault injection: a barrier nothing arrives at
    uint32_t tmem_base;
    int32_t item_idx[2];
    int32_t abort;
    int32_t last;
    int32_t n_items;                  // work items of the launch
    int32_t n_pre;                    // items [0, n_pre) are prefill items
    int32_t dec_first;                // this CTA draws decode items first (1) or prefill items (0)
    int32_t queue;                    // thread 0's queue: 0 its first, 1 the other, 2 none left
    int32_t has_prefill;              // the launch has prefill items (TMEM allocated)
    PrefillInfo pre[kMaxPrefills];    // the launch's prefill chunks
};
static_assert(sizeof(Misc) <= kSmemMiscBytes, "misc block too large");

// Named barriers: 1 = every thread of the CTA between items, 2 = the 256
// consumer threads (0 is __syncthreads, used only outside the item loops).
constexpr uint32_t kBarItem = 1, kBarCons = 2;
constexpr uint32_t kBarHead0 = 3;   // kBarHead0 + e: the 128 threads of head slot e's softmax
__device__ __forceinline__ void cons_sync() { named_sync(kBarCons, kConsThreads); }

// Instruction descriptors: S = Q K^T (both K-major) and O = P V (V MN-major).
constexpr uint32_t kIdescS = idesc_bf16_f32(128, 128, false, false);
constexpr uint32_t kIdescO = idesc_bf16_f32(128, 128, false, true);
constexpr uint32_t kSwz128 = 2;

__device__ __forceinline__ void flag_error(const LayerParams &P, uint32_t bit)
{
    atomicOr(P.err, bit);
}

__device__ __forceinline__ void set_abort(const LayerParams &P, Misc *misc)
{
    *(volatile int32_t *)&misc->abort = 1;
    flag_error(P, ERR_TIMEOUT);
}

__device__ __forceinline__ float neg_inf() { return -__int_as_float(0x7f800000); }

// ---------------------------------------------------------------------------
// A decode of at most kShortKeys keys, KV head h: exact fp32 attention on the
// CUDA cores (the bf16 rounding of one dominant weight of P in the
// tensor-core path would show in the output).  The scores go through shared
// memory; cached K/V rows are read from their pages, the new key from the k/v
// inputs (as in the split path), which it appends.
// ---------------------------------------------------------------------------
__device__ void decode_short_item(const LayerParams &P, uint8_t *smem, int di, int h, int seq, int n, int tid)
{
    const int nrep = P.n_rep, nk = n + 1;   // tid: consumer thread 0..255
    float *ss = reinterpret_cast<float *>(smem);   // [kMaxRep][kShortKeys] scores (log2 domain)
    int *spid = reinterpret_cast<int *>(ss + kMaxRep * kShortKeys);   // page of each cached key's page
    if (tid < 32) {
        const int slot = P.slots[di];
        if (slot >= P.num_pages * kPage) {
            if (tid == 0)
                flag_error(P, ERR_SLOT);
        } else if (slot >= 0) {
            const size_t dst = (((size_t)(slot / kPage) * P.hkv + h) * kPage + slot % kPage) * kHeadDim;
            const size_t src = ((size_t)di * P.hkv + h) * kHeadDim;
            const int c = tid & 15;
            if (tid < 16)
                reinterpret_cast<uint4 *>(P.k_pool + dst)[c] = __ldg(reinterpret_cast<const uint4 *>(P.k + src) + c);
            else
                reinterpret_cast<uint4 *>(P.v_pool + dst)[c] = __ldg(reinterpret_cast<const uint4 *>(P.v + src) + c);
        }
    } else if (tid < 32 + kShortKeys / kPage) {
        const int lp = tid - 32;   // page index of the sequence
        int pid = -1;
        if (lp * kPage < n) {
            pid = __ldg(P.page_table + (size_t)seq * P.max_pages + lp);
            if (pid < 0 || pid >= P.num_pages) {
                flag_error(P, ERR_PAGE);
                pid = -1;
            }
        }
        spid[lp] = pid;
    }
    cons_sync();
    const uint16_t *knew = P.k + ((size_t)di * P.hkv + h) * kHeadDim;
    const uint16_t *vnew = P.v + ((size_t)di * P.hkv + h) * kHeadDim;
    for (int e = tid; e < nrep * kShortKeys; e += kConsThreads) {
        const int q = e / kShortKeys, k = e % kShortKeys;
        float s = neg_inf();
        const int pid = k < n ? spid[k / kPage] : -1;
        if (q < nrep && k < nk && (k == n || pid >= 0)) {
            const uint4 *qr = reinterpret_cast<const uint4 *>(P.q + ((size_t)di * P.hq + h * nrep + q) * kHeadDim);
            const uint4 *kr = reinterpret_cast<const uint4 *>(
                k < n ? P.k_pool + (((size_t)pid * P.hkv + h) * kPage + k % kPage) * kHeadDim : knew);
            float acc = 0.f;
#pragma unroll 4
            for (int c = 0; c < 16; ++c) {
                const uint4 a = __ldg(qr + c), b = __ldg(kr + c);
                const uint32_t aw[4] = {a.x, a.y, a.z, a.w}, bw[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
                for (int x = 0; x < 4; ++x)
                    acc += bf16lo(aw[x]) * bf16lo(bw[x]) + bf16hi(aw[x]) * bf16hi(bw[x]);
            }
            s = acc * P.scale_log2;
        }
        ss[q * kShortKeys + k] = s;
    }
    cons_sync();
    for (int e = tid; e < nrep * kHeadDim; e += kConsThreads) {
        const int q = e / kHeadDim, d = e % kHeadDim;
        float m = neg_inf();
        for (int k = 0; k < nk; ++k)
            m = fmaxf(m, ss[q * kShortKeys + k]);
        float l = 0.f, o = 0.f;
        for (int k = 0; k < nk; ++k) {
            const float sk = ss[q * kShortKeys + k];
            if (sk == neg_inf())
                continue;
            const float pk = ex2(sk - m);
            const int pid = k < n ? spid[k / kPage] : -1;
            const uint16_t vb =
                k < n ? P.v_pool[(((size_t)pid * P.hkv + h) * kPage + k % kPage) * kHeadDim + d] : vnew[d];
            l += pk;
            o += pk * __uint_as_float((uint32_t)vb << 16);
        }
        __nv_bfloat16 b = __float2bfloat16_rn(o / l);
        P.out[((size_t)di * P.hq + h * nrep + q) * kHeadDim + d] = *reinterpret_cast<uint16_t *>(&b);
    }
}

// ---------------------------------------------------------------------------
// Decode split: keys [k_lo, k_hi) of decode di, KV head h.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void decode_issue_page(const LayerParams &P, uint32_t stage,
                                                  int pid, int kb, int n, int k_hi, int di,
                                                  int h, int lane, uint64_t pol)
{
    const size_t pbase = ((size_t)(pid < 0 ? 0 : pid) * P.hkv + h) * kPage * kHeadDim;
    if (pid >= 0 && kb + kPage <= n && kb + kPage <= k_hi) {
        // a whole cached page (the common case): no per-row selection
        const int c = lane & 15, r0 = lane >> 4;
        const size_t off = pbase + r0 * kHeadDim + c * 8;
        const uint16_t *ks = P.k_pool + off, *vs = P.v_pool + off;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int row = r0 + 2 * e;
            const uint32_t dst = stage + row * 256 + ((c ^ (row & 7)) << 4);
            cp_async16_hint(dst, ks + 2 * e * kHeadDim, 16u, pol);
            cp_async16_hint(dst + kPageBytes, vs + 2 * e * kHeadDim, 16u, pol);
        }
        return;
    }
    const uint16_t *kin = P.k + ((size_t)di * P.hkv + h) * kHeadDim;
    const uint16_t *vin = P.v + ((size_t)di * P.hkv + h) * kHeadDim;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
        const int ci = lane + 32 * e;  // 16-byte chunk of the 16 x 256 B page tile
        const int row = ci >> 4, c = ci & 15;
        const int key = kb + row;
        const uint16_t *ks, *vs;
        uint32_t bytes = key < k_hi ? 16u : 0u;
        if (key < n) {
            ks = P.k_pool + pbase + row * kHeadDim + c * 8;
            vs = P.v_pool + pbase + row * kHeadDim + c * 8;
            if (pid < 0)
                bytes = 0;
        } else {
            ks = kin + c * 8;  // key == n: the decode's own new key
            vs = vin + c * 8;
            if (key != n)
                bytes = 0;
        }
        const uint32_t dst = stage + row * 256 + ((c ^ (row & 7)) << 4);
        cp_async16_hint(dst, ks, bytes, pol);
        cp_async16_hint(dst + kPageBytes, vs, bytes, pol);
    }
}

__device__ void decode_item(const LayerParams &P, uint8_t *smem, Misc *misc, int di, int h,
                            int s, int seq, int n, int split_len, int tid)
{
    // tid: consumer thread 0..255, warp: decode warp 0..7
    const int warp = tid >> 5, lane = tid & 31;
    // split count and partial slots are needed only at the end: the load
    // overlaps the page-id loads (the row and length came with the item)
    const DecodeInfo D = P.dec[di];
    const int nrep = P.n_rep;
    const int k_lo = s * split_len;
    const int k_hi = min(k_lo + split_len, n + 1);
    const int pg_lo = k_lo / kPage;
    const int npg = (k_hi - k_lo + kPage - 1) / kPage;
    const int g = lane >> 2, tq = lane & 3;

    // The split holding the new key appends it (each slot written once).
    if (k_hi == n + 1 && warp == 0) {
        const int slot = P.slots[di];
        if (slot >= 0) {
            if (slot >= P.num_pages * kPage) {
                if (lane == 0)
                    flag_error(P, ERR_SLOT);
            } else {
                const size_t dst = (((size_t)(slot / kPage) * P.hkv + h) * kPage + slot % kPage) * kHeadDim;
                const size_t src = ((size_t)di * P.hkv + h) * kHeadDim;
                const int c = lane & 15;
                if (lane < 16)
                    reinterpret_cast<uint4 *>(P.k_pool + dst)[c] =
                        __ldg(reinterpret_cast<const uint4 *>(P.k + src) + c);
                else
                    reinterpret_cast<uint4 *>(P.v_pool + dst)[c] =
                        __ldg(reinterpret_cast<const uint4 *>(P.v + src) + c);
            }
        }
    }

    // Q^T fragments (B operand of S^T = K Q^T): query row g of the group.
    uint32_t qb[8][2];
    {
        const uint16_t *qrow = P.q + ((size_t)di * P.hq + h * nrep + (g < nrep ? g : 0)) * kHeadDim;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            if (g < nrep) {
                qb[kk][0] = __ldg(reinterpret_cast<const uint32_t *>(qrow + kk * 16 + 2 * tq));
                qb[kk][1] = __ldg(reinterpret_cast<const uint32_t *>(qrow + kk * 16 + 8 + 2 * tq));
            } else {
                qb[kk][0] = qb[kk][1] = 0u;
            }
        }
    }

    // This warp's pages: local indices warp, warp + 8, ...
    const int my_n = npg > warp ? (npg - warp + kWarps - 1) / kWarps : 0;
    int pid_l = -1;
    if (lane < my_n) {
        const int lp = pg_lo + warp + kWarps * lane;
        if (lp * kPage < n) {  // pages holding cached keys only
            int pid = __ldg(P.page_table + (size_t)seq * P.max_pages + lp);
            if (pid < 0 || pid >= P.num_pages) {
                flag_error(P, ERR_PAGE);
                pid = -1;
            }
            pid_l = pid;
        }
    }

    const uint32_t ring = smem_u32(smem) + warp * (kDecStages * kDecStageBytes);
    // the pages stream through once: evict_first keeps them from displacing
    // the prefill's K/V tiles, which several query heads and tiles re-read
    const uint64_t pol = l2_policy_evict_first();
    float acc[8][4];
#pragma unroll
    for (int mt = 0; mt < 8; ++mt)
        acc[mt][0] = acc[mt][1] = acc[mt][2] = acc[mt][3] = 0.f;
    float m0 = neg_inf(), m1 = neg_inf(), l0 = 0.f, l1 = 0.f;
    const float sl = P.scale_log2;

#pragma unroll
    for (int k = 0; k < kDecStages - 1; ++k) {
        const int pid = __shfl_sync(0xffffffffu, pid_l, k & 31);
        if (k < my_n)
            decode_issue_page(P, ring + k * kDecStageBytes, pid,
                              (pg_lo + warp + kWarps * k) * kPage, n, k_hi, di, h, lane, pol);
        cp_async_commit();
    }

    for (int k = 0; k < my_n; ++k) {
        {
            const int kn = k + kDecStages - 1;
            const int pid = __shfl_sync(0xffffffffu, pid_l, kn & 31);
            if (kn < my_n)
                decode_issue_page(P, ring + (kn % kDecStages) * kDecStageBytes, pid,
                                  (pg_lo + warp + kWarps * kn) * kPage, n, k_hi, di, h, lane, pol);
            cp_async_commit();
        }
        cp_async_wait<kDecStages - 1>();
        __syncwarp();

        const uint32_t kbase = ring + (k % kDecStages) * kDecStageBytes;
        const uint32_t vbase = kbase + kPageBytes;
        const int kb = (pg_lo + warp + kWarps * k) * kPage;
        const int nv = min(kPage, k_hi - kb);  // valid keys in this page (>= 1)

        // S^T (16 keys x 8 query rows) = K (16 x 128) * Q^T (128 x 8), in two
        // independent accumulation chains (even and odd 16-dim steps) so that
        // consecutive MMAs do not wait for each other
        float sc[4];
        {
            float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
            const int mi = lane >> 3;
            const int row = (lane & 7) + (mi & 1) * 8;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                const int chunk = kk * 2 + (mi >> 1);
                uint32_t a0, a1, a2, a3;
                ldsm_x4(kbase + row * 256 + ((chunk ^ (row & 7)) << 4), a0, a1, a2, a3);
                mma_bf16_16816((kk & 1) ? sb : sa, a0, a1, a2, a3, qb[kk][0], qb[kk][1]);
            }
#pragma unroll
            for (int x = 0; x < 4; ++x)
                sc[x] = sa[x] + sb[x];
        }
        // online softmax over this page's keys (log2 domain), per query column
        const float x0 = g < nv ? sc[0] * sl : neg_inf();
        const float x1 = g < nv ? sc[1] * sl : neg_inf();
        const float x2 = g + 8 < nv ? sc[2] * sl : neg_inf();
        const float x3 = g + 8 < nv ? sc[3] * sl : neg_inf();
        float mx0 = fmaxf(x0, x2), mx1 = fmaxf(x1, x3);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, o));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
        }
        // Lazy rescale: the running max moves (and O and l are rescaled) only
        // when some column's max grows by more than 8 in log2 units, so p
        // stays below 2^8; most pages skip the 32 multiplications.
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
        if (__any_sync(0xffffffffu, mn0 > m0 + 8.0f || mn1 > m1 + 8.0f)) {
            const float al0 = ex2(m0 - mn0), al1 = ex2(m1 - mn1);
            l0 *= al0;
            l1 *= al1;
            m0 = mn0;
            m1 = mn1;
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                acc[mt][0] *= al0;
                acc[mt][1] *= al1;
                acc[mt][2] *= al0;
                acc[mt][3] *= al1;
            }
        }
        const float p0 = ex2(x0 - m0), p1 = ex2(x1 - m1);
        const float p2 = ex2(x2 - m0), p3 = ex2(x3 - m1);
        l0 += p0 + p2;
        l1 += p1 + p3;
        // P^T as the B operand (keys x query rows): transpose the 8x8 blocks
        // (decodes of at most 16 keys, where the bf16 rounding of one weight
        // would show, are ITEM_DECODE_SHORT items and never come here)
        const uint32_t b0 = movmatrix_t(pack_bf16(p0, p1));
        const uint32_t b1 = movmatrix_t(pack_bf16(p2, p3));
        // O^T (128 d x 8 rows) += V^T (128 x 16 keys) * P^T (16 x 8)
        {
            const int mi = lane >> 3;
            const int key = (lane & 7) + (mi >> 1) * 8;
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                const int chunk = mt * 2 + (mi & 1);
                uint32_t a0, a1, a2, a3;
                ldsm_x4_t(vbase + key * 256 + ((chunk ^ (key & 7)) << 4), a0, a1, a2, a3);
                mma_bf16_16816(acc[mt], a0, a1, a2, a3, b0, b1);
            }
        }
        __syncwarp();
    }
    cp_async_wait<0>();

#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
        l0 += __shfl_xor_sync(0xffffffffu, l0, o);
        l1 += __shfl_xor_sync(0xffffffffu, l1, o);
    }

    // ---- combine the 8 decode warps (shared memory)
    cons_sync();
    float *so = reinterpret_cast<float *>(smem);               // [warp][8][128]
    float *sml = so + kWarps * kMaxRep * kHeadDim;              // [warp][8][2]
#pragma unroll
    for (int mt = 0; mt < 8; ++mt) {
        const int d = mt * 16 + g;
        so[(warp * kMaxRep + 2 * tq) * kHeadDim + d] = acc[mt][0];
        so[(warp * kMaxRep + 2 * tq + 1) * kHeadDim + d] = acc[mt][1];
        so[(warp * kMaxRep + 2 * tq) * kHeadDim + d + 8] = acc[mt][2];
        so[(warp * kMaxRep + 2 * tq + 1) * kHeadDim + d + 8] = acc[mt][3];
    }
    if (g == 0) {
        sml[(warp * kMaxRep + 2 * tq) * 2 + 0] = m0;
        sml[(warp * kMaxRep + 2 * tq) * 2 + 1] = l0;
        sml[(warp * kMaxRep + 2 * tq + 1) * 2 + 0] = m1;
        sml[(warp * kMaxRep + 2 * tq + 1) * 2 + 1] = l1;
    }
    cons_sync();

    const int nsp = D.n_splits;
    const int pslot = D.part_base + h * nsp + s;
    for (int e = tid; e < nrep * kHeadDim; e += kConsThreads) {
        const int q = e / kHeadDim, d = e % kHeadDim;
        float M = neg_inf();
#pragma unroll
        for (int w = 0; w < kWarps; ++w)
            M = fmaxf(M, sml[(w * kMaxRep + q) * 2]);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const float f = ex2(sml[(w * kMaxRep + q) * 2] - M);
            L += f * sml[(w * kMaxRep + q) * 2 + 1];
            O += f * so[(w * kMaxRep + q) * kHeadDim + d];
        }
        const float res = O / L;
        if (nsp == 1) {
            __nv_bfloat16 b = __float2bfloat16_rn(res);
            P.out[((size_t)di * P.hq + h * nrep + q) * kHeadDim + d] =
                *reinterpret_cast<uint16_t *>(&b);
        } else {
            P.part_o[((size_t)pslot * kMaxRep + q) * kHeadDim + d] = res;
            if (d == 0) {
                float lg;
                asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(lg) : "f"(L));
                P.part_lse[(size_t)pslot * kMaxRep + q] = M + lg;
            }
        }
    }
    if (nsp == 1)
        return;

    // ---- cross-split merge by the last-arriving split (no waiting)
    __threadfence();
    cons_sync();
    if (tid == 0) {
        const uint32_t prev = atomicAdd(P.merge_cnt + di * P.hkv + h, 1u);
        misc->last = (prev == (uint32_t)(nsp - 1)) ? 1 : 0;
    }
    cons_sync();
    if (!misc->last)
        return;
    __threadfence();
    // Every partial is read once, eight splits' (lse, 4 columns of O) at a
    // time with all their loads in flight, the max and the weight sum kept
    // online (a rescale per group): the merge sits on this split's critical
    // path, so its loads must not form a chain of round trips.
    const int base = D.part_base + h * nsp;
    for (int e = tid; e < nrep * (kHeadDim / 4); e += kConsThreads) {
        const int q = e / (kHeadDim / 4), d4 = e % (kHeadDim / 4);
        float M = neg_inf(), W = 0.f;
        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s0 = 0; s0 < nsp; s0 += 8) {
            float l[8];
            float4 o[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int sp = s0 + u;
                l[u] = neg_inf();
                o[u] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (sp < nsp) {
                    const size_t row = (size_t)(base + sp) * kMaxRep + q;
                    l[u] = __ldcg(P.part_lse + row);
                    o[u] = __ldcg(reinterpret_cast<const float4 *>(P.part_o + row * kHeadDim) + d4);
                }
            }
            float mb = M;
#pragma unroll
            for (int u = 0; u < 8; ++u)
                mb = fmaxf(mb, l[u]);
            const float c = ex2(M - mb);   // 0 for the first group (M = -inf)
            W *= c;
            O.x *= c;
            O.y *= c;
            O.z *= c;
            O.w *= c;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const float f = ex2(l[u] - mb);   // 0 past the last split
                W += f;
                O.x += f * o[u].x;
                O.y += f * o[u].y;
                O.z += f * o[u].z;
                O.w += f * o[u].w;
            }
            M = mb;
        }
        const float inv = 1.0f / W;
        uint2 pk;
        pk.x = pack_bf16(O.x * inv, O.y * inv);
        pk.y = pack_bf16(O.z * inv, O.w * inv);
        reinterpret_cast<uint2 *>(P.out + ((size_t)di * P.hq + h * nrep + q) * kHeadDim)[d4] = pk;
    }
    if (tid == 0)
        P.merge_cnt[di * P.hkv + h] = 0u;
}

// Keys [r0, end of r0's page) of the last cached tile are not cached yet (the
// chunk's own keys start there): zero their value rows in the staged V tile
// so that P.V adds nothing for them (later pages were zero-filled by TMA).
__device__ __forceinline__ void clear_uncached_rows(uint32_t dv, int r0)
{
    const int r1 = min(kTileN, (r0 + kPage - 1) / kPage * kPage);
#pragma unroll 1
    for (int r = r0; r < r1; ++r)
#pragma unroll 1
        for (int hf = 0; hf < 2; ++hf)
#pragma unroll 1
            for (int cc = 0; cc < 8; ++cc)
                asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(dv + hf * kHalfTile + r * 128 + cc * 16),
                             "r"(0u)
                             : "memory");
    fence_proxy_async_smem();
}

// Zero value rows [r0, r1) of a staged V tile (two SW128 halves).
__device__ __forceinline__ void zero_v_rows(uint32_t dv, int r0, int r1)
{
#pragma unroll 1
    for (int r = r0; r < r1; ++r)
#pragma unroll 1
        for (int hf = 0; hf < 2; ++hf)
#pragma unroll 1
            for (int cc = 0; cc < 8; ++cc)
                asm volatile("st.shared.v4.u32 [%0], {%1,%1,%1,%1};" ::"r"(dv + hf * kHalfTile + r * 128 + cc * 16),
                             "r"(0u)
                             : "memory");
    fence_proxy_async_smem();
}

// Row max of the raw scores of one S row held in registers (the scale is
// positive), 8 independent three-input chains.
__device__ __forceinline__ float row_max(const uint32_t (&sv)[128])
{
    float mx8[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
        mx8[u] = neg_inf();
#pragma unroll
    for (int cc = 0; cc < 64; ++cc) {
        mx8[cc & 7] = max3(mx8[cc & 7], __uint_as_float(sv[2 * cc]), __uint_as_float(sv[2 * cc + 1]));
    }
    return fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                 fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
}

// p = 2^(s*scale - m) of one S row as bf16 pairs into TMEM at taddr (64
// columns, stored 16 at a time), and the row sum of p in 4 packed pair
// chains: of p as computed, or (kRoundedSum) of p as rounded to bf16, the
// weights P.V actually uses.
template <bool kRoundedSum>
__device__ __forceinline__ float row_exp_store(const uint32_t (&sv)[128], float sl, float nm, uint32_t taddr)
{
    float rs8[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
        rs8[u] = 0.f;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint32_t pk[16];
#pragma unroll
        for (int cc = 0; cc < 16; ++cc) {
            const int k0 = 32 * q + 2 * cc;
            float x0, x1;
            ffma2(x0, x1, __uint_as_float(sv[k0]), __uint_as_float(sv[k0 + 1]), sl, sl, nm, nm);
            const float e0 = ex2(x0), e1 = ex2(x1);
            pk[cc] = pack_bf16(e0, e1);
            if (kRoundedSum)
                fadd2(rs8[2 * (cc & 3)], rs8[2 * (cc & 3) + 1], bf16lo(pk[cc]), bf16hi(pk[cc]));
            else
                fadd2(rs8[2 * (cc & 3)], rs8[2 * (cc & 3) + 1], e0, e1);
        }
        tmem_st16(taddr + 16 * q, pk);
    }
    return ((rs8[0] + rs8[1]) + (rs8[2] + rs8[3])) + ((rs8[4] + rs8[5]) + (rs8[6] + rs8[7]));
}

// 16-byte chunk c (8 elements) of row `row` of a 128 x 128 bf16 tile held as
// two SW128 halves of 64 columns (128-byte rows), as the TMA loads write it.
__device__ __forceinline__ uint4 sw128_chunk(uint32_t base, int row, int c)
{
    const uint32_t a = base + (uint32_t)(c >> 3) * kHalfTile + row * 128 + ((((c & 7) ^ (row & 7))) << 4);
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

// Chunk row r of a chunk that starts at position cs, with cs + r <
// kShortRowKeys, attends only keys 0..cs+r.  With so few keys the bf16 rounding
// of a dominant weight of P would show in the output, so such a row is
// recomputed here in fp32 from the tiles still in shared memory and its
// output row overwritten: key k < cs is row k of the cached tile (sKa, sVa:
// the item's first key tile), key k >= cs is row k - cs of the chunk's own
// first tile (sKb, sVb).
__device__ __forceinline__ void short_row_exact(uint32_t sQ, uint32_t sKa, uint32_t sVa, uint32_t sKb,
                                                uint32_t sVb, int cs, int r, float sl, uint16_t *orow)
{
    const int last = cs + r;   // keys 0..last, last < kShortRowKeys
    float s[kShortRowKeys];
#pragma unroll
    for (int k = 0; k < kShortRowKeys; ++k)
        s[k] = 0.f;
#pragma unroll 1
    for (int c = 0; c < 16; ++c) {
        const uint4 q4 = sw128_chunk(sQ, r, c);
        const uint32_t qw[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
        for (int k = 0; k < kShortRowKeys; ++k) {
            if (k <= last) {
                const uint4 k4 = k < cs ? sw128_chunk(sKa, k, c) : sw128_chunk(sKb, k - cs, c);
                const uint32_t kw[4] = {k4.x, k4.y, k4.z, k4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    s[k] += bf16lo(qw[e]) * bf16lo(kw[e]) + bf16hi(qw[e]) * bf16hi(kw[e]);
            }
        }
    }
    float m = neg_inf();
#pragma unroll
    for (int k = 0; k < kShortRowKeys; ++k)
        if (k <= last)
            m = fmaxf(m, s[k] * sl);
    float l = 0.f;
#pragma unroll
    for (int k = 0; k < kShortRowKeys; ++k) {
        s[k] = k <= last ? ex2(s[k] * sl - m) : 0.f;
        l += s[k];
    }
    const float inv = 1.0f / l;
#pragma unroll 1
    for (int c = 0; c < 16; ++c) {
        float acc[8];
#pragma unroll
        for (int e = 0; e < 8; ++e)
            acc[e] = 0.f;
#pragma unroll
        for (int k = 0; k < kShortRowKeys; ++k) {
            if (k <= last) {
                const uint4 v4 = k < cs ? sw128_chunk(sVa, k, c) : sw128_chunk(sVb, k - cs, c);
                const uint32_t vw[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc[2 * e] += s[k] * bf16lo(vw[e]);
                    acc[2 * e + 1] += s[k] * bf16hi(vw[e]);
                }
            }
        }
        uint4 o4;
        o4.x = pack_bf16(acc[0] * inv, acc[1] * inv);
        o4.y = pack_bf16(acc[2] * inv, acc[3] * inv);
        o4.z = pack_bf16(acc[4] * inv, acc[5] * inv);
        o4.w = pack_bf16(acc[6] * inv, acc[7] * inv);
        reinterpret_cast<uint4 *>(orow)[c] = o4;
    }
}

// ---------------------------------------------------------------------------
// Prefill item: rows [128t, 128t + 128) of the chunk, query heads hq0 ..
// hq0 + nh - 1 (one KV head), key tiles kt0 .. kt1 - 1 of the tile's nA + t + 1
// (nA paged tiles covering [0, chunk_start), then t + 1 tiles of the chunk's
// own keys read from the k/v inputs).  Counters carried across items give the
// barrier phases: tile0 = K/V tiles this CTA loaded before the item, item_no
// = prefill items before it, sph[e] = S/P phases head slot e completed.
// ---------------------------------------------------------------------------
struct PrefillArgs {
    int f, t, hq0, nh, s, ns, kt0, kt1, part_base;
    uint32_t tile0, item_no, sph0, sph1;
};

__device__ __forceinline__ PrefillArgs prefill_args(const int4 it, const Misc *misc, uint32_t tile_cnt,
                                                    uint32_t item_no, const uint32_t (&sph)[2])
{
    PrefillArgs a;
    a.f = (int)(((uint32_t)it.x >> 4) & 0xFu);
    a.nh = (int)(((uint32_t)it.x >> 8) & 1u) + 1;
    a.t = it.y & 0xFFFF;
    a.hq0 = it.y >> 16;
    a.s = it.z & 0xFFFF;
    a.ns = it.z >> 16;
    const int nT = (misc->pre[a.f].chunk_start + kTileN - 1) / kTileN + a.t + 1;
    a.kt0 = (int)((long long)a.s * nT / a.ns);
    a.kt1 = (int)((long long)(a.s + 1) * nT / a.ns);
    a.part_base = it.w;
    a.tile0 = tile_cnt;
    a.item_no = item_no;
    a.sph0 = sph[0];
    a.sph1 = sph[1];
    return a;
}

// Warp 0 (Q and K) or warp 2 (V): the item's tiles into a ring of `nst`
// stages; each stage waits only on its own "empty" barrier.  Cached tiles
// are one 2-D {64,16} box per (page, head) half from the pool map (a missing
// page reads an out-of-range row, zero filled), the chunk's own keys one 3-D
// box per half from the k/v map.  Page ids are read four tiles (32 pages, one
// per lane) at a time, one batch ahead: a page-table read under load takes
// about as long as a whole tile, so it must not sit in the issue loop.
__device__ void prefill_load_ring(const LayerParams &P, Misc *misc, const PrefillArgs &a, bool isK,
                                  uint32_t ring, int lane)
{
    const PrefillInfo &pf = misc->pre[a.f];
    const int kvh = a.hq0 / P.n_rep;
    const int cs = pf.chunk_start, tb = pf.token_base;
    const int nA = (cs + kTileN - 1) / kTileN;
    const int nT = a.kt1 - a.kt0;
    const int nst = isK ? kKStages : P.v_stages;
    const void *tm_pool = isK ? (const void *)&P.tm_kpool : (const void *)&P.tm_vpool;
    const void *tm_in = isK ? (const void *)&P.tm_k : (const void *)&P.tm_v;
    uint64_t *full = isK ? misc->bar_kfull : misc->bar_vfull;
    uint64_t *empty = isK ? misc->bar_kempty : misc->bar_vempty;
    volatile int *abort = &misc->abort;
    const uint64_t tmo = P.timeout_ns;
    const int oob_row = P.num_pages * P.hkv * kPage;
    const int32_t *prow = P.page_table + (size_t)pf.seq * P.max_pages;
    auto fetch_pids = [&](int i0) {
        const int lp = (a.kt0 + i0 + (lane >> 3)) * 8 + (lane & 7);
        int pid = -1;
        if (i0 + (lane >> 3) < nT && lp * kPage < cs) {
            pid = __ldg(prow + lp);
            if (pid < 0 || pid >= P.num_pages) {
                if (isK)
                    flag_error(P, ERR_PAGE);
                pid = -1;
            }
        }
        return pid;
    };
    int pid_cur = fetch_pids(0), pid_next = fetch_pids(4);
    // ring stage and phase of tile a.tile0 + i, advanced without a division
    int st = (int)(a.tile0 % (uint32_t)nst);
    uint32_t ph = (a.tile0 / (uint32_t)nst) & 1;
    for (int i = 0; i < nT; ++i, st = st + 1 == nst ? 0 : st + 1, ph ^= st == 0 ? 1u : 0u) {
        const int gi = a.kt0 + i;
        if (i > 0 && (i & 3) == 0) {
            pid_cur = pid_next;
            pid_next = fetch_pids(i + 4);
        }
        int ok = 1;
        if (lane == 0 && !mbar_wait(smem_u32(&empty[st]), ph ^ 1, abort, tmo)) {
            set_abort(P, misc);
            ok = 0;
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok)
            break;
        const uint32_t fb = smem_u32(&full[st]);
        const uint32_t dst = ring + st * kTileBytes;
        if (gi < nA) {
#pragma unroll
            for (int pg = 0; pg < 8; ++pg) {
                const int pid = __shfl_sync(0xffffffffu, pid_cur, (i & 3) * 8 + pg);
                if (lane == 0) {
                    if (pg == 0)
                        mbar_expect_tx(fb, kTileBytes);
                    const int y = pid >= 0 ? (pid * P.hkv + kvh) * kPage : oob_row;
                    tma_load_2d(dst + pg * 2048, tm_pool, fb, 0, y);
                    tma_load_2d(dst + kHalfTile + pg * 2048, tm_pool, fb, 64, y);
                }
            }
        } else if (lane == 0) {
            mbar_expect_tx(fb, kTileBytes);
            const int z = tb + kTileN * (gi - nA);
            tma_load_3d(dst, tm_in, fb, 0, kvh, z);
            tma_load_3d(dst + kHalfTile, tm_in, fb, 64, kvh, z);
        }
    }
}

// Warp 1, one thread: every MMA of the item.  Per key tile j (the loop runs
// one step past the last tile for the final P.V):
//   [P_0(j-1) written]  O_0 += P_0 V_{j-1}   [K_j landed]  S_0 = Q_0 K_j -> sfull[0]
//   [P_1(j-1) written]  O_1 += P_1 V_{j-1}                 S_1 = Q_1 K_j -> sfull[1]
//   -> kempty (K_j free), vempty (V_{j-1} free)
// so the softmax of head 0 for tile j runs while the tensor pipe works on
// head 1's P.V and S, and the other way round.  S_h = Q_h K_j overwrites the
// TMEM columns that P_h(j-1) occupied; it is issued after P_h(j-1) V_{j-1},
// and the pipe executes in order.  A commit covers every earlier MMA of the
// thread, so sfull[h] of tile j also says that O_h += P_h V_{j-1} is done.
template <bool kReplay>
__device__ void prefill_mma(const LayerParams &P, Misc *misc, const PrefillArgs &a, uint32_t tmem,
                            uint32_t sbase)
{
    const PrefillInfo &pf = misc->pre[a.f];
    const int cs = pf.chunk_start;
    const int nA = (cs + kTileN - 1) / kTileN;
    const int nT = a.kt1 - a.kt0;
    volatile int *abort = &misc->abort;
    const uint64_t tmo = P.timeout_ns;
    const uint32_t sK = sbase + kSmemK, sV = sbase + kSmemV;
    const uint32_t vst = (uint32_t)P.v_stages;
    // V stage and phase of the tile whose P.V comes next, advanced without a
    // division (the ring depth is a launch parameter)
    uint32_t vs = a.tile0 % vst, vph = (a.tile0 / vst) & 1;
    // Steps whose V tile needs rows zeroed (-1: none), computed once: clr_a,
    // the last cached tile, whose rows past chunk_start are not cached yet;
    // clr_b (replayed launches only), the chunk's last own tile, whose rows
    // past the chunk may be stale (the k/v maps span the buffers' capacity):
    // their weights are 0, but 0 x NaN is not.
    const int clr_a = (cs % kTileN) != 0 ? nA - a.kt0 : -1;
    const int clr_b = (kReplay && (pf.p_t % kTileN) != 0) ? nA + (pf.p_t - 1) / kTileN - a.kt0 + 1 : -1;
    bool ok = mbar_wait(smem_u32(&misc->bar_q), a.item_no & 1, abort, tmo);
    tc_fence_after();
    const uint64_t qd0 = smem_desc(sbase + kSmemQ, 16, 1024, kSwz128);
    const uint64_t qd1 = smem_desc(sbase + kSmemQ + kTileBytes, 16, 1024, kSwz128);
    for (int j = 0; ok && j <= nT; ++j) {
        const uint32_t c = a.tile0 + j;
        uint64_t vdesc = 0;
        const uint32_t vs_cur = vs;
        if (j > 0) {
            if (!mbar_wait(smem_u32(&misc->bar_vfull[vs_cur]), vph, abort, tmo)) {
                ok = false;
                break;
            }
            const uint32_t dv = sV + vs_cur * kTileBytes;
            if (j == clr_a)
                clear_uncached_rows(dv, cs - (a.kt0 + j - 1) * kTileN);
            if (kReplay && j == clr_b)
                zero_v_rows(dv, pf.p_t % kTileN, kTileN);
            vdesc = smem_desc(dv, kHalfTile, 1024, kSwz128);
            asm volatile("" : "+l"(vdesc));
        }
        uint64_t kdesc = 0;
        bool kready = false;
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            if (e >= a.nh)
                break;
            if (j > 0) {
                // O_e += P_e(j-1) V_{j-1}, as soon as head e's softmax wrote P
                if (!mbar_wait(smem_u32(&misc->bar_pfull[e]), ((e == 0 ? a.sph0 : a.sph1) + j - 1) & 1, abort,
                               tmo)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t pa = tmem + kTmemS + e * 128;   // P_e: 8 columns per 16 keys
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)   // 16 keys of MN-major V: +2 KiB
                    tc_mma_ts(tmem + kTmemO + e * 128, pa + kk * 8, vdesc + (uint64_t)((kk * 2048) >> 4),
                              kIdescO, (j > 1 || kk > 0) ? 1u : 0u);
            }
            if (j < nT) {
                if (!kready) {
                    if (!mbar_wait(smem_u32(&misc->bar_kfull[c % kKStages]), (c / kKStages) & 1, abort, tmo)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    kdesc = smem_desc(sK + (c % kKStages) * kTileBytes, 16, 1024, kSwz128);
                    asm volatile("" : "+l"(kdesc));
                    kready = true;
                }
                // S_e(j) = Q_e K_j^T.  Opaque per tile, so that the compiler
                // does not keep the 8 offset descriptors of both heads live
                // across the loop.
                uint64_t qd = e == 0 ? qd0 : qd1;
                asm volatile("" : "+l"(qd));
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    // 16 dims of K-major SW128: +32 B inside a 64-column half
                    const uint64_t off = (uint64_t)(((kk >> 2) * kHalfTile + (kk & 3) * 32) >> 4);
                    tc_mma_ss(tmem + kTmemS + e * 128, qd + off, kdesc + off, kIdescS, kk > 0 ? 1u : 0u);
                }
                tc_commit(smem_u32(&misc->bar_sfull[e]));
            }
        }
        if (!ok)
            break;
        if (j < nT)
            tc_commit(smem_u32(&misc->bar_kempty[c % kKStages]));
        if (j > 0) {
            tc_commit(smem_u32(&misc->bar_vempty[vs_cur]));
            vs = vs + 1 == vst ? 0u : vs + 1;
            vph ^= vs == 0 ? 1u : 0u;
        }
    }
    if (ok)
        tc_commit(smem_u32(&misc->bar_odone));
    else
        set_abort(P, misc);
}

// Piece 0 of each of the n_rep / nh items of a KV head appends its share of
// the tile's tokens (item r of the group takes tokens [r*128/(n_rep/nh),
// (r+1)*128/(n_rep/nh))); the 32 16-byte pieces of a token's K and V rows are
// spread over the 256 consumer threads, all loads in flight at once, while Q
// and the first K tile land.
__device__ __forceinline__ void prefill_append(const LayerParams &P, const PrefillInfo &pf, const PrefillArgs &a,
                                               int tid)
{
    const int groups = P.n_rep / a.nh;              // items per KV head and tile
    const int per = kTileM / groups;                // tokens of this item
    const int kvh = a.hq0 / P.n_rep;
    const int r0 = kTileM * a.t + ((a.hq0 % P.n_rep) / a.nh) * per;   // first chunk row
    const int n_pc = per * 32;                      // 16-byte pieces
    constexpr int kRound = 8;                       // loads in flight per thread
#pragma unroll 1
    for (int b = 0; b < n_pc; b += kRound * kConsThreads) {
        uint4 av[kRound];
        int slot[kRound];
#pragma unroll
        for (int x = 0; x < kRound; ++x) {
            const int pc = b + tid + kConsThreads * x;
            const int u = pc >> 5, w = pc & 31;
            slot[x] = -1;
            if (pc < n_pc && r0 + u < pf.p_t) {
                const size_t src = ((size_t)(pf.token_base + r0 + u) * P.hkv + kvh) * kHeadDim;
                slot[x] = __ldg(P.slots + pf.token_base + r0 + u);
                av[x] = __ldg(reinterpret_cast<const uint4 *>((w < 16 ? P.k : P.v) + src) + (w & 15));
            }
        }
#pragma unroll
        for (int x = 0; x < kRound; ++x) {
            const int w = (b + tid + kConsThreads * x) & 31;
            const int sl = slot[x];
            if (sl >= P.num_pages * kPage) {
                if (w == 0)
                    flag_error(P, ERR_SLOT);
            } else if (sl >= 0) {
                const size_t dst = (((size_t)(sl / kPage) * P.hkv + kvh) * kPage + sl % kPage) * kHeadDim;
                reinterpret_cast<uint4 *>((w < 16 ? P.k_pool : P.v_pool) + dst)[w & 15] = av[x];
            }
        }
    }
}

// Consumer warpgroup e (its 128 threads, TMEM lane = row): the softmax of
// query head hq0 + e over the item's key tiles, then its epilogue.
__device__ void prefill_softmax(const LayerParams &P, uint8_t *smem, Misc *misc, const PrefillArgs &a,
                                uint32_t tmem, int e, int r)
{
    const PrefillInfo &pf = misc->pre[a.f];
    const int cs = pf.chunk_start, p = pf.p_t, tb = pf.token_base;
    const int nA = (cs + kTileN - 1) / kTileN;
    const int nT = a.kt1 - a.kt0;
    const int hq = a.hq0 + e;
    const int j = kTileM * a.t + r;          // chunk row offset
    const int q4 = r >> 5;
    const uint32_t tl = tmem + ((uint32_t)(q4 * 32) << 16);
    const uint32_t tS = tl + kTmemS + e * 128, tO = tl + kTmemO + e * 128;
    const uint32_t sbase = smem_u32(smem);
    const float sl = P.scale_log2;
    const uint32_t ph0 = e == 0 ? a.sph0 : a.sph1;
    volatile int *abort = &misc->abort;
    const uint64_t tmo = P.timeout_ns;

    // the item holds a prompt's first positions, where a row has few keys
    const bool few_keys = a.t == 0 && cs < kShortKeys;
    float m_run = neg_inf(), l_run = 0.f;
    bool ok = true;
    for (int i = 0; i < nT; ++i) {
        // the warp agrees on the outcome: the TMEM accesses below are
        // warp-collective, so no lane may leave the loop alone
        const bool got = mbar_wait(smem_u32(&misc->bar_sfull[e]), (ph0 + i) & 1, abort, tmo);
        if (!__all_sync(0xffffffffu, got)) {
            ok = false;
            break;
        }
        tc_fence_after();
        const int gi = a.kt0 + i;
        const int nvalid = gi < nA ? min(kTileN, cs - gi * kTileN) : min(kTileN, j - kTileN * (gi - nA) + 1);
        // Row r of S: all 128 raw scores read from TMEM once (a second read
        // would compete with the tensor core's own TMEM traffic).
        uint32_t sv[128];
#pragma unroll
        for (int q = 0; q < 4; ++q)
            tmem_ld32(tS + 32 * q, *reinterpret_cast<uint32_t(*)[32]>(&sv[32 * q]));
        tmem_wait_ld();
        if (nvalid < kTileN) {  // boundary tiles only: masked keys -> -inf
#pragma unroll
            for (int cc = 0; cc < 128; ++cc)
                if (cc >= nvalid)
                    sv[cc] = 0xFF800000u;
        }
        // FA4-style lazy rescale: the running max m (log2 domain) moves only
        // when a row's max exceeds it by more than 8, so every weight of P is
        // at most 2^8.  From the second tile on P is first computed with m as
        // it stands, without the row max: a tile sum of at most 2^8 shows
        // that no weight exceeds 2^8, which is all the lazy rule would have
        // checked (m stays), so the result is the same.  Otherwise the warp
        // takes the full path: row max, new m where it grew by more than 8, P
        // computed again (the same bits in the rows whose m stays).  P goes
        // over the first 64 columns of S (the A operand of P.V).
        auto exp_store = [&](float m) {
            return few_keys ? row_exp_store<true>(sv, sl, -m, tS) : row_exp_store<false>(sv, sl, -m, tS);
        };
        float m_use = m_run, rs = 0.f;
        bool rescale = false, resc = false;
        if (i > 0)
            rs = exp_store(m_run);
        if (i == 0 || __any_sync(0xffffffffu, !(rs <= 256.0f))) {
            const float m_new = fmaxf(m_run, row_max(sv) * sl);
            rescale = m_new > m_run + 8.0f;
            m_use = rescale ? m_new : m_run;
            rs = exp_store(m_use);
            resc = i > 0 && __any_sync(0xffffffffu, rescale);
        }
        // O_e is stable here: sfull of this tile was committed after O_e +=
        // P_e V of the previous tile, and the next P.V waits for this tile's
        // P.  tcgen05.ld/st are warp-collective, so the whole warp rescales
        // when any of its rows must (alpha = 1 for the others): a branch
        // taken by some lanes only would run them in a diverged warp.
        if (resc) {
            const float alpha = rescale ? ex2(m_run - m_use) : 1.0f;
#pragma unroll
            for (int gq = 0; gq < 4; ++gq) {
                uint32_t o[32];
                tmem_ld32(tO + 32 * gq, o);
                tmem_wait_ld();
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
                tmem_st32(tO + 32 * gq, o);
            }
            l_run *= alpha;
        }
        l_run += rs;
        m_run = m_use;
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(smem_u32(&misc->bar_pfull[e]));
    }
    if (ok && !mbar_wait(smem_u32(&misc->bar_odone), a.item_no & 1, abort, tmo))
        ok = false;
    if (!__all_sync(0xffffffffu, ok)) {   // warp-uniform, as above
        set_abort(P, misc);
        return;
    }
    tc_fence_after();
    const float inv = 1.0f / l_run;
    if (a.ns > 1) {
        // One piece of a split tile: normalised partial O and its lse.  O
        // goes through shared memory (head 0 the K ring, head 1 the V ring:
        // odone means every MMA of the item, so every load into the rings,
        // has completed, and the next item's loads start only after the
        // item boundary), so that each global write is a whole 512-byte row
        // rather than one 16-byte piece of 32 rows.  A row's 16-byte chunk c
        // sits at chunk c ^ (row & 31): writes by rows and reads along a row
        // are both free of bank conflicts.
        const int part_slot = a.part_base + e * a.ns + a.s;
        const uint32_t stg = sbase + (e == 0 ? kSmemK : kSmemV);
#pragma unroll
        for (int gq = 0; gq < 4; ++gq) {
            uint32_t o[32];
            tmem_ld32(tO + 32 * gq, o);
            tmem_wait_ld();
#pragma unroll
            for (int x = 0; x < 8; ++x) {
                const uint32_t addr = stg + r * 512 + (((gq * 8 + x) ^ (r & 31)) << 4);
                asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                             "f"(__uint_as_float(o[4 * x]) * inv), "f"(__uint_as_float(o[4 * x + 1]) * inv),
                             "f"(__uint_as_float(o[4 * x + 2]) * inv), "f"(__uint_as_float(o[4 * x + 3]) * inv)
                             : "memory");
            }
        }
        float lg;
        asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(lg) : "f"(l_run));
        P.pre_lse[(size_t)part_slot * kTileM + r] = m_run + lg;
        if (e == 0)   // the head's 128 rows are staged (barrier ids fixed at compile time)
            named_sync(kBarHead0, kTileM);
        else
            named_sync(kBarHead0 + 1, kTileM);
        // warp q4 of the head writes rows [32 q4, 32 q4 + 32), four at a time
        const int lane = r & 31;
        float *pbase = P.pre_o + (size_t)part_slot * kTileM * kHeadDim;
#pragma unroll 1
        for (int rr = 0; rr < 32; rr += 4) {
            float4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int row = q4 * 32 + rr + u;
                const uint32_t addr = stg + row * 512 + ((lane ^ (row & 31)) << 4);
                asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                             : "=f"(v[u].x), "=f"(v[u].y), "=f"(v[u].z), "=f"(v[u].w)
                             : "r"(addr));
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                reinterpret_cast<float4 *>(pbase + (size_t)(q4 * 32 + rr + u) * kHeadDim)[lane] = v[u];
        }
        __threadfence();
        return;
    }
    uint16_t *orow = P.out + ((size_t)(tb + j) * P.hq + hq) * kHeadDim;
    if (!(a.t == 0 && cs < kShortRowKeys)) {
        // No short rows to recompute from the tiles, so the head's Q tile
        // (read by its last MMA, complete at odone) stages the bf16 rows and
        // the warps write whole 256-byte rows, two per instruction.  A row's
        // 16-byte chunk c sits at chunk c ^ (row & 15): conflict-free both
        // ways.
        const uint32_t stg = sbase + kSmemQ + e * kTileBytes;
#pragma unroll
        for (int gq = 0; gq < 4; ++gq) {
            uint32_t o[32];
            tmem_ld32(tO + 32 * gq, o);
            tmem_wait_ld();
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                const uint32_t addr = stg + r * 256 + (((gq * 4 + x) ^ (r & 15)) << 4);
                asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                             "r"(pack_bf16(__uint_as_float(o[8 * x + 0]) * inv, __uint_as_float(o[8 * x + 1]) * inv)),
                             "r"(pack_bf16(__uint_as_float(o[8 * x + 2]) * inv, __uint_as_float(o[8 * x + 3]) * inv)),
                             "r"(pack_bf16(__uint_as_float(o[8 * x + 4]) * inv, __uint_as_float(o[8 * x + 5]) * inv)),
                             "r"(pack_bf16(__uint_as_float(o[8 * x + 6]) * inv, __uint_as_float(o[8 * x + 7]) * inv))
                             : "memory");
            }
        }
        if (e == 0)
            named_sync(kBarHead0, kTileM);
        else
            named_sync(kBarHead0 + 1, kTileM);
        // warp q4 of the head writes rows [32 q4, 32 q4 + 32), two per
        // instruction (lanes 0-15 and 16-31), eight rows per round
        const int lane = r & 31, half = lane >> 4, c = lane & 15;
#pragma unroll 1
        for (int rr = 0; rr < 32; rr += 8) {
            uint4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int row = q4 * 32 + rr + 2 * u + half;
                const uint32_t addr = stg + row * 256 + ((c ^ (row & 15)) << 4);
                asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                             : "=r"(v[u].x), "=r"(v[u].y), "=r"(v[u].z), "=r"(v[u].w)
                             : "r"(addr));
            }
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int row = q4 * 32 + rr + 2 * u + half;
                const int jr = kTileM * a.t + row;
                if (jr < p)
                    reinterpret_cast<uint4 *>(P.out + ((size_t)(tb + jr) * P.hq + hq) * kHeadDim)[c] = v[u];
            }
        }
        return;
    }
#pragma unroll
    for (int gq = 0; gq < 4; ++gq) {
        uint32_t o[32];
        tmem_ld32(tO + 32 * gq, o);
        tmem_wait_ld();
        if (j < p) {
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                uint4 v4;
                v4.x = pack_bf16(__uint_as_float(o[8 * x + 0]) * inv, __uint_as_float(o[8 * x + 1]) * inv);
                v4.y = pack_bf16(__uint_as_float(o[8 * x + 2]) * inv, __uint_as_float(o[8 * x + 3]) * inv);
                v4.z = pack_bf16(__uint_as_float(o[8 * x + 4]) * inv, __uint_as_float(o[8 * x + 5]) * inv);
                v4.w = pack_bf16(__uint_as_float(o[8 * x + 6]) * inv, __uint_as_float(o[8 * x + 7]) * inv);
                reinterpret_cast<uint4 *>(orow + 32 * gq)[x] = v4;
            }
        }
    }
    // rows with at most kShortRowKeys keys (positions 0..15 of a prompt):
    // exact fp32 recomputation.  The item (t = 0, never split) has one key
    // tile (cs = 0) or two (0 < cs < 16: the cached tile, then the chunk's
    // own), all still in their K and V stages (at least two of each).
    static_assert(kShortRowKeys <= kTileN, "the short rows' keys lie in the first two tiles");
    if (a.t == 0 && cs < kShortRowKeys && cs + r < kShortRowKeys && j < p) {
        const uint32_t ca = a.tile0, cb = a.tile0 + (cs > 0 ? 1u : 0u);
        static_assert(kKStages >= 2, "the short rows need two tiles in the rings");   // and v_stages >= 2
        const uint32_t sK = sbase + kSmemK, sV = sbase + kSmemV;
        const uint32_t vst = (uint32_t)P.v_stages;
        // the tiles' TMA writes, observed on their own (completed) barriers
        if (!(mbar_wait(smem_u32(&misc->bar_q), a.item_no & 1, abort, tmo) &&
              mbar_wait(smem_u32(&misc->bar_kfull[ca % kKStages]), (ca / kKStages) & 1, abort, tmo) &&
              mbar_wait(smem_u32(&misc->bar_vfull[ca % vst]), (ca / vst) & 1, abort, tmo) &&
              mbar_wait(smem_u32(&misc->bar_kfull[cb % kKStages]), (cb / kKStages) & 1, abort, tmo) &&
              mbar_wait(smem_u32(&misc->bar_vfull[cb % vst]), (cb / vst) & 1, abort, tmo)))
            set_abort(P, misc);
        else
            short_row_exact(sbase + kSmemQ + e * kTileBytes, sK + (ca % kKStages) * kTileBytes,
                            sV + (ca % vst) * kTileBytes, sK + (cb % kKStages) * kTileBytes,
                            sV + (cb % vst) * kTileBytes, cs, r, sl, orow);
    }
}

// Merge the n_s pieces of prefill tile (t, hq0 .. hq0 + nh - 1) if this CTA's
// piece arrived last (no waiting): out = sum_s w_s O_s / sum_s w_s,
// w_s = 2^(lse_s - max).  Run by the 256 consumer threads.
__device__ void prefill_merge(const LayerParams &P, Misc *misc, const PrefillInfo &pf, const PrefillArgs &a,
                              int tid)
{
    // the tile's arrival counter, indexed over the query tiles of all chunks
    uint32_t *cnt = P.pre_cnt + (size_t)(pf.tile_base + a.t) * P.hq + a.hq0;
    cons_sync();   // every consumer thread's partial is written (and fenced)
    if (tid == 0) {
        const uint32_t prev = atomicAdd(cnt, 1u);
        misc->last = (prev == (uint32_t)(a.ns - 1)) ? 1 : 0;
    }
    cons_sync();
    if (!misc->last)
        return;
    __threadfence();
    // Consumer warp w merges rows [16 w, 16 w + 16) of the tile, four rows
    // at a time: a row's 128 columns are one float4 per lane, so every load
    // reads whole rows (coalesced), and the partials of four pieces of four
    // rows are in flight together; the max and the weight sum of a row are
    // kept online over the groups of pieces.
    const int warp = tid >> 5, lane = tid & 31;
    for (int e = 0; e < a.nh; ++e) {
        const int base = a.part_base + e * a.ns;
        for (int r4 = 0; r4 < kTileM / kWarps; r4 += 4) {
            const int r0 = warp * (kTileM / kWarps) + r4;
            float M[4], W[4];
            float4 acc[4];
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) {
                M[rr] = neg_inf();
                W[rr] = 0.f;
                acc[rr] = make_float4(0.f, 0.f, 0.f, 0.f);
            }
            for (int s0 = 0; s0 < a.ns; s0 += 4) {
                float l[4][4];
                float4 v[4][4];
#pragma unroll
                for (int rr = 0; rr < 4; ++rr) {
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const bool ok = s0 + u < a.ns;
                        const size_t row = (size_t)(base + s0 + u) * kTileM + r0 + rr;
                        l[rr][u] = ok ? __ldcg(P.pre_lse + row) : neg_inf();
                        v[rr][u] = ok ? __ldcg(reinterpret_cast<const float4 *>(P.pre_o + row * kHeadDim) + lane)
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
                    }
                }
#pragma unroll
                for (int rr = 0; rr < 4; ++rr) {
                    const float mb = fmaxf(fmaxf(M[rr], fmaxf(l[rr][0], l[rr][1])), fmaxf(l[rr][2], l[rr][3]));
                    const float c = ex2(M[rr] - mb);   // 0 for the first group (M = -inf)
                    W[rr] *= c;
                    acc[rr].x *= c;
                    acc[rr].y *= c;
                    acc[rr].z *= c;
                    acc[rr].w *= c;
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const float f = ex2(l[rr][u] - mb);   // 0 past the last piece
                        W[rr] += f;
                        acc[rr].x += f * v[rr][u].x;
                        acc[rr].y += f * v[rr][u].y;
                        acc[rr].z += f * v[rr][u].z;
                        acc[rr].w += f * v[rr][u].w;
                    }
                    M[rr] = mb;
                }
            }
#pragma unroll
            for (int rr = 0; rr < 4; ++rr) {
                const int j = kTileM * a.t + r0 + rr;
                if (j < pf.p_t) {
                    const float inv = 1.0f / W[rr];
                    uint2 pk;
                    pk.x = pack_bf16(acc[rr].x * inv, acc[rr].y * inv);
                    pk.y = pack_bf16(acc[rr].z * inv, acc[rr].w * inv);
                    reinterpret_cast<uint2 *>(P.out + ((size_t)(pf.token_base + j) * P.hq + a.hq0 + e) *
                                                          kHeadDim)[lane] = pk;
                }
            }
        }
    }
    if (tid == 0)
        *cnt = 0u;
}

// The next work item of this CTA (thread 0 only).  The items form two
// queues: the prefill items [0, n_pre), heaviest first, and the decode items
// [n_pre, n), longest first.  CTAs below dec_ctas draw from the decode queue
// first and the others from the prefill queue, and each turns to the other
// queue once its own is empty: HBM-bound decode splits then stream on some
// SMs while tensor-bound prefill tiles run on the rest.  n when both are empty.
__device__ __forceinline__ int32_t claim_item(const LayerParams &P, Misc *misc)
{
    while (misc->queue < 2) {
        const int32_t dec = misc->dec_first ^ misc->queue;
        const int32_t i = (dec ? misc->n_pre : 0) + (int32_t)atomicAdd(P.work_cnt + 2 * dec, 1u);
        if (i < (dec ? misc->n_items : misc->n_pre))
            return i;
        misc->queue += 1;
    }
    return misc->n_items;
}

// Between items: every thread of the CTA has finished the previous item.
__device__ __forceinline__ void item_boundary()
{
    tc_fence_before();
    named_sync(kBarItem, kThreads);
    tc_fence_after();
}

// Warpgroup 0's item loop: claims the next item, loads tiles, issues MMAs.
template <bool kReplay>
__device__ void producer_loop(const LayerParams &P, uint8_t *smem, Misc *misc, uint32_t tmem)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t sbase = smem_u32(smem);
    uint32_t tile_cnt = 0, item_no = 0, sph[2] = {0u, 0u};
    int buf = 0;
    for (;;) {
        item_boundary();
        const int idx = misc->item_idx[buf];
        if (idx >= (kReplay ? misc->n_items : P.n_items) || misc->abort)
            break;
        if (tid == 0)
            misc->item_idx[buf ^ 1] = claim_item(P, misc);
        const int4 it = P.items[idx];
        if ((it.x & 0xF) == ITEM_PREFILL) {
            const PrefillArgs a = prefill_args(it, misc, tile_cnt, item_no, sph);
            if (warp == 0) {
                if (lane == 0) {
                    // Q of the item's heads (the previous item's MMAs and
                    // short rows are done: every thread passed the boundary)
                    fence_proxy_async_smem();
                    const uint32_t bq = smem_u32(&misc->bar_q);
                    const PrefillInfo &pf = misc->pre[a.f];
                    mbar_expect_tx(bq, a.nh * kTileBytes);
                    for (int e = 0; e < a.nh; ++e) {
                        const uint32_t dq = sbase + kSmemQ + e * kTileBytes;
                        tma_load_3d(dq, &P.tm_q, bq, 0, a.hq0 + e, pf.token_base + kTileM * a.t);
                        tma_load_3d(dq + kHalfTile, &P.tm_q, bq, 64, a.hq0 + e, pf.token_base + kTileM * a.t);
                    }
                }
                prefill_load_ring(P, misc, a, true, sbase + kSmemK, lane);
            } else if (warp == 2) {
                prefill_load_ring(P, misc, a, false, sbase + kSmemV, lane);
            } else if (warp == 1 && lane == 0) {
                prefill_mma<kReplay>(P, misc, a, tmem, sbase);
            }
            const uint32_t nT = (uint32_t)(a.kt1 - a.kt0);
            tile_cnt += nT;
            item_no += 1;
            sph[0] += nT;
            if (a.nh == 2)
                sph[1] += nT;
        }
        __syncwarp();
        buf ^= 1;
    }
}

// The consumer warpgroups' item loop: softmax and epilogue of prefill items,
// all of a decode item.
template <bool kReplay>
__device__ void consumer_loop(const LayerParams &P, uint8_t *smem, Misc *misc, uint32_t tmem)
{
    const int tid = threadIdx.x - kProdThreads;     // 0..255
    uint32_t tile_cnt = 0, item_no = 0, sph[2] = {0u, 0u};
    int buf = 0;
    for (;;) {
        item_boundary();
        const int idx = misc->item_idx[buf];
        if (idx >= (kReplay ? misc->n_items : P.n_items) || misc->abort)
            break;
        const int4 it = P.items[idx];
        if ((it.x & 0xF) == ITEM_PREFILL) {
            const PrefillArgs a = prefill_args(it, misc, tile_cnt, item_no, sph);
            const PrefillInfo &pf = misc->pre[a.f];
            if (a.kt0 == 0)
                prefill_append(P, pf, a, tid);
            const int e = tid >> 7;
            if (e < a.nh)
                prefill_softmax(P, smem, misc, a, tmem, e, tid & 127);
            // every consumer thread takes part in the merge's barriers, also
            // after an abort (the merge then writes what it finds; the call
            // reports the error and the host clears the counters)
            if (a.ns > 1)
                prefill_merge(P, misc, pf, a, tid);
            const uint32_t nT = (uint32_t)(a.kt1 - a.kt0);
            tile_cnt += nT;
            item_no += 1;
            sph[0] += nT;
            if (a.nh == 2)
                sph[1] += nT;
        } else if ((it.x & 0xF) == ITEM_DECODE_SHORT) {
            decode_short_item(P, smem, it.y, (int)(((uint32_t)it.x >> 4) & 0x7Fu), it.z, it.w, tid);
        } else {
            const uint32_t dx = (uint32_t)it.x;
            decode_item(P, smem, misc, it.y, (int)((dx >> 4) & 0x7Fu), (int)((dx >> 11) & 0xFFFu), it.z, it.w,
                        (int)(dx >> 23) * 16, tid);
        }
        fence_proxy_async_smem();  // generic smem accesses before later TMA writes
        buf ^= 1;
    }
}

// ---------------------------------------------------------------------------
// kReplay: a launch replayed from a graph (P.hdr holds the plan's counts);
// compiled apart so that the ordinary launch carries none of its code.
template <bool kReplay>
__global__ void __launch_bounds__(kThreads, 1) mixed_layer_kernel(const __grid_constant__ LayerParams P)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    Misc *misc = reinterpret_cast<Misc *>(smem + smem_data_bytes(P.v_stages));
    const int tid = threadIdx.x, warp = tid >> 5;

    // The launch's counts: from its parameters, or (a replayed launch) from
    // the plan header that the upload kernel wrote before the first layer.
    const PlanHeader *hdr = kReplay ? P.hdr : nullptr;
    const int has_prefill = hdr ? hdr->has_prefill : P.has_prefill;
    const int n_prefills = hdr ? hdr->n_prefills : P.n_prefills;
    if (tid == 0) {
        misc->n_items = hdr ? hdr->n_items : P.n_items;
        misc->n_pre = hdr ? hdr->n_pre_items : P.n_pre_items;
        misc->dec_first = (int32_t)blockIdx.x < (hdr ? hdr->dec_ctas : P.dec_ctas) ? 1 : 0;
        misc->queue = 0;
        misc->has_prefill = has_prefill;   // read again at the end (not kept in a register)
        mbar_init(smem_u32(&misc->bar_q), 1);
        for (int b = 0; b < kKStages; ++b) {
            mbar_init(smem_u32(&misc->bar_kfull[b]), 1);
            mbar_init(smem_u32(&misc->bar_kempty[b]), 1);
        }
        for (int b = 0; b < P.v_stages; ++b) {
            mbar_init(smem_u32(&misc->bar_vfull[b]), 1);
            mbar_init(smem_u32(&misc->bar_vempty[b]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&misc->bar_sfull[b]), 1);
            mbar_init(smem_u32(&misc->bar_pfull[b]), 128);
        }
        mbar_init(smem_u32(&misc->bar_odone), 1);
        mbar_init(smem_u32(&misc->bar_never), 1);
        misc->abort = 0;
        fence_mbar_init();
        if (has_prefill) {
            tma_prefetch_desc(&P.tm_q);
            tma_prefetch_desc(&P.tm_k);
            tma_prefetch_desc(&P.tm_v);
            tma_prefetch_desc(&P.tm_kpool);
            tma_prefetch_desc(&P.tm_vpool);
        }
    }
    if (has_prefill && warp == 1) {
        tmem_alloc(smem_u32(&misc->tmem_base), kTmemCols);
        tmem_relinquish();
    }
    if (tid >= 64 && tid < 64 + n_prefills)
        misc->pre[tid - 64] = P.pre[tid - 64];
    // Dependent order (early_start = 0): the previous launch in the stream
    // (the previous layer) must have completed, and its writes be visible,
    // before anything it may have written is read: this layer's q/k/v may be
    // computed from the previous layer's output.  Its CTAs signalled this
    // launch only when they ran out of work, so the wait is short.  Without
    // the programmatic launch attribute this is a no-op.
    if (!P.early_start)
        pdl_wait();
    // Consecutive launches use the workspace sets in turn, and the launch
    // that last used this one's set has completed before this one was
    // launched (see the end of the kernel), so work starts at once.
    if (tid == 0) {
        misc->item_idx[0] = claim_item(P, misc);
        // Fault injection for the bounded waits: the chosen block waits on a
        // barrier that nothing arrives at, with its first item claimed, so
        // the launch ends with that item undone and its counters left set.
        if ((int)blockIdx.x == P.stall_block &&
            !mbar_wait(smem_u32(&misc->bar_never), 0, &misc->abort, P.timeout_ns))
            set_abort(P, misc);
    }
    // Independent layers (early_start): the next launch may start once every
    // CTA of this one is resident; its CTAs take the SMs this grid frees, so
    // the next layer's work fills this layer's tail.  Consecutive launches
    // use different workspace sets (three in turn) and touch disjoint
    // tensors.
    if (P.early_start)
        pdl_launch_dependents();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = has_prefill ? misc->tmem_base : 0u;

    if (warp < kProdThreads / 32) {
        regs_dec<kProdRegs>();
        producer_loop<kReplay>(P, smem, misc, tmem);
    } else {
        regs_inc<kConsRegs>();
        consumer_loop<kReplay>(P, smem, misc, tmem);
    }
    // Every role left its loop at the same item boundary.

    // Out of work: wait until the previous launch has completed before
    // exiting (independent layers: so that when a later launch reuses that
    // launch's workspace set, it is complete; dependent layers waited at the
    // start already).  Dependent layers signal the next launch only now, so
    // it runs after this one, its launch latency hidden.
    pdl_wait();
    if (!P.early_start)
        pdl_launch_dependents();
    if (misc->abort) {
        // give in-flight copies and MMAs time to land before TMEM is freed
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 200000ull)
            __nanosleep(1000);
    }
    tc_fence_before();
    named_sync(kBarItem, kThreads);
    tc_fence_after();
    if (misc->has_prefill && warp == 1)
        tmem_dealloc(tmem, kTmemCols);
    if (tid == 0) {
        __threadfence();
        const uint32_t prev = atomicAdd(P.work_cnt + 1, 1u);
        if (prev == gridDim.x - 1) {
            P.work_cnt[0] = 0u;
            P.work_cnt[1] = 0u;
            P.work_cnt[2] = 0u;
            __threadfence();
        }
    }
}

// Standalone KV append: one warp per (token, KV head), 16-byte vectors.
__global__ void kv_append_kernel(const int32_t *__restrict__ slots, int n_tokens, int hkv,
                                 int num_pages, const uint16_t *__restrict__ k,
                                 const uint16_t *__restrict__ v, uint16_t *k_pool,
                                 uint16_t *v_pool, uint32_t *err)
{
    const int gw = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (gw >= n_tokens * hkv)
        return;
    const int tok = gw / hkv, h = gw % hkv;
    const int slot = __ldg(slots + tok);
    if (slot < 0)
        return;
    if (slot >= num_pages * kPage) {
        if (lane == 0)
            atomicOr(err, ERR_SLOT);
        return;
    }
    const size_t dst = (((size_t)(slot / kPage) * hkv + h) * kPage + slot % kPage) * kHeadDim;
    const size_t src = ((size_t)tok * hkv + h) * kHeadDim;
    const int c = lane & 15;
    if (lane < 16)
        reinterpret_cast<uint4 *>(k_pool + dst)[c] = __ldg(reinterpret_cast<const uint4 *>(k + src) + c);
    else
        reinterpret_cast<uint4 *>(v_pool + dst)[c] = __ldg(reinterpret_cast<const uint4 *>(v + src) + c);
}

// ---------------------------------------------------------------------------
// Host-side launchers (called from mx_api.cpp)
cudaError_t init_layer_kernel()
{
    cudaError_t e = cudaFuncSetAttribute(mixed_layer_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemTotalMax);
    if (e != cudaSuccess)
        return e;
    return cudaFuncSetAttribute(mixed_layer_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                kSmemTotalMax);
}

cudaError_t launch_mixed_layer(const LayerParams &P, int grid, cudaStream_t stream, bool pdl)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem_total_bytes(P.v_stages);   // only what the launch uses: the rest is L1
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 1 : 0;
    return P.hdr ? cudaLaunchKernelEx(&cfg, mixed_layer_kernel<true>, P)
                 : cudaLaunchKernelEx(&cfg, mixed_layer_kernel<false>, P);
}

// Plan upload: the work list and decode table, read by the GPU from mapped
// pinned host memory (16-byte words).
__global__ void plan_upload_kernel(const uint4 *__restrict__ src, uint4 *__restrict__ dst, int n)
{
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        dst[i] = src[i];
}

// The same for a replayed iteration: the plan's size is read from its
// header (at most max_words words).
__global__ void plan_upload_sized_kernel(const uint4 *__restrict__ src, uint4 *__restrict__ dst, int max_words)
{
    const int n = min(reinterpret_cast<const PlanHeader *>(src)->words, max_words);
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
        dst[i] = src[i];
}

cudaError_t launch_plan_upload_sized(const void *src, void *dst, size_t max_bytes, cudaStream_t stream)
{
    plan_upload_sized_kernel<<<8, 256, 0, stream>>>(static_cast<const uint4 *>(src), static_cast<uint4 *>(dst),
                                                    (int)(max_bytes / sizeof(uint4)));
    return cudaGetLastError();
}

cudaError_t launch_plan_upload(const void *src, void *dst, size_t bytes, cudaStream_t stream)
{
    const int n = (int)(bytes / sizeof(uint4));
    if (n == 0)
        return cudaSuccess;
    const int blocks = n < 8 * 256 ? (n + 255) / 256 : 8;
    plan_upload_kernel<<<blocks, 256, 0, stream>>>(static_cast<const uint4 *>(src), static_cast<uint4 *>(dst), n);
    return cudaGetLastError();
}

cudaError_t launch_kv_append(const int32_t *slots, int n_tokens, int hkv, int num_pages,
                             const uint16_t *k, const uint16_t *v, uint16_t *k_pool,
                             uint16_t *v_pool, uint32_t *err, cudaStream_t stream)
{
    const long long warps = (long long)n_tokens * hkv;
    const int block = 256;
    const long long grid = (warps * 32 + block - 1) / block;
    if (grid == 0)
        return cudaSuccess;
    kv_append_kernel<<<(unsigned)grid, block, 0, stream>>>(slots, n_tokens, hkv, num_pages, k, v,
                                                          k_pool, v_pool, err);
    return cudaGetLastError();
}

}  // namespace mx
