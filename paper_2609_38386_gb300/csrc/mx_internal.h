// Shared host/device definitions of the mixed-iteration kernels.
#pragma once

#include <cuda.h>
#include <vector_types.h>

#include <cstdint>

namespace mx {

constexpr int kHeadDim = 128;
constexpr int kPage = 16;
// 12 warps per CTA: warpgroup 0 (warps 0-3) loads tiles and issues the
// tensor-core MMAs of prefill items; warpgroups 1 and 2 (the 256 "consumer"
// threads) run the softmax of one query head each in prefill items and all
// of a decode item.
constexpr int kThreads = 384;
constexpr int kProdThreads = 128;
constexpr int kConsThreads = kThreads - kProdThreads;   // 256
constexpr int kWarps = kConsThreads / 32;               // warps of a decode item (8)
constexpr int kMaxRep = 8;               // Hq / Hkv supported up to 8
// Registers per thread after the split (setmaxnreg): the launch gives 168
// to each of the 384 threads (64512); warpgroup 0 keeps 56, the consumers
// take 224: 128 x 56 + 256 x 224 = 64512.
constexpr int kProdRegs = 56;
constexpr int kConsRegs = 224;
static_assert(kProdThreads * kProdRegs + kConsThreads * kConsRegs <= kThreads * 168, "register split");

// Prefill tile geometry: 128 query rows x 128 keys per tcgen05 tile.
constexpr int kTileM = 128;
constexpr int kTileN = 128;

// Shared-memory plan (bytes, offsets from a 1024-aligned base).
constexpr int kHalfTile = kTileM * 64 * 2;             // 128 rows x 64 bf16 = 16 KiB
constexpr int kTileBytes = 2 * kHalfTile;              // 32 KiB
// A prefill item serves one or two query heads of one KV head: a Q tile per
// head, and K / V rings shared by both.  K stage c % kKStages is released
// once both heads' S_c = Q K_c^T have completed, V stage c % v_stages once
// both heads' P_c V_c have.  A V tile can be requested only when the P.V two
// (or three) tiles back has completed, one tile period before (or two before)
// its own P.V, and under load a tile takes about as long as a period to land:
// launches with a large prefill share use three V stages (224 KiB of shared
// memory); the others use two, which leaves 32 KiB more to the L1 cache that
// the decode splits and short items depend on.
constexpr int kKStages = 2;
constexpr int kVStagesMax = 3;
constexpr int kSmemQ = 0;                              // Q of head 0, then head 1
constexpr int kSmemK = kSmemQ + 2 * kTileBytes;
constexpr int kSmemV = kSmemK + kKStages * kTileBytes;
constexpr int kSmemMiscBytes = 1024;
// Data (192 or 224 KiB), then the barrier block at its end.
__host__ __device__ constexpr int smem_data_bytes(int v_stages) { return kSmemV + v_stages * kTileBytes; }
__host__ __device__ constexpr int smem_total_bytes(int v_stages)
{
    return smem_data_bytes(v_stages) + kSmemMiscBytes + 1024;   // + alignment slack
}
constexpr int kSmemTotalMax = smem_total_bytes(kVStagesMax);
static_assert(kSmemTotalMax <= 227 * 1024, "shared memory per CTA");

// Decode splits per SM that the split length aims at (total keys / (this x
// SMs)).  Each split pays a fixed start-up and merge cost, so splits are as
// long as load balance allows: about 1.5 per SM for a decode-only launch.
// Beside prefill items, which hold SMs from the start, the decode splits
// must fill around them: the fewer the query tiles, the finer (3.5 per SM
// beside one tile, 3 beside 2, 2 beside 3, 1 from 4 on), and at least 3
// when an SM's share of the decode keys is under 8192 (a longer split would
// be most of that share, and the last ones the launch's tail: on the
// Qwen3-0.6B sweep, 1024-key splits beat one per SM by up to 9 %, while the
// 8B and 32B sweeps, with 10K and 37K keys per SM, were best unchanged).
// With independent layers the next layer fills the tail: 1 per SM.
inline double decode_splits_per_sm(int n_qt, bool independent_layers, long long total_keys, int num_sms)
{
    if (n_qt <= 0)
        return 1.5;
    if (independent_layers)
        return 1.0;
    const double beside[3] = {3.5, 3.0, 2.0};
    double k = n_qt <= 3 ? beside[n_qt - 1] : 1.0;
    if (total_keys < 8192LL * num_sms && k < 3.0)
        k = 3.0;
    return k;
}

// Launch rule for the V ring depth: three stages when the launch's prefill
// tensor work (flops) is at least 150 times its decode key/value bytes (at
// the measured peaks, about 0.65 of the decode streaming time).
__host__ __device__ inline int choose_v_stages(double prefill_flops, double decode_bytes)
{
    return prefill_flops > 0.0 && prefill_flops >= 150.0 * decode_bytes ? 3 : 2;
}

// Makespan, in key tiles, of the prefill items (tiles[0..n), in claim
// order, heaviest first) claimed by m SMs, each taking the next item when it
// is free (list scheduling; every item also pays kItemStartTiles of
// start-up).  heap: caller storage for m entries (no allocation).
constexpr int kItemStartTiles = 2;
inline long long prefill_makespan(const int *tiles, int n, int m, long long *heap)
{
    for (int i = 0; i < m; ++i)
        heap[i] = 0;   // a min-heap of the SMs' free times (all zero: valid)
    long long span = 0;
    for (int i = 0; i < n; ++i) {
        const long long t = heap[0] + tiles[i] + kItemStartTiles;
        span = t > span ? t : span;
        int j = 0;   // replace the root and sift down
        for (;;) {
            const int l = 2 * j + 1, r = l + 1;
            int c = j;
            long long v = t;
            if (l < m && heap[l] < v) { c = l; v = heap[l]; }
            if (r < m && heap[r] < v) { c = r; v = heap[r]; }
            if (c == j)
                break;
            heap[j] = heap[c];
            j = c;
        }
        heap[j] = t;
    }
    return span;
}

// Launch rule for the CTAs that start on the decode queue (the others start
// on the prefill queue).  Prefill items are long and few per SM, so SMs
// taken from them must not lengthen their schedule: D is the largest count
// up to kMaxDecodeFirst for which the prefill makespan on grid - D SMs stays
// within 3 % of that on grid SMs.  Only launches with more prefill items
// than SMs (a single round of prefill items leaves SMs to the decode from
// the start anyway) and with decode streaming at least a quarter of the
// launch's time (HBM and tensor rates measured for this kernel on the
// GB300: 6.8 TB/s, 1.2 PFLOP/s) take any: measured on Qwen3-32B and -8B
// attention, decode splits running beside the prefill tiles stream more
// than one SM's share of HBM, up to 4 % faster launches.  heap: kMaxGrid
// entries of caller storage.
constexpr int kMaxDecodeFirst = 24;
constexpr int kMaxGrid = 1024;
inline int decode_first_ctas(const int *tiles, int n_pre, double prefill_flops, double decode_bytes, int grid,
                             long long *heap)
{
    if (n_pre <= grid || decode_bytes <= 0.0 || grid > kMaxGrid || grid <= kMaxDecodeFirst)
        return 0;
    const double t_dec = decode_bytes / 6.8e12, t_pre = prefill_flops / 1.2e15;
    if (t_dec < 0.25 * (t_dec + t_pre))
        return 0;
    const double limit = 1.03 * (double)prefill_makespan(tiles, n_pre, grid, heap);
    int lo = 0, hi = kMaxDecodeFirst;
    while (lo < hi) {
        const int mid = (lo + hi + 1) / 2;
        if ((double)prefill_makespan(tiles, n_pre, grid - mid, heap) <= limit)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// Decode ring: each of the 8 decode warps owns kDecStages stages of one page
// (K 4 KiB + V 4 KiB).
constexpr int kPageBytes = kPage * kHeadDim * 2;       // 4 KiB
constexpr int kDecStageBytes = 2 * kPageBytes;         // 8 KiB
constexpr int kDecStages = 3;
static_assert(kWarps * kDecStages * kDecStageBytes <= smem_data_bytes(2), "decode ring too large");

// TMEM columns (fp32): S of head 0 [0,128), S of head 1 [128,256), O of
// head 0 [256,384), O of head 1 [384,512).  P_h (bf16 pairs, the A operand
// of P.V) overwrites the first 64 columns of S_h once they are read; the next
// S_h = Q K^T is issued after that P.V, so the tensor pipe's in-order
// execution keeps the two apart.
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemS = 0;
constexpr uint32_t kTmemO = 256;

enum : int32_t { ITEM_PREFILL = 0, ITEM_DECODE = 1, ITEM_DECODE_SHORT = 2 };

// Accuracy of rows with few keys.  With few keys one weight of P can
// dominate the row, and the tensor-core paths multiply V by P rounded to
// bf16: unless the row is normalised by the sum of the same rounded weights,
// that weight's rounding (2^-9 relative, and the lazy rescale lets it reach
// 2^8) times |v| up to ~4.5, plus the bf16 rounding of an output of
// magnitude 2-4, can exceed the 1e-2 tolerance.
//  - decodes of at most kShortKeys keys are computed exactly in fp32 on the
//    CUDA cores (ITEM_DECODE_SHORT);
//  - chunk rows of at most kShortRowKeys keys are recomputed exactly in fp32
//    from the tiles in shared memory;
//  - prefill items that hold positions below kShortKeys of a prompt sum the
//    row's weights as rounded to bf16, so that P.V / l is a normalised
//    average of V.
constexpr int kShortKeys = 64;
constexpr int kShortRowKeys = 16;

// Prefill chunks of one iteration (several prompts' chunks may share it).
constexpr int kMaxPrefills = 16;
struct PrefillInfo {
    int32_t seq;          // page-table row
    int32_t chunk_start;  // position of the chunk's row 0
    int32_t p_t;          // chunk rows
    int32_t token_base;   // token index of row 0 in q/k/v/out/slots
    int32_t tile_base;    // its first query tile, counted over all chunks
    int32_t pad[3];
};

// Work-item encodings (int4):
//   prefill: {ITEM_PREFILL | chunk f << 4 | (heads - 1) << 8, t | hq << 16,
//             s | n_s << 16, partial slot base}: piece s of n_s of query tile
//            t (rows [128t, 128t+128) of chunk f) of query heads hq .. hq +
//            heads - 1 (heads 1 or 2, one KV head); the tile's key tiles are
//            split evenly between its n_s pieces; head e of piece s writes
//            partial slot base + e * n_s + s.
//   short decode (at most kShortKeys keys, one split): the decode record
//            with kind ITEM_DECODE_SHORT;
//   decode:  {ITEM_DECODE | kv head << 4 | split index << 11 | split
//             length / 16 << 23, decode index, page-table row, cached tokens}:
//             split s of decode i covers keys [s * len, (s + 1) * len) of
//             [0, ctx]; the row, length and split size travel in the item so
//             that the page-id loads need no other lookup first
__host__ __device__ inline int4 prefill_item_code(int f, int t, int hq, int heads, int s, int n_s, int part_base)
{
    int4 r;
    r.x = ITEM_PREFILL | (f << 4) | ((heads - 1) << 8);
    r.y = t | (hq << 16);
    r.z = s | (n_s << 16);
    r.w = part_base;
    return r;
}
constexpr int kMaxDecodeKvHeads = 127;   // item field widths: head 7 bits,
constexpr int kMaxDecodeSplits = 4095;   // split index 12 bits, length/16 9 bits
__host__ __device__ inline int4 decode_item_code(int i, int h, int s, int seq, int ctx, int split_len)
{
    int4 r;
    r.x = (int32_t)((uint32_t)ITEM_DECODE | ((uint32_t)h << 4) | ((uint32_t)s << 11) |
                    ((uint32_t)(split_len / 16) << 23));
    r.y = i;
    r.z = seq;
    r.w = ctx;
    return r;
}

// Error bits (mirror MX_ERRBIT_* of the public header).
constexpr uint32_t ERR_PAGE = 1u, ERR_SLOT = 2u, ERR_TIMEOUT = 4u;

// Per-decode metadata uploaded with the work list.
struct DecodeInfo {
    int32_t seq;        // page-table row
    int32_t ctx;        // cached tokens before this iteration
    int32_t n_splits;   // splits of its key range [0, ctx]
    int32_t part_base;  // first partial slot of (this decode, head 0)
};

// Header of a plan uploaded for a replayed (captured) iteration: the
// per-iteration counts that the layer kernel then reads from device memory
// instead of its parameters, and the size of the plan that the upload copies.
struct PlanHeader {
    int32_t n_items, n_decodes, n_prefills, has_prefill;
    int32_t words;         // 16-byte words of the whole plan, this header included
    int32_t n_pre_items;   // items [0, n_pre_items) are prefill items
    int32_t dec_ctas;      // CTAs that start on the decode items
    int32_t pad;
};

struct LayerParams {
    CUtensorMap tm_q;      // 3-D {128, Hq, n_tokens}, box {64, 1, 128}
    CUtensorMap tm_k;      // 3-D {128, Hkv, n_tokens}, box {64, 1, 128}
    CUtensorMap tm_v;
    CUtensorMap tm_kpool;  // 2-D {128, num_pages*Hkv*16}, box {64, 16}
    CUtensorMap tm_vpool;

    const uint16_t *q, *k, *v;
    uint16_t *k_pool, *v_pool, *out;

    const int32_t *page_table;
    const int32_t *slots;
    const int4 *items;
    const DecodeInfo *dec;

    float *part_o;         // [slot][kMaxRep][128] normalised partial outputs
    float *part_lse;       // [slot][kMaxRep] log2-sum-exp of each partial
    uint32_t *merge_cnt;   // [max_decodes * Hkv] arrival counters (self-resetting)
    float *pre_o;          // [slot][128 rows][128] normalised prefill-piece outputs
    float *pre_lse;        // [slot][128 rows] log2-sum-exp of each piece
    uint32_t *pre_cnt;     // [q tiles * Hq] piece arrival counters (self-resetting)
    uint32_t *work_cnt;    // [0] next prefill item, [1] CTAs finished, [2] next decode
                           // item (self-resetting)
    uint32_t *err;         // error word

    int32_t n_items;
    int32_t n_pre_items;   // items [0, n_pre_items) are prefill items, the rest decode items
    int32_t dec_ctas;      // CTAs [0, dec_ctas) take decode items first, the others prefill items
    int32_t n_decodes;
    const PrefillInfo *pre; // [n_prefills] prefill chunks
    int32_t n_prefills;
    int32_t hq, hkv, n_rep;
    int32_t num_pages, max_pages;
    int32_t split_keys;    // keys per decode split (multiple of 128)
    int32_t has_prefill;   // allocate TMEM only when prefill tiles exist
    int32_t v_stages;      // V ring depth of prefill items (2 or 3); sets the shared memory size
    int32_t early_start;   // let the next launch start as soon as this one is resident
    float scale_log2;      // log2(e) / sqrt(head_dim)
    uint64_t timeout_ns;   // bound on every in-kernel wait
    int32_t stall_block;   // fault injection: this block's first wait never completes (-1 = none)
    // Replayed launches: the plan header (counts above are then ignored),
    // and the tensor maps span the buffers' capacity rather than the
    // iteration's tokens.  Null for ordinary launches.
    const PlanHeader *hdr;
};

}  // namespace mx
