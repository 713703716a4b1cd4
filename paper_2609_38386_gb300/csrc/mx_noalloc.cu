// mx_mixed_attention_noalloc: one mixed layer call for callers that cannot
// allocate device memory.
//
// Who needs it: code that runs where cudaMalloc is off limits — inside a host
// framework whose caching allocator owns all device memory and forbids direct
// cudaMalloc, in a plug-in loaded into a process that pre-reserves the GPU
// with a fixed budget, or in latency-critical paths where an allocation (an
// implicit device synchronisation and a possible OOM) is not acceptable.
// Such a caller cannot create an mx_ctx, because mx_create allocates the
// context's workspace.  This entry point needs no context: the scratch the
// kernel uses (work list, split partials, arrival counters, error word) lives
// in one fixed file-scope device array that the module loader places in
// device memory together with the code.
//
// Limits (the size of that array, 4.11 MiB): at most 256 decodes, 4096 work
// items, 1024 decode split partials, 16 KV heads.  Larger requests are
// rejected with MX_ECAPACITY before anything is enqueued.
//
// Sharing: every call, from any thread, uses the same array on a given GPU
// and leaves its contents behind; calls whose GPU work overlaps (two streams,
// or two host threads) race on it.  Serialise them.
#include "../../include/mixattn.h"
#include "mx_internal.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

namespace mx {
cudaError_t init_layer_kernel();
cudaError_t launch_mixed_layer(const LayerParams &P, int grid, cudaStream_t stream, bool pdl);
}  // namespace mx

using namespace mx;

namespace {

constexpr int kNaMaxDecodes = 256;
constexpr int kNaMaxItems = 4096;
constexpr int kNaPartSlots = 1024;
constexpr int kNaMaxKvHeads = 16;
constexpr int kNaMaxSplitKeys = kWarps * 32 * kPage;  // 4096

constexpr size_t kOffPartO = 0;
constexpr size_t kOffPartLse = kOffPartO + (size_t)kNaPartSlots * kMaxRep * kHeadDim * sizeof(float);
constexpr size_t kOffMerge = kOffPartLse + (size_t)kNaPartSlots * kMaxRep * sizeof(float);
constexpr size_t kMergeBytes = (size_t)kNaMaxDecodes * kNaMaxKvHeads * sizeof(uint32_t);
constexpr size_t kOffWork = kOffMerge + kMergeBytes;  // [0] next item, [1] CTAs done, [4] error word
constexpr size_t kWorkBytes = 256;
constexpr size_t kOffPlan = kOffWork + kWorkBytes;    // DecodeInfo[256], then int4 items[4096]
constexpr size_t kPlanBytes = (size_t)kNaMaxDecodes * sizeof(DecodeInfo) + (size_t)kNaMaxItems * sizeof(int4);
constexpr size_t kOffPre = kOffPlan + kPlanBytes;    // PrefillInfo of the one chunk
constexpr size_t kScratchBytes = kOffPre + 256;

}  // namespace

// The scratch.  In host code this name is only a host-side stand-in for the
// device symbol: its device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_mx_noalloc_scratch[kScratchBytes];

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

struct DeviceState {
    bool ready = false;
    uint8_t *scratch = nullptr;  // device address of g_mx_noalloc_scratch
    EncodeTiledFn encode = nullptr;
    int num_sms = 0;
};
constexpr int kMaxDevices = 64;
DeviceState g_dev[kMaxDevices];
std::mutex g_setup_mu;

int report(char *buf, int32_t len, int code, const char *fmt, ...)
{
    if (buf && len > 0) {
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, (size_t)len, fmt, ap);
        va_end(ap);
    }
    return code;
}

// Once per device, with that device current: resolve the scratch's device
// address, set the kernel's shared-memory limit, find the tensor-map encoder.
int setup_device(int dev, DeviceState **out, char *eb, int32_t el)
{
    if (dev < 0 || dev >= kMaxDevices)
        return report(eb, el, MX_EDEVICE, "device %d outside the supported range", dev);
    std::lock_guard<std::mutex> lock(g_setup_mu);
    DeviceState &s = g_dev[dev];
    if (!s.ready) {
        cudaDeviceProp prop;
        if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess || prop.major != 10)
            return report(eb, el, MX_EDEVICE, "device %d is not an sm_100-family GPU", dev);
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_mx_noalloc_scratch);
        if (e != cudaSuccess || !p)
            return report(eb, el, MX_ECUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(e));
        if ((e = init_layer_kernel()) != cudaSuccess)
            return report(eb, el, MX_ECUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(e));
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
            return report(eb, el, MX_ECUDA, "cuTensorMapEncodeTiled entry point not found");
        s.scratch = static_cast<uint8_t *>(p);
        s.encode = reinterpret_cast<EncodeTiledFn>(fn);
        s.num_sms = prop.multiProcessorCount;
        s.ready = true;
    }
    *out = &s;
    return MX_OK;
}

int encode(EncodeTiledFn fn, CUtensorMap *m, const void *base, int rank, const cuuint64_t *dims,
           const cuuint64_t *strides, const cuuint32_t *box)
{
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void *>(base), dims,
              strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS
               ? MX_OK
               : MX_ECUDA;
}

}  // namespace

extern "C" int mx_mixed_attention_noalloc(const mx_geom *g, const mx_iter_desc *d,
                                          const mx_layer_bufs *b, void *stream, char *err_buf,
                                          int32_t err_len)
{
    if (!g || !d || !b)
        return report(err_buf, err_len, MX_EINVAL, "null geometry, descriptor or buffers");
    if (g->head_dim != kHeadDim || g->page_size != kPage || g->num_kv_heads <= 0 ||
        g->num_q_heads <= 0 || g->num_q_heads % g->num_kv_heads != 0 ||
        g->num_q_heads / g->num_kv_heads > kMaxRep || g->num_pages <= 0 || g->num_seqs <= 0 ||
        g->max_pages_per_seq <= 0 || (int64_t)g->num_pages * g->num_kv_heads * kPage > INT32_MAX)
        return report(err_buf, err_len, MX_EINVAL, "unsupported geometry");
    const int rep = g->num_q_heads / g->num_kv_heads;
    if (rep & (rep - 1))
        return report(err_buf, err_len, MX_EINVAL, "Hq / Hkv must be 1, 2, 4 or 8");
    if (g->num_kv_heads > kNaMaxKvHeads)
        return report(err_buf, err_len, MX_ECAPACITY, "num_kv_heads %d > %d (scratch limit)",
                      g->num_kv_heads, kNaMaxKvHeads);
    const int nd = d->n_decodes, p = d->p_t;
    if (nd < 0 || p < 0 || d->chunk_start < 0)
        return report(err_buf, err_len, MX_EINVAL, "negative n_decodes, p_t or chunk_start");
    if (d->n_prefills != 0)
        return report(err_buf, err_len, MX_EINVAL,
                      "several prefill chunks (n_prefills > 0) need a context: use mx_mixed_attention");
    if (nd > kNaMaxDecodes)
        return report(err_buf, err_len, MX_ECAPACITY, "n_decodes %d > %d (scratch limit)", nd,
                      kNaMaxDecodes);
    const int64_t cap = (int64_t)g->max_pages_per_seq * kPage;
    if (nd > 0 && (!d->decode_seq_ids || !d->decode_ctx_lens))
        return report(err_buf, err_len, MX_EINVAL, "decode arrays are null");
    for (int i = 0; i < nd; ++i) {
        const int s = d->decode_seq_ids[i], n = d->decode_ctx_lens[i];
        if (s < 0 || s >= g->num_seqs)
            return report(err_buf, err_len, MX_EINVAL, "decode %d: seq id %d out of range", i, s);
        if (n < 0 || (int64_t)n + 1 > cap)
            return report(err_buf, err_len, MX_ECAPACITY, "decode %d: ctx %d exceeds the page table", i, n);
    }
    if (p > 0) {
        if (d->prefill_seq_id < 0 || d->prefill_seq_id >= g->num_seqs)
            return report(err_buf, err_len, MX_EINVAL, "prefill seq id out of range");
        if ((int64_t)d->chunk_start + p > cap)
            return report(err_buf, err_len, MX_ECAPACITY, "chunk exceeds the page table");
    }
    {
        // a sequence takes part once: as one decode or as the chunk (two
        // entries of one sequence would append to and read the same pages)
        int32_t ids[kNaMaxDecodes + 1];
        int n_ids = 0;
        for (int i = 0; i < nd; ++i)
            ids[n_ids++] = d->decode_seq_ids[i];
        if (p > 0)
            ids[n_ids++] = d->prefill_seq_id;
        std::sort(ids, ids + n_ids);
        for (int i = 1; i < n_ids; ++i)
            if (ids[i] == ids[i - 1])
                return report(err_buf, err_len, MX_EINVAL, "sequence %d appears twice in the iteration", ids[i]);
    }
    const int n_tok = nd + p;
    if (n_tok == 0)
        return MX_OK;
    if (!d->page_table || !d->slots)
        return report(err_buf, err_len, MX_EINVAL, "page_table / slots are null");
    const void *ptrs[] = {b->q, b->k, b->v, b->k_pool, b->v_pool, b->out};
    for (const void *q : ptrs)
        if (!q || (reinterpret_cast<uintptr_t>(q) & 15u))
            return report(err_buf, err_len, MX_EINVAL, "a tensor pointer is null or not 16-byte aligned");

    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return report(err_buf, err_len, MX_ECUDA, "cudaGetDevice failed");
    DeviceState *st = nullptr;
    int rc = setup_device(dev, &st, err_buf, err_len);
    if (rc)
        return rc;

    // Work list on the stack, built by the rule of the context planner:
    // prefill tiles (heaviest first), then decode splits (longest first),
    // each decode cut into equal page-aligned parts.  The split length is the
    // context planner's automatic choice, doubled while the splits exceed
    // this entry point's partial slots or work items.
    const int hkv = g->num_kv_heads, hq = g->num_q_heads;
    const int n_qt = (p + kTileM - 1) / kTileM;
    const int nh = rep >= 2 ? 2 : 1;        // query heads per prefill item
    const int n_pre = n_qt * (hq / nh);     // prefill items
    if (n_pre > kNaMaxItems)
        return report(err_buf, err_len, MX_ECAPACITY, "%d prefill items exceed %d work items", n_pre,
                      kNaMaxItems);
    int64_t total_keys = 0;
    for (int i = 0; i < nd; ++i)
        total_keys += (int64_t)d->decode_ctx_lens[i] + 1;
    total_keys *= hkv;
    int split;
    {
        const double per_sm = decode_splits_per_sm(n_qt, false, total_keys, st->num_sms);
        const int64_t target = std::max<int64_t>(1, (int64_t)(per_sm * st->num_sms));
        int64_t sk = (total_keys + target - 1) / target;
        sk = (sk + 127) / 128 * 128;
        split = (int)std::min<int64_t>(std::max<int64_t>(sk, 512), kNaMaxSplitKeys);
    }
    auto count = [&](int sk, int64_t *parts, int64_t *items) {
        *parts = 0;
        *items = 0;
        for (int i = 0; i < nd; ++i) {
            const int ns = (d->decode_ctx_lens[i] + 1 + sk - 1) / sk;
            *items += (int64_t)ns * hkv;
            if (ns > 1)
                *parts += (int64_t)ns * hkv;
        }
    };
    int64_t parts = 0, ditems = 0;
    for (;;) {
        count(split, &parts, &ditems);
        if ((parts <= kNaPartSlots && (int64_t)n_pre + ditems <= kNaMaxItems) ||
            split >= kNaMaxSplitKeys)
            break;
        split = std::min(split * 2, kNaMaxSplitKeys);
    }
    if (parts > kNaPartSlots || (int64_t)n_pre + ditems > kNaMaxItems)
        return report(err_buf, err_len, MX_ECAPACITY,
                      "decode splits need %lld partial slots / %lld items (limits %d / %d)",
                      (long long)parts, (long long)(n_pre + ditems), kNaPartSlots, kNaMaxItems);

    alignas(16) unsigned char plan[kPlanBytes];
    DecodeInfo *dec = reinterpret_cast<DecodeInfo *>(plan);
    int4 *items = reinterpret_cast<int4 *>(plan + (size_t)kNaMaxDecodes * sizeof(DecodeInfo));
    int n = 0;
    // key tiles of each prefill item (for the decode-first rule), then keys
    // of each decode item (for their longest-first order, stable)
    int32_t item_keys[kNaMaxItems];
    const int n_ahead = (d->chunk_start + kTileN - 1) / kTileN;
    for (int t = n_qt - 1; t >= 0; --t)
        for (int h = 0; h < hq; h += nh) {
            item_keys[n] = n_ahead + t + 1;
            items[n++] = prefill_item_code(0, t, h, nh, 0, 1, 0);
        }
    const int n_prefill = n;
    int part = 0;
    for (int i = 0; i < nd; ++i) {
        const int keys = d->decode_ctx_lens[i] + 1;
        const int ns = (keys + split - 1) / split;
        const int len = ((keys + ns - 1) / ns + kPage - 1) / kPage * kPage;   // <= split
        dec[i].seq = d->decode_seq_ids[i];
        dec[i].ctx = d->decode_ctx_lens[i];
        dec[i].n_splits = ns;
        dec[i].part_base = ns > 1 ? part : 0;
        if (ns > 1)
            part += ns * hkv;
        for (int h = 0; h < hkv; ++h)
            for (int sp = 0; sp < ns; ++sp) {
                int4 code = decode_item_code(i, h, sp, dec[i].seq, dec[i].ctx, len);
                if (keys <= kShortKeys)   // few keys: the exact short path
                    code.x = (int32_t)(((uint32_t)code.x & ~0xFu) | (uint32_t)ITEM_DECODE_SHORT);
                item_keys[n] = std::min(len, keys - sp * len);
                items[n++] = code;
            }
    }
    // stable longest-first order of the decode items (insertion sort on the
    // stack: no allocation)
    for (int x = n_prefill + 1; x < n; ++x) {
        const int4 code = items[x];
        const int32_t kx = item_keys[x];
        int y = x;
        for (; y > n_prefill && item_keys[y - 1] < kx; --y) {
            items[y] = items[y - 1];
            item_keys[y] = item_keys[y - 1];
        }
        items[y] = code;
        item_keys[y] = kx;
    }

    cudaStream_t s = static_cast<cudaStream_t>(stream);
    uint8_t *sc = st->scratch;

    LayerParams P;
    std::memset(&P, 0, sizeof P);
    P.q = static_cast<const uint16_t *>(b->q);
    P.k = static_cast<const uint16_t *>(b->k);
    P.v = static_cast<const uint16_t *>(b->v);
    P.k_pool = static_cast<uint16_t *>(b->k_pool);
    P.v_pool = static_cast<uint16_t *>(b->v_pool);
    P.out = static_cast<uint16_t *>(b->out);
    P.page_table = d->page_table;
    P.slots = d->slots;
    P.dec = reinterpret_cast<const DecodeInfo *>(sc + kOffPlan);
    P.items = reinterpret_cast<const int4 *>(sc + kOffPlan + (size_t)kNaMaxDecodes * sizeof(DecodeInfo));
    P.part_o = reinterpret_cast<float *>(sc + kOffPartO);
    P.part_lse = reinterpret_cast<float *>(sc + kOffPartLse);
    P.merge_cnt = reinterpret_cast<uint32_t *>(sc + kOffMerge);
    P.work_cnt = reinterpret_cast<uint32_t *>(sc + kOffWork);
    P.err = P.work_cnt + 4;
    P.n_items = n;
    P.n_decodes = nd;
    PrefillInfo pre{};
    pre.seq = d->prefill_seq_id;
    pre.chunk_start = d->chunk_start;
    pre.p_t = p;
    pre.token_base = nd;
    pre.tile_base = 0;
    P.pre = reinterpret_cast<const PrefillInfo *>(sc + kOffPre);
    P.n_prefills = p > 0 ? 1 : 0;
    P.hq = hq;
    P.hkv = hkv;
    P.n_rep = rep;
    P.num_pages = g->num_pages;
    P.max_pages = g->max_pages_per_seq;
    P.split_keys = split;
    P.has_prefill = n_prefill > 0 ? 1 : 0;
    const double pre_flops = 4.0 * hq * kHeadDim * ((double)p * pre.chunk_start + 0.5 * (double)p * (p + 1));
    const double dec_bytes = (double)total_keys * kHeadDim * 2 * 2;
    P.v_stages = choose_v_stages(pre_flops, dec_bytes);
    P.n_pre_items = n_prefill;
    long long heap[kMaxGrid];
    P.dec_ctas = n > n_prefill ? decode_first_ctas(item_keys, n_prefill, pre_flops, dec_bytes, st->num_sms, heap) : 0;
    P.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)kHeadDim));
    P.timeout_ns = 1000000000ull;
    P.stall_block = -1;
    if (P.has_prefill) {
        const cuuint64_t hd = kHeadDim;
        const cuuint64_t dq[3] = {hd, (cuuint64_t)hq, (cuuint64_t)n_tok};
        const cuuint64_t sq[2] = {hd * 2, hd * 2 * hq};
        const cuuint64_t dk[3] = {hd, (cuuint64_t)hkv, (cuuint64_t)n_tok};
        const cuuint64_t sk[2] = {hd * 2, hd * 2 * hkv};
        const cuuint32_t box3[3] = {64, 1, (cuuint32_t)kTileM};
        const cuuint64_t dp[2] = {hd, (cuuint64_t)g->num_pages * hkv * kPage};
        const cuuint64_t spl[1] = {hd * 2};
        const cuuint32_t box2[2] = {64, (cuuint32_t)kPage};
        if (encode(st->encode, &P.tm_q, b->q, 3, dq, sq, box3) ||
            encode(st->encode, &P.tm_k, b->k, 3, dk, sk, box3) ||
            encode(st->encode, &P.tm_v, b->v, 3, dk, sk, box3) ||
            encode(st->encode, &P.tm_kpool, b->k_pool, 2, dp, spl, box2) ||
            encode(st->encode, &P.tm_vpool, b->v_pool, 2, dp, spl, box2))
            return report(err_buf, err_len, MX_ECUDA, "cuTensorMapEncodeTiled failed");
    }

    // Counters and the error word must start at zero: the last call may have
    // left them set (an aborted launch does not reset them).
    cudaError_t e = cudaMemsetAsync(sc + kOffMerge, 0, kMergeBytes + kWorkBytes, s);
    if (e == cudaSuccess && nd > 0)
        e = cudaMemcpyAsync(sc + kOffPlan, dec, (size_t)nd * sizeof(DecodeInfo), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess && p > 0)
        e = cudaMemcpyAsync(sc + kOffPre, &pre, sizeof pre, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(const_cast<int4 *>(P.items), items, (size_t)n * sizeof(int4),
                            cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess)
        return report(err_buf, err_len, MX_ECUDA, "staging the work list: %s", cudaGetErrorString(e));
    e = launch_mixed_layer(P, std::max(1, std::min(st->num_sms, n)), s, false);
    if (e != cudaSuccess)
        return report(err_buf, err_len, MX_ECUDA, "launch: %s", cudaGetErrorString(e));
    if ((e = cudaStreamSynchronize(s)) != cudaSuccess)
        return report(err_buf, err_len, MX_ECUDA, "cudaStreamSynchronize: %s", cudaGetErrorString(e));
    uint32_t w = 0;
    if ((e = cudaMemcpy(&w, P.err, sizeof w, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return report(err_buf, err_len, MX_ECUDA, "reading the error word: %s", cudaGetErrorString(e));
    if (w & ERR_TIMEOUT)
        return report(err_buf, err_len, MX_ETIMEOUT, "a bounded in-kernel wait timed out");
    if (w & ERR_PAGE)
        return report(err_buf, err_len, MX_ERANGE_PAGE, "a page id outside the pool was read");
    if (w & ERR_SLOT)
        return report(err_buf, err_len, MX_ERANGE_SLOT, "a slot outside the pool was skipped");
    return MX_OK;
}
