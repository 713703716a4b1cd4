// C-ABI of the mixed-iteration library: context, host validation, the
// per-iteration planner (work list), TMA descriptors and launches.
#include "../../include/mixattn.h"
#include "mx_internal.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

namespace mx {
cudaError_t init_layer_kernel();
cudaError_t launch_mixed_layer(const LayerParams &P, int grid, cudaStream_t stream, bool pdl);
cudaError_t launch_plan_upload(const void *src, void *dst, size_t bytes, cudaStream_t stream);
cudaError_t launch_plan_upload_sized(const void *src, void *dst, size_t max_bytes, cudaStream_t stream);
cudaError_t launch_kv_append(const int32_t *slots, int n_tokens, int hkv, int num_pages,
                             const uint16_t *k, const uint16_t *v, uint16_t *k_pool,
                             uint16_t *v_pool, uint32_t *err, cudaStream_t stream);
}  // namespace mx

using namespace mx;

static_assert(sizeof(DecodeInfo) == 16 && sizeof(int4) == 16, "plan records are four int32");

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

constexpr int kPlanSlots = 4;         // ring of work-list buffers
constexpr int kPartSlots = 16384;     // decode split partials capacity
// Workspace sets (counters, partials), used by consecutive launches in turn.
// A launch lets its successor start as soon as its own CTAs are resident and
// waits for its predecessor before it exits, so when launch n + 3 starts,
// launch n has completed and its set is free again.
constexpr int kWorkSets = 3;
constexpr int kPrePartSlots = 1024;   // prefill piece partials capacity (64 KiB each)
constexpr int kMinPieceTiles = 16;    // smallest prefill piece, in 128-key tiles
constexpr int kMaxSplitKeys = kWarps * 32 * kPage;  // 4096: one page id per lane
constexpr uint64_t kTimeoutNs = 1000000000ull;      // 1 s bound on in-kernel waits

}  // namespace

struct mx_ctx {
    mx_geom g{};
    int device = 0;
    int num_sms = 0;
    int max_items = 0;
    // workspace (device)
    uint8_t *ws = nullptr;
    // kWorkSets workspace sets, used by consecutive launches in turn: a layer
    // kernel may start while the previous one drains (programmatic dependent
    // launch), and by the time a set comes round again, the launch that last
    // used it has completed.
    struct Set {
        float *part_o, *part_lse;
        uint32_t *merge_cnt;
        float *pre_o, *pre_lse;
        uint32_t *pre_cnt;
        uint32_t *work_cnt;
    } set[kWorkSets] = {};
    uint64_t launch_seq = 0;
    uint32_t *err = nullptr;
    uint8_t *plan_dev[kPlanSlots] = {};
    // pinned staging for the work list
    uint8_t *plan_host[kPlanSlots] = {};
    const void *plan_host_dev[kPlanSlots] = {};  // device view of plan_host (mapped pinned memory)
    cudaEvent_t plan_ev[kPlanSlots] = {};    // upload of the slot done
    bool plan_ev_used[kPlanSlots] = {};
    cudaEvent_t slot_done[kPlanSlots] = {};  // last kernel reading the slot done
    bool slot_done_used[kPlanSlots] = {};
    cudaStream_t up_stream = nullptr;        // plan uploads, off the caller's stream
    size_t plan_bytes = 0;
    int plan_next = 0;
    cudaEvent_t ev_start = nullptr, ev_end = nullptr;
    EncodeTiledFn encode = nullptr;
    // options
    int split_keys_opt = 0;
    int grid_opt = 0;
    int piece_tiles_opt = 0;
    int pdl = 1;  // MX_OPT_PDL: 0 stream order, 1 dependent layers, 2 independent layers
    uint64_t wait_limit_ns = kTimeoutNs;  // MX_OPT_WAIT_LIMIT_US
    int stall_block = -1;                 // MX_OPT_TEST_STALL_BLOCK - 1
    int v_stages_opt = 0;                 // MX_OPT_V_STAGES (0 = automatic)
    int dec_ctas_opt = 0;                 // MX_OPT_DECODE_CTAS (0 = automatic, -1 = none)
    size_t merge_bytes = 0, pre_cnt_bytes = 0;
    // last plan
    int last_items = 0, last_split = 0, last_prefill_items = 0, last_piece_tiles = 0;
    std::string last_error;
    // Replayed iterations (mx_iteration_graph): a plan slot of fixed layout
    // (header, decode table, chunk table, items), allocated on first use, and
    // one captured graph per V ring depth.
    uint8_t *gplan_dev = nullptr, *gplan_host = nullptr;
    const void *gplan_host_dev = nullptr;
    size_t gplan_bytes = 0;
    cudaEvent_t gdone = nullptr;   // the last replay has finished (its plan was read)
    bool gdone_used = false;
    cudaStream_t cap_stream = nullptr;
    struct Graph {
        // what the captured launches hold as constants: a change re-captures
        std::vector<mx_layer_bufs> layers;
        const int32_t *page_table = nullptr, *slots = nullptr;
        int grid = 0, pdl = -1, stall_block = -1;
        uint64_t wait_ns = 0;
        cudaGraphExec_t exec = nullptr;
    } graphs[2];   // [v_stages - 2]
};

namespace {

// Why the calling thread's last mx_create failed (there is no context to
// hold it); mx_error_detail(NULL, ...) returns it.
thread_local std::string t_create_error;

int create_fail(int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_create_error = buf;
    return code;
}

int fail(mx_ctx *c, int code, const char *fmt, ...)
{
    if (c) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, sizeof buf, fmt, ap);
        va_end(ap);
        c->last_error = buf;
    }
    return code;
}

int cuda_fail(mx_ctx *c, cudaError_t e, const char *what)
{
    return fail(c, MX_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Plan {
    const PrefillInfo *pre_dev = nullptr;
    int n_prefills = 0;
    int n_items = 0;
    int n_prefill = 0;
    int split_keys = 0;
    int v_stages = 2;
    int dec_ctas = 0;
    int slot = 0;
    const int4 *items_dev = nullptr;
    const DecodeInfo *dec_dev = nullptr;
};

// Staging layout of one plan: DecodeInfo[n_decodes], then int4 items[n_items]
// (both 16-byte records), uploaded with one copy.
size_t plan_capacity_bytes(const mx_ctx *c)
{
    return (size_t)std::max(c->g.max_decodes, 1) * sizeof(DecodeInfo) + (size_t)kMaxPrefills * sizeof(PrefillInfo) +
           (size_t)c->max_items * sizeof(int4);
}

// The geometries the kernels support.
bool geom_ok(const mx_geom &g)
{
    if (g.head_dim != kHeadDim || g.page_size != kPage || g.num_kv_heads <= 0 ||
        g.num_kv_heads > kMaxDecodeKvHeads || g.num_q_heads <= 0 || g.num_q_heads % g.num_kv_heads != 0 ||
        g.num_q_heads / g.num_kv_heads > kMaxRep || g.num_pages <= 0 || g.num_seqs <= 0 ||
        g.max_pages_per_seq <= 0 || g.max_tokens < 0 || g.max_decodes < 0 ||
        (int64_t)g.num_pages * g.num_kv_heads * kPage > INT32_MAX)
        return false;
    const int rep = g.num_q_heads / g.num_kv_heads;
    return (rep & (rep - 1)) == 0;
}

// Errors of the context-free helpers below go to a string.
int fail_to(std::string *err, int code, const char *fmt, ...)
{
    if (err) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(buf, sizeof buf, fmt, ap);
        va_end(ap);
        *err = buf;
    }
    return code;
}

// Host validation of a descriptor against the geometry.  need_tables: the
// device page table and slots must be given (a launch); planning alone reads
// only the host arrays.
int validate_desc(const mx_geom &g, const mx_iter_desc *d, bool need_tables, std::string *err)
{
    if (!d)
        return fail_to(err, MX_EINVAL, "null descriptor");
    if (d->n_decodes < 0 || d->p_t < 0 || d->chunk_start < 0)
        return fail_to(err, MX_EINVAL, "negative n_decodes, p_t or chunk_start");
    if (d->n_decodes > g.max_decodes)
        return fail_to(err, MX_ECAPACITY, "n_decodes %d > max_decodes %d", d->n_decodes, g.max_decodes);
    if (d->n_prefills < 0 || d->n_prefills > kMaxPrefills || (d->n_prefills > 0 && !d->prefills))
        return fail_to(err, MX_EINVAL, "n_prefills %d outside [0, %d] or prefills null", d->n_prefills,
                       kMaxPrefills);
    if (d->n_prefills > 0 && (d->p_t != 0 || d->chunk_start != 0))
        return fail_to(err, MX_EINVAL, "with n_prefills > 0, p_t and chunk_start must be 0");
    const int64_t cap = (int64_t)g.max_pages_per_seq * kPage;
    int64_t n_tok = d->n_decodes + (int64_t)d->p_t;
    for (int f = 0; f < d->n_prefills; ++f) {
        const mx_prefill &x = d->prefills[f];
        if (x.p_t <= 0 || x.chunk_start < 0)
            return fail_to(err, MX_EINVAL, "prefill %d: p_t %d <= 0 or chunk_start %d < 0", f, x.p_t,
                           x.chunk_start);
        if (x.seq_id < 0 || x.seq_id >= g.num_seqs)
            return fail_to(err, MX_EINVAL, "prefill %d: seq id %d outside [0, %d)", f, x.seq_id, g.num_seqs);
        if ((int64_t)x.chunk_start + x.p_t > cap)
            return fail_to(err, MX_ECAPACITY, "prefill %d: chunk end %lld exceeds %lld page-table slots", f,
                           (long long)x.chunk_start + x.p_t, (long long)cap);
        for (int e = 0; e < f; ++e)
            if (d->prefills[e].seq_id == x.seq_id)
                return fail_to(err, MX_EINVAL, "prefills %d and %d are chunks of the same sequence", e, f);
        n_tok += x.p_t;
    }
    if (n_tok > g.max_tokens)
        return fail_to(err, MX_ECAPACITY, "n_tokens = %lld > max_tokens %d", (long long)n_tok, g.max_tokens);
    if (d->n_decodes > 0 && (!d->decode_seq_ids || !d->decode_ctx_lens))
        return fail_to(err, MX_EINVAL, "decode_seq_ids / decode_ctx_lens are null");
    for (int i = 0; i < d->n_decodes; ++i) {
        const int s = d->decode_seq_ids[i], n = d->decode_ctx_lens[i];
        if (s < 0 || s >= g.num_seqs)
            return fail_to(err, MX_EINVAL, "decode %d: seq id %d outside [0, %d)", i, s, g.num_seqs);
        if (n < 0 || (int64_t)n + 1 > cap)
            return fail_to(err, MX_ECAPACITY, "decode %d: ctx %d + 1 exceeds %lld page-table slots", i, n,
                           (long long)cap);
    }
    if (d->p_t > 0) {
        if (d->prefill_seq_id < 0 || d->prefill_seq_id >= g.num_seqs)
            return fail_to(err, MX_EINVAL, "prefill seq id %d outside [0, %d)", d->prefill_seq_id,
                           g.num_seqs);
        if ((int64_t)d->chunk_start + d->p_t > cap)
            return fail_to(err, MX_ECAPACITY, "chunk end %lld exceeds %lld page-table slots",
                           (long long)d->chunk_start + d->p_t, (long long)cap);
    }
    // A sequence takes part once per iteration, as one decode or as one
    // prefill chunk: two entries of one sequence would append to and read
    // the same pages in the same launch.
    {
        std::vector<int32_t> ids(d->decode_seq_ids, d->decode_seq_ids + d->n_decodes);
        for (int f = 0; f < d->n_prefills; ++f)
            ids.push_back(d->prefills[f].seq_id);
        if (d->n_prefills == 0 && d->p_t > 0)
            ids.push_back(d->prefill_seq_id);
        std::sort(ids.begin(), ids.end());
        const auto rep = std::adjacent_find(ids.begin(), ids.end());
        if (rep != ids.end())
            return fail_to(err, MX_EINVAL, "sequence %d appears twice in the iteration (decodes and chunks)",
                           *rep);
    }
    if (need_tables && n_tok > 0 && (!d->page_table || !d->slots))
        return fail_to(err, MX_EINVAL, "page_table / slots are null");
    return MX_OK;
}

// The iteration's prefill chunks in token order (the single chunk of the
// descriptor, or its array), with their token and query-tile offsets.
std::vector<PrefillInfo> prefill_list(const mx_iter_desc *d)
{
    std::vector<PrefillInfo> v;
    int tb = d->n_decodes, tile = 0;
    auto add = [&](int seq, int cs, int p) {
        PrefillInfo x{};
        x.seq = seq;
        x.chunk_start = cs;
        x.p_t = p;
        x.token_base = tb;
        x.tile_base = tile;
        v.push_back(x);
        tb += p;
        tile += (p + kTileM - 1) / kTileM;
    };
    if (d->n_prefills > 0) {
        for (int f = 0; f < d->n_prefills; ++f)
            add(d->prefills[f].seq_id, d->prefills[f].chunk_start, d->prefills[f].p_t);
    } else if (d->p_t > 0) {
        add(d->prefill_seq_id, d->chunk_start, d->p_t);
    }
    return v;
}

int64_t token_count(const mx_iter_desc *d)
{
    int64_t n = d->n_decodes + (int64_t)d->p_t;
    for (int f = 0; f < d->n_prefills; ++f)
        n += d->prefills[f].p_t;
    return n;
}

int validate(mx_ctx *c, const mx_iter_desc *d)
{
    if (!c)
        return MX_EINVAL;
    return validate_desc(c->g, d, true, &c->last_error);
}

int validate_bufs(mx_ctx *c, const mx_layer_bufs *b, int n_tokens)
{
    if (!b)
        return fail(c, MX_EINVAL, "null layer buffers");
    if (n_tokens == 0)
        return MX_OK;
    const void *ps[] = {b->q, b->k, b->v, b->k_pool, b->v_pool, b->out};
    for (const void *p : ps) {
        if (!p)
            return fail(c, MX_EINVAL, "a layer tensor pointer is null");
        if (!aligned16(p))
            return fail(c, MX_EINVAL, "a layer tensor pointer is not 16-byte aligned");
    }
    return MX_OK;
}

// Tunables of the planner and what it chose.
struct PlanKnobs {
    int num_sms;
    int split_keys_opt;    // 0 = automatic
    int piece_tiles_opt;   // 0 = automatic
    int pdl;               // launch order (MX_OPT_PDL)
    int max_items;         // capacity of the items array
    int v_stages_opt = 0;  // MX_OPT_V_STAGES (0 = automatic)
    int dec_ctas_opt = 0;  // MX_OPT_DECODE_CTAS (0 = automatic, -1 = none)
    int grid = 0;          // CTAs of the launch (0 = num_sms)
};
struct WorkList {
    int n_items = 0, n_prefill = 0, n_prefills = 0, split_keys = 0, piece_tiles = 0, v_stages = 2, dec_ctas = 0;
};

// Key pieces of query tile t of a chunk at chunk_start with nT key tiles.
// A prompt's first tile at chunk_start < kShortRowKeys stays whole: its rows
// of at most 16 keys are recomputed exactly in fp32 from the key tiles the
// item holds (with so few keys, P rounded to bf16 would show in the output),
// and a piece would hold only some of them.
int tile_pieces(int chunk_start, int t, int nT, int piece)
{
    if (t == 0 && chunk_start < kShortRowKeys)
        return 1;
    return (nT + piece - 1) / piece;
}

// a1: the per-iteration work list, on the host, into dec[n_decodes] and
// items[].  Prefill tiles first, heaviest (latest rows, most keys) first;
// then decode splits, longest first.
int build_work_list(const mx_geom &g, const mx_iter_desc *d, const PlanKnobs &k, DecodeInfo *dec,
                    PrefillInfo *pre, int4 *items, WorkList *out, std::string *err)
{
    const int hkv = g.num_kv_heads, hq = g.num_q_heads;
    const std::vector<PrefillInfo> pfs = prefill_list(d);
    const int n_pf = (int)pfs.size();
    int n_qt = 0;  // query tiles over all chunks
    for (const PrefillInfo &x : pfs)
        n_qt += (x.p_t + kTileM - 1) / kTileM;
    const int nd = d->n_decodes;
    int64_t total_keys = 0;
    for (int i = 0; i < nd; ++i)
        total_keys += (int64_t)d->decode_ctx_lens[i] + 1;
    total_keys *= hkv;

    int split = k.split_keys_opt;
    if (split <= 0) {
        // splits per SM: the rule of decode_splits_per_sm (mx_internal.h)
        const double per_sm = decode_splits_per_sm(n_qt, k.pdl == 2, total_keys, k.num_sms);
        const int64_t target_items = std::max<int64_t>(1, (int64_t)(per_sm * k.num_sms));
        int64_t s = (total_keys + target_items - 1) / target_items;
        s = (s + 127) / 128 * 128;
        split = (int)std::min<int64_t>(std::max<int64_t>(s, 512), kMaxSplitKeys);
    }
    split = std::min(std::max(split / 128 * 128, 128), kMaxSplitKeys);
    auto count_parts = [&](int sk) {
        int64_t parts = 0;
        for (int i = 0; i < nd; ++i) {
            const int ns = (d->decode_ctx_lens[i] + 1 + sk - 1) / sk;
            if (ns > 1)
                parts += (int64_t)ns * hkv;
        }
        return parts;
    };
    while (count_parts(split) > kPartSlots && split < kMaxSplitKeys)
        split = std::min(split * 2, kMaxSplitKeys);
    if (count_parts(split) > kPartSlots)
        return fail_to(err, MX_ECAPACITY, "decode splits exceed the partial workspace");

    // Prefill items: a query tile of two query heads of one KV head (one K/V
    // tile load serves both; one head when Hq = Hkv), split along their key
    // tiles into pieces of at most piece_tiles tiles so that long causal rows
    // spread over several SMs.
    const int nh = hq / hkv >= 2 ? 2 : 1;   // heads per prefill item
    const int n_grp = hq / nh;              // prefill items per query tile
    int n = 0;
    int64_t pre_work = 0;
    for (const PrefillInfo &x : pfs) {
        const int nA = (x.chunk_start + kTileN - 1) / kTileN;
        for (int t = 0; t < (x.p_t + kTileM - 1) / kTileM; ++t)
            pre_work += (int64_t)(nA + t + 1) * n_grp;
    }
    // Splitting costs a partial write and a merge; it pays only when the
    // chunk has too few items to occupy the GPU (short chunks deep into a
    // long prompt), so tiles are split only then, into pieces of twice the
    // per-SM share of the prefill work, at least 16 tiles (on the 0.6B
    // sweep's 256- to 1024-row chunks at position 4096 this matched the best
    // of a 8-32-tile sweep; wider geometries have enough items unsplit).
    int piece = k.piece_tiles_opt;
    if (piece <= 0) {
        if ((int64_t)n_qt * n_grp * 2 >= k.num_sms)
            piece = 65535;
        else
            piece = (int)std::max<int64_t>(kMinPieceTiles, 2 * ((pre_work + k.num_sms - 1) / k.num_sms));
    }
    auto count_pre_parts = [&](int pc) {
        int64_t parts = 0;
        for (const PrefillInfo &x : pfs) {
            const int nA = (x.chunk_start + kTileN - 1) / kTileN;
            for (int t = 0; t < (x.p_t + kTileM - 1) / kTileM; ++t) {
                const int ns = tile_pieces(x.chunk_start, t, nA + t + 1, pc);
                if (ns > 1)
                    parts += (int64_t)ns * hq;   // one partial per piece and head
            }
        }
        return parts;
    };
    while (count_pre_parts(piece) > kPrePartSlots)
        piece *= 2;
    struct PItem { int tiles; int4 code; };
    std::vector<PItem> pitems;
    pitems.reserve(64);
    int pre_part = 0;
    for (int f = 0; f < n_pf; ++f) {
        pre[f] = pfs[f];
        const int nA = (pfs[f].chunk_start + kTileN - 1) / kTileN;
        for (int t = (pfs[f].p_t + kTileM - 1) / kTileM - 1; t >= 0; --t) {
            const int nT = nA + t + 1;
            const int ns = tile_pieces(pfs[f].chunk_start, t, nT, piece);
            for (int gq = 0; gq < n_grp; ++gq) {
                const int base = ns > 1 ? pre_part : 0;
                if (ns > 1)
                    pre_part += ns * nh;   // head e of piece s: base + e * ns + s
                for (int s2 = 0; s2 < ns; ++s2) {
                    const int len = (int)((int64_t)(s2 + 1) * nT / ns - (int64_t)s2 * nT / ns);
                    pitems.push_back({len, prefill_item_code(f, t, gq * nh, nh, s2, ns, base)});
                }
            }
        }
    }
    std::stable_sort(pitems.begin(), pitems.end(),
                     [](const PItem &a, const PItem &b) { return a.tiles > b.tiles; });
    if ((int64_t)pitems.size() > k.max_items)
        return fail_to(err, MX_ECAPACITY, "%zu prefill items exceed capacity %d", pitems.size(), k.max_items);
    std::vector<int> pre_tiles;
    pre_tiles.reserve(pitems.size());
    for (const PItem &x : pitems) {
        items[n++] = x.code;
        pre_tiles.push_back(x.tiles);
    }
    const int n_prefill = n;

    // A decode with more keys than the split size is cut into equal
    // page-aligned parts (no short remainder split: each split pays a fixed
    // start-up and a merge).
    int part = 0;
    struct DItem { int keys; int i, h, s, len; };
    std::vector<DItem> ditems;
    ditems.reserve(64);
    for (int i = 0; i < nd; ++i) {
        const int keys = d->decode_ctx_lens[i] + 1;
        const int ns = (keys + split - 1) / split;
        const int len = ((keys + ns - 1) / ns + kPage - 1) / kPage * kPage;
        if (ns > kMaxDecodeSplits)
            return fail_to(err, MX_ECAPACITY, "decode %d needs %d splits (limit %d)", i, ns, kMaxDecodeSplits);
        dec[i].seq = d->decode_seq_ids[i];
        dec[i].ctx = d->decode_ctx_lens[i];
        dec[i].n_splits = ns;
        dec[i].part_base = ns > 1 ? part : 0;
        if (ns > 1)
            part += ns * hkv;
        for (int h = 0; h < hkv; ++h)
            for (int s = 0; s < ns; ++s)
                ditems.push_back({std::min(len, keys - s * len), i, h, s, len});
    }
    if (n_prefill + (int)ditems.size() > k.max_items)
        return fail_to(err, MX_ECAPACITY, "work list of %zu items exceeds capacity %d",
                       n_prefill + ditems.size(), k.max_items);
    std::stable_sort(ditems.begin(), ditems.end(),
                     [](const DItem &a, const DItem &b) { return a.keys > b.keys; });
    for (const DItem &x : ditems) {
        int4 code = decode_item_code(x.i, x.h, x.s, dec[x.i].seq, dec[x.i].ctx, x.len);
        if (dec[x.i].ctx + 1 <= kShortKeys)  // few keys: the exact short path
            code.x = (int32_t)(((uint32_t)code.x & ~0xFu) | (uint32_t)ITEM_DECODE_SHORT);
        items[n++] = code;
    }

    // V ring depth: the prefill chunks' causal tensor work against the
    // decode splits' key/value bytes
    double pre_flops = 0.0;
    for (const PrefillInfo &x : pfs)
        pre_flops += 4.0 * hq * kHeadDim * ((double)x.p_t * x.chunk_start + 0.5 * (double)x.p_t * (x.p_t + 1));
    const double dec_bytes = (double)total_keys * kHeadDim * 2 * 2;

    out->n_items = n;
    out->n_prefill = n_prefill;
    out->n_prefills = n_pf;
    out->split_keys = split;
    out->piece_tiles = piece;
    out->v_stages = k.v_stages_opt > 0 ? k.v_stages_opt : choose_v_stages(pre_flops, dec_bytes);
    // CTAs that start on the decode queue (none without both kinds of item)
    if (n_prefill == 0 || n == n_prefill || k.dec_ctas_opt < 0)
        out->dec_ctas = 0;
    else if (k.dec_ctas_opt > 0)
        out->dec_ctas = k.dec_ctas_opt;
    else {
        std::vector<long long> heap(kMaxGrid);
        out->dec_ctas = decode_first_ctas(pre_tiles.data(), n_prefill, pre_flops, dec_bytes,
                                          k.grid > 0 ? k.grid : k.num_sms, heap.data());
    }
    return MX_OK;
}

// Plans into the next pinned staging slot and uploads it.
int plan(mx_ctx *c, const mx_iter_desc *d, cudaStream_t stream, Plan *out)
{
    // staging slot: wait until its previous upload has been consumed
    const int slot = c->plan_next;
    c->plan_next = (slot + 1) % kPlanSlots;
    if (c->plan_ev_used[slot]) {
        cudaError_t e = cudaEventSynchronize(c->plan_ev[slot]);
        if (e != cudaSuccess)
            return cuda_fail(c, e, "cudaEventSynchronize(plan)");
    }
    uint8_t *host = c->plan_host[slot];
    DecodeInfo *dec = reinterpret_cast<DecodeInfo *>(host);
    const size_t pre_off = (size_t)d->n_decodes * sizeof(DecodeInfo);
    PrefillInfo *pre = reinterpret_cast<PrefillInfo *>(host + pre_off);
    const size_t items_off = pre_off + (size_t)kMaxPrefills * sizeof(PrefillInfo);
    int4 *items = reinterpret_cast<int4 *>(host + items_off);
    const PlanKnobs knobs{c->num_sms,   c->split_keys_opt, c->piece_tiles_opt, c->pdl,
                          c->max_items, c->v_stages_opt,   c->dec_ctas_opt,    c->grid_opt};
    WorkList wl;
    int rc = build_work_list(c->g, d, knobs, dec, pre, items, &wl, &c->last_error);
    if (rc)
        return rc;
    const int n = wl.n_items;

    const size_t bytes = items_off + (size_t)n * sizeof(int4);
    // A kernel, not a copy engine, moves the plan (an H2D memcpy would queue
    // behind the caller's own large uploads: one copy engine per direction
    // serves all streams in order), on the context's own stream so that it
    // runs while the caller's stream is still busy with earlier work: it
    // waits only for the last kernel that read this slot, and the caller's
    // stream waits for it.
    cudaError_t e = cudaSuccess;
    if (c->slot_done_used[slot] && (e = cudaStreamWaitEvent(c->up_stream, c->slot_done[slot], 0)) != cudaSuccess)
        return cuda_fail(c, e, "cudaStreamWaitEvent(slot)");
    e = launch_plan_upload(c->plan_host_dev[slot], c->plan_dev[slot], bytes, c->up_stream);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "plan upload");
    if ((e = cudaEventRecord(c->plan_ev[slot], c->up_stream)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(plan)");
    c->plan_ev_used[slot] = true;
    if ((e = cudaStreamWaitEvent(stream, c->plan_ev[slot], 0)) != cudaSuccess)
        return cuda_fail(c, e, "cudaStreamWaitEvent(plan)");

    out->n_items = n;
    out->n_prefill = wl.n_prefill;
    out->split_keys = wl.split_keys;
    out->v_stages = wl.v_stages;
    out->dec_ctas = wl.dec_ctas;
    out->slot = slot;
    out->items_dev = reinterpret_cast<const int4 *>(c->plan_dev[slot] + items_off);
    out->dec_dev = reinterpret_cast<const DecodeInfo *>(c->plan_dev[slot]);
    out->pre_dev = reinterpret_cast<const PrefillInfo *>(c->plan_dev[slot] + pre_off);
    out->n_prefills = wl.n_prefills;
    c->last_items = n;
    c->last_split = wl.split_keys;
    c->last_prefill_items = wl.n_prefill;
    c->last_piece_tiles = wl.piece_tiles;
    return MX_OK;
}

int encode_map(mx_ctx *c, CUtensorMap *m, const void *base, int rank, const cuuint64_t *dims,
               const cuuint64_t *strides_bytes, const cuuint32_t *box)
{
    const cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = c->encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank,
                           const_cast<void *>(base), dims, strides_bytes, box, estr,
                           CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(c, MX_ECUDA, "cuTensorMapEncodeTiled failed (%d)", (int)r);
    return MX_OK;
}

int make_params(mx_ctx *c, const mx_iter_desc *d, const mx_layer_bufs *b, const Plan &pl,
                LayerParams *P, int set, const PlanHeader *hdr = nullptr)
{
    const mx_geom &g = c->g;
    std::memset(P, 0, sizeof *P);
    // a replayed launch's maps span the buffers' capacity (its token count
    // changes from one replay to the next)
    const int n_tok = hdr ? g.max_tokens : (int)token_count(d);
    P->hdr = hdr;
    P->q = static_cast<const uint16_t *>(b->q);
    P->k = static_cast<const uint16_t *>(b->k);
    P->v = static_cast<const uint16_t *>(b->v);
    P->k_pool = static_cast<uint16_t *>(b->k_pool);
    P->v_pool = static_cast<uint16_t *>(b->v_pool);
    P->out = static_cast<uint16_t *>(b->out);
    P->page_table = d->page_table;
    P->slots = d->slots;
    P->items = pl.items_dev;
    P->dec = pl.dec_dev;
    const mx_ctx::Set &w = c->set[set % kWorkSets];
    P->part_o = w.part_o;
    P->part_lse = w.part_lse;
    P->merge_cnt = w.merge_cnt;
    P->pre_o = w.pre_o;
    P->pre_lse = w.pre_lse;
    P->pre_cnt = w.pre_cnt;
    P->work_cnt = w.work_cnt;
    P->err = c->err;
    P->n_items = pl.n_items;
    P->n_pre_items = pl.n_prefill;
    P->dec_ctas = pl.dec_ctas;
    P->n_decodes = d->n_decodes;
    P->pre = pl.pre_dev;
    P->n_prefills = pl.n_prefills;
    P->hq = g.num_q_heads;
    P->hkv = g.num_kv_heads;
    P->n_rep = g.num_q_heads / g.num_kv_heads;
    P->num_pages = g.num_pages;
    P->max_pages = g.max_pages_per_seq;
    P->split_keys = pl.split_keys;
    P->has_prefill = (pl.n_prefill > 0 || hdr) ? 1 : 0;
    P->v_stages = pl.v_stages;
    P->scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)kHeadDim));
    P->timeout_ns = c->wait_limit_ns;
    P->stall_block = c->stall_block;
    if (P->has_prefill) {
        const cuuint64_t hd = kHeadDim;
        {
            const cuuint64_t dims[3] = {hd, (cuuint64_t)g.num_q_heads, (cuuint64_t)n_tok};
            const cuuint64_t str[2] = {hd * 2, hd * 2 * g.num_q_heads};
            const cuuint32_t box[3] = {64, 1, (cuuint32_t)kTileM};
            int rc = encode_map(c, &P->tm_q, b->q, 3, dims, str, box);
            if (rc)
                return rc;
        }
        {
            const cuuint64_t dims[3] = {hd, (cuuint64_t)g.num_kv_heads, (cuuint64_t)n_tok};
            const cuuint64_t str[2] = {hd * 2, hd * 2 * g.num_kv_heads};
            const cuuint32_t box[3] = {64, 1, (cuuint32_t)kTileN};
            int rc = encode_map(c, &P->tm_k, b->k, 3, dims, str, box);
            if (!rc)
                rc = encode_map(c, &P->tm_v, b->v, 3, dims, str, box);
            if (rc)
                return rc;
        }
        {
            const cuuint64_t rows = (cuuint64_t)g.num_pages * g.num_kv_heads * kPage;
            const cuuint64_t dims[2] = {hd, rows};
            const cuuint64_t str[1] = {hd * 2};
            const cuuint32_t box[2] = {64, (cuuint32_t)kPage};
            int rc = encode_map(c, &P->tm_kpool, b->k_pool, 2, dims, str, box);
            if (!rc)
                rc = encode_map(c, &P->tm_vpool, b->v_pool, 2, dims, str, box);
            if (rc)
                return rc;
        }
    }
    return MX_OK;
}

int grid_for(const mx_ctx *c, const Plan &pl)
{
    int grid = c->grid_opt > 0 ? c->grid_opt : c->num_sms;
    return std::max(1, std::min(grid, pl.n_items));
}

// The plan slot may be rewritten once the kernels enqueued on `st` so far
// (the last ones reading it) have finished.
int release_slot(mx_ctx *c, const Plan &pl, cudaStream_t st)
{
    cudaError_t e = cudaEventRecord(c->slot_done[pl.slot], st);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(slot)");
    c->slot_done_used[pl.slot] = true;
    return MX_OK;
}

int read_error_word(mx_ctx *c)
{
    uint32_t w = 0;
    cudaError_t e = cudaMemcpy(&w, c->err, sizeof w, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "reading the error word");
    if (w == 0)
        return MX_OK;
    // A launch that flagged an error may have left items undone, so its
    // arrival and work counters (normally reset by the launch itself) are
    // cleared too; the stream has been waited on, so the workspace is idle.
    cudaStream_t s = c->up_stream;
    for (int k = 0; k < kWorkSets && e == cudaSuccess; ++k)
        if ((e = cudaMemsetAsync(c->set[k].merge_cnt, 0, c->merge_bytes, s)) == cudaSuccess &&
            (e = cudaMemsetAsync(c->set[k].pre_cnt, 0, c->pre_cnt_bytes, s)) == cudaSuccess)
            e = cudaMemsetAsync(c->set[k].work_cnt, 0, 256, s);
    if (e == cudaSuccess && (e = cudaMemsetAsync(c->err, 0, sizeof(uint32_t), s)) == cudaSuccess)
        e = cudaStreamSynchronize(s);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "clearing the error word and counters");
    if (w & ERR_TIMEOUT)
        return fail(c, MX_ETIMEOUT, "a bounded in-kernel wait timed out (error word 0x%x)", w);
    if (w & ERR_PAGE)
        return fail(c, MX_ERANGE_PAGE, "a page id outside [0, num_pages) was read (error word 0x%x)", w);
    return fail(c, MX_ERANGE_SLOT, "a slot outside the pool was skipped (error word 0x%x)", w);
}

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev)
    {
        if (cudaGetDevice(&prev) == cudaSuccess && prev != dev)
            cudaSetDevice(dev);
        else
            prev = -1;
    }
    ~DeviceGuard()
    {
        if (prev >= 0)
            cudaSetDevice(prev);
    }
};

}  // namespace

extern "C" {

int mx_create(mx_ctx **out, const mx_geom *g, int device)
{
    t_create_error.clear();
    if (!out || !g)
        return create_fail(MX_EINVAL, "null out or geometry");
    *out = nullptr;
    if (!geom_ok(*g))
        return create_fail(MX_EINVAL,
                           "unsupported geometry: head_dim must be 128, page_size 16, Hq / Hkv a power of "
                           "two of at most 8, Hkv <= %d, and the sizes positive",
                           kMaxDecodeKvHeads);
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || device < 0 || device >= ndev)
        return create_fail(MX_EDEVICE, "device %d: no such CUDA device (%d found)", device, ndev);
    DeviceGuard guard(device);
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, device) != cudaSuccess || prop.major != 10)
        return create_fail(MX_EDEVICE, "device %d is not an sm_100-family GPU", device);

    mx_ctx *c = new mx_ctx();
    c->g = *g;
    c->device = device;
    c->num_sms = prop.multiProcessorCount;
    // every chunk may end in a ragged tile
    const int max_qtiles = std::max((g->max_tokens + kTileM - 1) / kTileM, 1) + kMaxPrefills - 1;
    const int max_prefill_items = max_qtiles * g->num_q_heads + kPrePartSlots;
    c->max_items = max_prefill_items + kPartSlots + std::max(g->max_decodes, 1) * g->num_kv_heads;

    auto bail = [&](cudaError_t e, const char *what) {
        mx_destroy(c);
        return create_fail(MX_ECUDA, "%s: %s", what, cudaGetErrorString(e));
    };
    cudaError_t e;
    if ((e = init_layer_kernel()) != cudaSuccess)
        return bail(e, "cudaFuncSetAttribute");

    const size_t part_o_bytes = (size_t)kPartSlots * kMaxRep * kHeadDim * sizeof(float);
    const size_t part_lse_bytes = (size_t)kPartSlots * kMaxRep * sizeof(float);
    const size_t merge_bytes = (size_t)std::max(g->max_decodes, 1) * g->num_kv_heads * sizeof(uint32_t);
    const size_t pre_o_bytes = (size_t)kPrePartSlots * kTileM * kHeadDim * sizeof(float);
    const size_t pre_lse_bytes = (size_t)kPrePartSlots * kTileM * sizeof(float);
    const size_t pre_cnt_bytes = (((size_t)max_qtiles * g->num_q_heads * sizeof(uint32_t)) + 255) & ~size_t(255);
    c->merge_bytes = merge_bytes;
    c->pre_cnt_bytes = pre_cnt_bytes;
    c->plan_bytes = plan_capacity_bytes(c);
    const size_t plan_stride = (c->plan_bytes + 255) & ~size_t(255);
    const size_t set_bytes = part_o_bytes + part_lse_bytes + ((merge_bytes + 255) & ~size_t(255)) +
                             pre_o_bytes + pre_lse_bytes + pre_cnt_bytes + 256 /*work counters*/;
    const size_t total = kWorkSets * set_bytes + 256 /*error word*/ + kPlanSlots * plan_stride;
    if ((e = cudaMalloc(&c->ws, total)) != cudaSuccess)
        return bail(e, "cudaMalloc(workspace)");
    uint8_t *p = c->ws;
    for (int k = 0; k < kWorkSets; ++k) {
        mx_ctx::Set &w = c->set[k];
        w.part_o = reinterpret_cast<float *>(p);
        p += part_o_bytes;
        w.part_lse = reinterpret_cast<float *>(p);
        p += part_lse_bytes;
        w.merge_cnt = reinterpret_cast<uint32_t *>(p);
        p += (merge_bytes + 255) & ~size_t(255);
        w.pre_o = reinterpret_cast<float *>(p);
        p += pre_o_bytes;
        w.pre_lse = reinterpret_cast<float *>(p);
        p += pre_lse_bytes;
        w.pre_cnt = reinterpret_cast<uint32_t *>(p);
        p += pre_cnt_bytes;
        w.work_cnt = reinterpret_cast<uint32_t *>(p);
        p += 256;
    }
    c->err = reinterpret_cast<uint32_t *>(p);
    p += 256;
    for (int s = 0; s < kPlanSlots; ++s) {
        c->plan_dev[s] = p;
        p += plan_stride;
        if ((e = cudaMallocHost(&c->plan_host[s], c->plan_bytes)) != cudaSuccess)
            return bail(e, "cudaMallocHost(plan)");
        void *dv = nullptr;
        if ((e = cudaHostGetDevicePointer(&dv, c->plan_host[s], 0)) != cudaSuccess)
            return bail(e, "cudaHostGetDevicePointer(plan)");
        c->plan_host_dev[s] = dv;
        if ((e = cudaEventCreateWithFlags(&c->plan_ev[s], cudaEventDisableTiming)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&c->slot_done[s], cudaEventDisableTiming)) != cudaSuccess)
            return bail(e, "cudaEventCreate");
    }
    for (int k = 0; k < kWorkSets; ++k)
        if ((e = cudaMemset(c->set[k].merge_cnt, 0, merge_bytes)) != cudaSuccess ||
            (e = cudaMemset(c->set[k].pre_cnt, 0, pre_cnt_bytes)) != cudaSuccess ||
            (e = cudaMemset(c->set[k].work_cnt, 0, 256)) != cudaSuccess)
            return bail(e, "cudaMemset(workspace)");
    if ((e = cudaMemset(c->err, 0, 256)) != cudaSuccess)
        return bail(e, "cudaMemset(error word)");
    if ((e = cudaEventCreate(&c->ev_start)) != cudaSuccess ||
        (e = cudaEventCreate(&c->ev_end)) != cudaSuccess)
        return bail(e, "cudaEventCreate");
    if ((e = cudaStreamCreateWithFlags(&c->up_stream, cudaStreamNonBlocking)) != cudaSuccess)
        return bail(e, "cudaStreamCreate");

    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
        mx_destroy(c);
        return create_fail(MX_ECUDA, "cuTensorMapEncodeTiled entry point not found");
    }
    c->encode = reinterpret_cast<EncodeTiledFn>(fn);
    if ((e = cudaDeviceSynchronize()) != cudaSuccess)
        return bail(e, "cudaDeviceSynchronize");
    *out = c;
    return MX_OK;
}

int mx_destroy(mx_ctx *c)
{
    if (!c)
        return MX_OK;
    DeviceGuard guard(c->device);
    cudaDeviceSynchronize();
    for (int s = 0; s < kPlanSlots; ++s) {
        if (c->plan_host[s])
            cudaFreeHost(c->plan_host[s]);
        if (c->plan_ev[s])
            cudaEventDestroy(c->plan_ev[s]);
        if (c->slot_done[s])
            cudaEventDestroy(c->slot_done[s]);
    }
    for (mx_ctx::Graph &gr : c->graphs)
        if (gr.exec)
            cudaGraphExecDestroy(gr.exec);
    if (c->gplan_host)
        cudaFreeHost(c->gplan_host);
    if (c->gplan_dev)
        cudaFree(c->gplan_dev);
    if (c->gdone)
        cudaEventDestroy(c->gdone);
    if (c->cap_stream)
        cudaStreamDestroy(c->cap_stream);
    if (c->up_stream)
        cudaStreamDestroy(c->up_stream);
    if (c->ev_start)
        cudaEventDestroy(c->ev_start);
    if (c->ev_end)
        cudaEventDestroy(c->ev_end);
    if (c->ws)
        cudaFree(c->ws);
    delete c;
    return MX_OK;
}

int mx_kv_append(mx_ctx *c, const int32_t *slots, int32_t n_tokens, const void *k, const void *v,
                 void *k_pool, void *v_pool, void *stream)
{
    if (!c)
        return MX_EINVAL;
    if (n_tokens < 0)
        return fail(c, MX_EINVAL, "n_tokens < 0");
    if (n_tokens == 0)
        return MX_OK;
    if (!slots || !k || !v || !k_pool || !v_pool)
        return fail(c, MX_EINVAL, "null pointer");
    if (!aligned16(k) || !aligned16(v) || !aligned16(k_pool) || !aligned16(v_pool))
        return fail(c, MX_EINVAL, "tensor pointers must be 16-byte aligned");
    DeviceGuard guard(c->device);
    cudaError_t e = launch_kv_append(slots, n_tokens, c->g.num_kv_heads, c->g.num_pages,
                                     static_cast<const uint16_t *>(k), static_cast<const uint16_t *>(v),
                                     static_cast<uint16_t *>(k_pool), static_cast<uint16_t *>(v_pool),
                                     c->err, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess)
        return cuda_fail(c, e, "kv_append launch");
    return MX_OK;
}

int mx_mixed_attention(mx_ctx *c, const mx_iter_desc *d, const mx_layer_bufs *b, void *stream)
{
    int rc = validate(c, d);
    if (rc)
        return rc;
    const int n_tok = (int)token_count(d);
    if ((rc = validate_bufs(c, b, n_tok)))
        return rc;
    if (n_tok == 0)
        return MX_OK;
    DeviceGuard guard(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Plan pl;
    if ((rc = plan(c, d, st, &pl)))
        return rc;
    LayerParams P;
    if ((rc = make_params(c, d, b, pl, &P, (int)(c->launch_seq % kWorkSets))))
        return rc;
    // ordinary stream order: the caller's next or previous work may depend on it
    cudaError_t e = launch_mixed_layer(P, grid_for(c, pl), st, false);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "mixed_layer launch");
    ++c->launch_seq;
    return release_slot(c, pl, st);
}

int mx_iteration(mx_ctx *c, const mx_iter_desc *d, int32_t n_layers, const mx_layer_bufs *layers,
                 float *device_us_out, void *stream)
{
    int rc = validate(c, d);
    if (rc)
        return rc;
    if (n_layers < 0 || (n_layers > 0 && !layers))
        return fail(c, MX_EINVAL, "bad n_layers / layers");
    const bool timed = device_us_out != nullptr;
    const int n_tok = (int)token_count(d);
    for (int l = 0; l < n_layers; ++l)
        if ((rc = validate_bufs(c, layers + l, n_tok)))
            return rc;
    DeviceGuard guard(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Plan pl;
    const bool work = n_tok > 0 && n_layers > 0;
    if (work && (rc = plan(c, d, st, &pl)))
        return rc;
    // all descriptors are encoded before the timed region starts
    std::vector<LayerParams> params(work ? n_layers : 0);
    for (int l = 0; work && l < n_layers; ++l)
        if ((rc = make_params(c, d, layers + l, pl, &params[l], (int)((c->launch_seq + l) % kWorkSets))))
            return rc;
    cudaError_t e;
    if (timed && (e = cudaEventRecord(c->ev_start, st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(start)");
    // Layer l > 0 is launched with programmatic dependent launch; the first
    // layer keeps ordinary stream order behind whatever the caller enqueued
    // before.
    for (int l = 0; work && l < n_layers; ++l) {
        // Mode 1: layer l+1 launches as layer l's CTAs run out of work, and
        // each of its CTAs waits for layer l to complete (griddepcontrol.wait)
        // before reading anything: layer l+1 may read what layer l wrote, the
        // order of a model whose layers depend on each other, with the launch
        // latency hidden.  Mode 2 (independent layers only): layer l+1's CTAs
        // start on the SMs layer l frees.  That is safe only when a launch
        // occupies every SM (one CTA per SM): then launch n + 3 cannot start
        // before launch n has completed (see kWorkSets); smaller grids keep
        // mode 1.
        const int grid = grid_for(c, pl);
        params[l].early_start = (c->pdl == 2 && grid == c->num_sms) ? 1 : 0;
        e = launch_mixed_layer(params[l], grid, st, c->pdl != 0 && l > 0);
        if (e != cudaSuccess)
            return cuda_fail(c, e, "mixed_layer launch");
        ++c->launch_seq;
    }
    if (work && (rc = release_slot(c, pl, st)))
        return rc;
    if (!timed)
        return MX_OK;
    if ((e = cudaEventRecord(c->ev_end, st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(end)");
    if ((e = cudaEventSynchronize(c->ev_end)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventSynchronize(end)");
    float ms = 0.f;
    if ((e = cudaEventElapsedTime(&ms, c->ev_start, c->ev_end)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventElapsedTime");
    *device_us_out = ms * 1000.0f;
    return read_error_word(c);
}

namespace {

// Fixed layout of the replay plan slot: header, decode table (max_decodes),
// chunk table (kMaxPrefills), items (max_items).
size_t gplan_dec_off() { return sizeof(PlanHeader); }
size_t gplan_pre_off(const mx_ctx *c) { return gplan_dec_off() + (size_t)std::max(c->g.max_decodes, 1) * sizeof(DecodeInfo); }
size_t gplan_items_off(const mx_ctx *c) { return gplan_pre_off(c) + (size_t)kMaxPrefills * sizeof(PrefillInfo); }

int graph_setup(mx_ctx *c)
{
    if (c->gplan_dev)
        return MX_OK;
    const size_t bytes = gplan_items_off(c) + (size_t)c->max_items * sizeof(int4);
    cudaError_t e;
    if ((e = cudaMalloc(&c->gplan_dev, bytes)) != cudaSuccess)
        return cuda_fail(c, e, "cudaMalloc(replay plan)");
    if ((e = cudaMallocHost(&c->gplan_host, bytes)) != cudaSuccess)
        return cuda_fail(c, e, "cudaMallocHost(replay plan)");
    void *dv = nullptr;
    if ((e = cudaHostGetDevicePointer(&dv, c->gplan_host, 0)) != cudaSuccess)
        return cuda_fail(c, e, "cudaHostGetDevicePointer(replay plan)");
    c->gplan_host_dev = dv;
    if ((e = cudaEventCreateWithFlags(&c->gdone, cudaEventDisableTiming)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventCreate(replay)");
    if ((e = cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking)) != cudaSuccess)
        return cuda_fail(c, e, "cudaStreamCreate(capture)");
    c->gplan_bytes = bytes;
    return MX_OK;
}

// Capture the plan upload and the n_layers layer launches of a replayed
// iteration with V ring depth v_stages into a graph.
int graph_capture(mx_ctx *c, const mx_iter_desc *d, int n_layers, const mx_layer_bufs *layers, int v_stages,
                  int grid, cudaGraphExec_t *out)
{
    Plan pl;
    pl.v_stages = v_stages;
    pl.n_prefill = 1;
    pl.items_dev = reinterpret_cast<const int4 *>(c->gplan_dev + gplan_items_off(c));
    pl.dec_dev = reinterpret_cast<const DecodeInfo *>(c->gplan_dev + gplan_dec_off());
    pl.pre_dev = reinterpret_cast<const PrefillInfo *>(c->gplan_dev + gplan_pre_off(c));
    const PlanHeader *hdr = reinterpret_cast<const PlanHeader *>(c->gplan_dev);
    std::vector<LayerParams> params((size_t)n_layers);
    for (int l = 0; l < n_layers; ++l) {
        int rc = make_params(c, d, layers + l, pl, &params[l], l % kWorkSets, hdr);
        if (rc)
            return rc;
        params[l].early_start = (c->pdl == 2 && grid == c->num_sms) ? 1 : 0;
    }
    cudaError_t e = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "cudaStreamBeginCapture");
    cudaError_t le = launch_plan_upload_sized(c->gplan_host_dev, c->gplan_dev, c->gplan_bytes, c->cap_stream);
    for (int l = 0; le == cudaSuccess && l < n_layers; ++l)
        le = launch_mixed_layer(params[l], grid, c->cap_stream, c->pdl != 0 && l > 0);
    cudaGraph_t graph = nullptr;
    e = cudaStreamEndCapture(c->cap_stream, &graph);
    if (le != cudaSuccess || e != cudaSuccess) {
        if (graph)
            cudaGraphDestroy(graph);
        return cuda_fail(c, le != cudaSuccess ? le : e, "capture of the iteration");
    }
    e = cudaGraphInstantiate(out, graph, 0);
    cudaGraphDestroy(graph);
    if (e != cudaSuccess)
        return cuda_fail(c, e, "cudaGraphInstantiate");
    return MX_OK;
}

}  // namespace

int mx_iteration_graph(mx_ctx *c, const mx_iter_desc *d, int32_t n_layers, const mx_layer_bufs *layers,
                       float *device_us_out, void *stream)
{
    int rc = validate(c, d);
    if (rc)
        return rc;
    if (n_layers <= 0 || !layers)
        return fail(c, MX_EINVAL, "bad n_layers / layers");
    // the captured launches read the buffers up to their capacity
    for (int l = 0; l < n_layers; ++l)
        if ((rc = validate_bufs(c, layers + l, std::max(c->g.max_tokens, 1))))
            return rc;
    if (token_count(d) == 0) {
        if (device_us_out)
            *device_us_out = 0.f;
        return MX_OK;
    }
    DeviceGuard guard(c->device);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if ((rc = graph_setup(c)))
        return rc;
    cudaError_t e;
    // the host plan may be rewritten once the last replay has read it
    if (c->gdone_used && (e = cudaEventSynchronize(c->gdone)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventSynchronize(replay)");
    PlanHeader *h = reinterpret_cast<PlanHeader *>(c->gplan_host);
    DecodeInfo *dec = reinterpret_cast<DecodeInfo *>(c->gplan_host + gplan_dec_off());
    PrefillInfo *pre = reinterpret_cast<PrefillInfo *>(c->gplan_host + gplan_pre_off(c));
    int4 *items = reinterpret_cast<int4 *>(c->gplan_host + gplan_items_off(c));
    const PlanKnobs knobs{c->num_sms,   c->split_keys_opt, c->piece_tiles_opt, c->pdl,
                          c->max_items, c->v_stages_opt,   c->dec_ctas_opt,    c->grid_opt};
    WorkList wl;
    if ((rc = build_work_list(c->g, d, knobs, dec, pre, items, &wl, &c->last_error)))
        return rc;
    std::memset(h, 0, sizeof *h);
    h->n_items = wl.n_items;
    h->n_decodes = d->n_decodes;
    h->n_prefills = wl.n_prefills;
    h->has_prefill = wl.n_prefill > 0 ? 1 : 0;
    h->n_pre_items = wl.n_prefill;
    h->dec_ctas = wl.dec_ctas;
    h->words = (int32_t)((gplan_items_off(c) + (size_t)wl.n_items * sizeof(int4)) / sizeof(int4));
    c->last_items = wl.n_items;
    c->last_split = wl.split_keys;
    c->last_prefill_items = wl.n_prefill;
    c->last_piece_tiles = wl.piece_tiles;

    // the graph of this layer array, ring depth, grid and launch order
    const int grid = c->grid_opt > 0 ? c->grid_opt : c->num_sms;
    mx_ctx::Graph &gr = c->graphs[wl.v_stages == 3 ? 1 : 0];
    const bool same = gr.exec && gr.grid == grid && gr.pdl == c->pdl && gr.page_table == d->page_table &&
                      gr.slots == d->slots && gr.stall_block == c->stall_block && gr.wait_ns == c->wait_limit_ns &&
                      gr.layers.size() == (size_t)n_layers &&
                      std::memcmp(gr.layers.data(), layers, sizeof(mx_layer_bufs) * (size_t)n_layers) == 0;
    if (!same) {
        if (gr.exec) {
            cudaGraphExecDestroy(gr.exec);
            gr.exec = nullptr;
        }
        if ((rc = graph_capture(c, d, n_layers, layers, wl.v_stages, grid, &gr.exec)))
            return rc;
        gr.layers.assign(layers, layers + n_layers);
        gr.page_table = d->page_table;
        gr.slots = d->slots;
        gr.grid = grid;
        gr.pdl = c->pdl;
        gr.stall_block = c->stall_block;
        gr.wait_ns = c->wait_limit_ns;
    }
    const bool timed = device_us_out != nullptr;
    if (timed && (e = cudaEventRecord(c->ev_start, st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(start)");
    if ((e = cudaGraphLaunch(gr.exec, st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaGraphLaunch");
    if ((e = cudaEventRecord(c->gdone, st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(replay)");
    c->gdone_used = true;
    if (!timed)
        return MX_OK;
    if ((e = cudaEventRecord(c->ev_end, st)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventRecord(end)");
    if ((e = cudaEventSynchronize(c->ev_end)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventSynchronize(end)");
    float ms = 0.f;
    if ((e = cudaEventElapsedTime(&ms, c->ev_start, c->ev_end)) != cudaSuccess)
        return cuda_fail(c, e, "cudaEventElapsedTime");
    *device_us_out = ms * 1000.0f;
    return read_error_word(c);
}

int mx_sync_status(mx_ctx *c, void *stream)
{
    if (!c)
        return MX_EINVAL;
    DeviceGuard guard(c->device);
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess)
        return cuda_fail(c, e, "cudaStreamSynchronize");
    return read_error_word(c);
}

int mx_error_detail(mx_ctx *c, char *buf, int32_t len)
{
    if (!buf || len <= 0)
        return MX_EINVAL;
    const std::string &msg = c ? c->last_error : t_create_error;
    const size_t n = std::min<size_t>(msg.size(), (size_t)len - 1);
    std::memcpy(buf, msg.data(), n);
    buf[n] = '\0';
    return (int)n;
}

int mx_set_option(mx_ctx *c, int32_t option, int64_t value)
{
    if (!c)
        return MX_EINVAL;
    switch (option) {
    case MX_OPT_SPLIT_KEYS:
        if (value < 0 || value > kMaxSplitKeys || value % 128)
            return fail(c, MX_EINVAL, "split keys must be 0 or a multiple of 128 up to %d", kMaxSplitKeys);
        c->split_keys_opt = (int)value;
        return MX_OK;
    case MX_OPT_PREFILL_PIECE_TILES:
        if (value < 0 || value > 65535)
            return fail(c, MX_EINVAL, "prefill piece tiles must be in [0, 65535]");
        c->piece_tiles_opt = (int)value;
        return MX_OK;
    case MX_OPT_PDL:
        if (value < 0 || value > 2)
            return fail(c, MX_EINVAL, "MX_OPT_PDL is 0, 1 or 2");
        c->pdl = (int)value;
        return MX_OK;
    case MX_OPT_GRID:
        if (value < 0 || value > 65535)
            return fail(c, MX_EINVAL, "grid must be in [0, 65535]");
        c->grid_opt = (int)value;
        return MX_OK;
    case MX_OPT_WAIT_LIMIT_US:
        if (value < 0 || value > 10000000)
            return fail(c, MX_EINVAL, "wait limit must be in [0, 10^7] us");
        c->wait_limit_ns = value == 0 ? kTimeoutNs : (uint64_t)value * 1000ull;
        return MX_OK;
    case MX_OPT_TEST_STALL_BLOCK:
        if (value < 0 || value > 65535)
            return fail(c, MX_EINVAL, "stall block must be in [0, 65535]");
        c->stall_block = (int)value - 1;
        return MX_OK;
    case MX_OPT_V_STAGES:
        if (value != 0 && value != 2 && value != 3)
            return fail(c, MX_EINVAL, "MX_OPT_V_STAGES is 0, 2 or 3");
        c->v_stages_opt = (int)value;
        return MX_OK;
    case MX_OPT_DECODE_CTAS:
        if (value < -1 || value > 65535)
            return fail(c, MX_EINVAL, "MX_OPT_DECODE_CTAS is -1, 0 or a CTA count up to 65535");
        c->dec_ctas_opt = (int)value;
        return MX_OK;
    default:
        return fail(c, MX_EINVAL, "unknown option %d", option);
    }
}

int mx_plan_work(const mx_geom *geom, const mx_iter_desc *desc, int32_t num_sms, int32_t split_keys_opt,
                 int32_t piece_tiles_opt, int32_t pdl, int32_t *items, int32_t max_items, int32_t *decodes,
                 int32_t *counts, char *err_buf, int32_t err_len)
{
    std::string err;
    int rc = MX_OK;
    if (!geom || !desc || !counts || (!items && max_items > 0) || max_items < 0 || num_sms <= 0 ||
        pdl < 0 || pdl > 2 || split_keys_opt < 0 || split_keys_opt > kMaxSplitKeys || split_keys_opt % 128 ||
        piece_tiles_opt < 0 || piece_tiles_opt > 65535)
        rc = fail_to(&err, MX_EINVAL, "null argument or option out of range");
    else if (!geom_ok(*geom))
        rc = fail_to(&err, MX_EINVAL, "unsupported geometry");
    else if ((rc = validate_desc(*geom, desc, false, &err)) == MX_OK && desc->n_decodes > 0 && !decodes)
        rc = fail_to(&err, MX_EINVAL, "decodes is null");
    if (rc == MX_OK) {
        std::vector<DecodeInfo> dec((size_t)std::max(desc->n_decodes, 1));
        std::vector<PrefillInfo> pre(kMaxPrefills);
        std::vector<int4> it((size_t)std::max(max_items, 1));
        const PlanKnobs knobs{num_sms, split_keys_opt, piece_tiles_opt, pdl, max_items};
        WorkList wl;
        rc = build_work_list(*geom, desc, knobs, dec.data(), pre.data(), it.data(), &wl, &err);
        if (rc == MX_OK) {
            if (wl.n_items > 0)
                std::memcpy(items, it.data(), (size_t)wl.n_items * sizeof(int4));
            if (desc->n_decodes > 0)
                std::memcpy(decodes, dec.data(), (size_t)desc->n_decodes * sizeof(DecodeInfo));
            counts[0] = wl.n_items;
            counts[1] = wl.n_prefill;
            counts[2] = wl.split_keys;
            counts[3] = wl.piece_tiles;
            counts[4] = wl.dec_ctas;
        }
    }
    if (rc != MX_OK && err_buf && err_len > 0) {
        const size_t n = std::min<size_t>(err.size(), (size_t)err_len - 1);
        std::memcpy(err_buf, err.data(), n);
        err_buf[n] = '\0';
    }
    return rc;
}

int mx_last_plan(mx_ctx *c, int32_t *n_items, int32_t *split_keys, int32_t *n_prefill_items)
{
    if (!c)
        return MX_EINVAL;
    if (n_items)
        *n_items = c->last_items;
    if (split_keys)
        *split_keys = c->last_split;
    if (n_prefill_items)
        *n_prefill_items = c->last_prefill_items;
    return MX_OK;
}

}  // extern "C"
