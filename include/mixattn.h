/*
 * mixattn — one mixed prefill/decode scheduler iteration on a GB300 (sm_103a).
 *
 * The operation is the one the paper's controller observes (§2.1, Eq. 1):
 * in iteration t, the |D_t| requests that are decoding each bring one new
 * query token, and one prompt receives a prefill chunk of p_t tokens.  All of
 * them run causal GQA softmax attention over a paged bf16 KV cache (§2.1,
 * PagedAttention and chunked prefill; §3.2: attention backend, BF16 precision
 * and KV layout unchanged), and every new token's K/V is appended to its page
 * slot.  The iteration call returns the iteration's device-completion time
 * from CUDA events — the completion-timed signal §6.4 and §9 call for in
 * place of the scheduler-call interval of §3.2.
 *
 * Conventions for every entry point
 *  - Return value: MX_OK (0) or a negative MX_E* code.  Nothing aborts or
 *    traps.  A short text for the last failure of a context is available from
 *    mx_error_detail().
 *  - bf16 tensors are passed as `void *` to 16-bit elements (bf16 bit
 *    patterns); int32 arrays as int32_t *.  "device" pointers must be device
 *    memory of the context's GPU, 16-byte aligned; "host" pointers are read
 *    before the call returns (they may be reused immediately).
 *  - All tensors are owned by the caller.  The context owns only a fixed
 *    workspace allocated by mx_create (work list, split partials, counters,
 *    error word); no call allocates device memory afterwards.
 *  - Enqueueing calls are asynchronous on `stream` (a cudaStream_t, NULL for
 *    the legacy default stream).  One context must not have work in flight on
 *    two streams at once: its workspace is shared by its calls.
 *  - Errors a kernel detects (a page id outside the pool, a slot outside the
 *    pool, an internal wait that timed out) set the context's device error
 *    word; it is read and cleared by mx_iteration() and mx_sync_status().
 *
 * Fixed geometry: head_dim 128, page_size 16, num_q_heads a multiple of
 * num_kv_heads with num_q_heads / num_kv_heads in {1, 2, 4, 8}.
 *
 * Layouts (row-major, bf16):
 *   q, out   [n_tokens][num_q_heads][128]
 *   k, v     [n_tokens][num_kv_heads][128]
 *   k_pool, v_pool  [num_pages][num_kv_heads][16][128]
 *   page_table      int32 [num_seqs][max_pages_per_seq]; entry = physical page
 *   slots           int32 [n_tokens]; slot = page * 16 + offset, < 0: skip
 * Token order in q/k/v/out/slots: the n_decodes decode tokens first (in
 * decode_seq_ids order), then the p_t chunk tokens in position order.
 */
#ifndef MIXATTN_H
#define MIXATTN_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define MX_OK 0
#define MX_EINVAL (-1)      /* bad argument: null pointer, size, geometry   */
#define MX_ERANGE_PAGE (-2) /* a page id outside [0, num_pages)             */
#define MX_ERANGE_SLOT (-3) /* a slot outside [0, num_pages * 16)           */
#define MX_ECUDA (-4)       /* a CUDA runtime/driver call failed            */
#define MX_ETIMEOUT (-5)    /* a bounded in-kernel wait gave up             */
#define MX_EDEVICE (-6)     /* no usable sm_100-family device               */
#define MX_ECAPACITY (-7)   /* request exceeds the context's geometry       */

/* Device error-word bits (reported through the codes above). */
#define MX_ERRBIT_PAGE 1u
#define MX_ERRBIT_SLOT 2u
#define MX_ERRBIT_TIMEOUT 4u

typedef struct mx_ctx mx_ctx;

/* Geometry and capacity of a context.  num_pages is the page count of every
 * pool the context will see; max_tokens bounds n_decodes + p_t per call;
 * max_decodes bounds n_decodes; num_seqs and max_pages_per_seq give the
 * page-table shape. */
typedef struct {
    int32_t num_q_heads;       /* Hq: 16, 32 or 64 in the Qwen3 geometries */
    int32_t num_kv_heads;      /* Hkv: 8 (1..127; Hq / Hkv a power of two
                                  of at most 8)                           */
    int32_t head_dim;          /* must be 128                             */
    int32_t page_size;         /* must be 16                              */
    int32_t num_pages;         /* pages per pool                          */
    int32_t num_seqs;          /* page-table rows                         */
    int32_t max_pages_per_seq; /* page-table row length                   */
    int32_t max_tokens;        /* max n_decodes + p_t per call            */
    int32_t max_decodes;       /* max n_decodes per call                  */
} mx_geom;

/* One prefill chunk: positions [chunk_start, chunk_start + p_t) of the
 * prompt in page-table row seq_id; its row j attends keys [0, chunk_start + j]
 * of that sequence. */
typedef struct {
    int32_t seq_id;       /* page-table row                                 */
    int32_t chunk_start;  /* first position of the chunk                    */
    int32_t p_t;          /* chunk length, >= 1                             */
} mx_prefill;

#define MX_MAX_PREFILLS 16

/* What one iteration schedules (§2.1: the decode set D_t and the prefill
 * budget p_t; §3.1 caps p_t).  decode_seq_ids / decode_ctx_lens are HOST
 * arrays of n_decodes entries: the page-table row of each decoding sequence
 * and the number of tokens it has cached (its new token goes to position
 * ctx; it attends ctx + 1 keys).  prefill_seq_id is the page-table row of the
 * prompt being prefilled (ignored when p_t == 0); its chunk covers positions
 * [chunk_start, chunk_start + p_t) and row j attends keys
 * [0, chunk_start + j].  A sequence takes part at most once per iteration,
 * as one decode or as one prefill chunk (otherwise MX_EINVAL, nothing
 * launched).  page_table and slots are DEVICE arrays. */
typedef struct {
    const int32_t *decode_seq_ids;  /* host  [n_decodes]                  */
    const int32_t *decode_ctx_lens; /* host  [n_decodes]                  */
    int32_t n_decodes;              /* |D_t| >= 0                         */
    int32_t prefill_seq_id;         /* row of page_table, or -1           */
    int32_t chunk_start;            /* first position of the chunk        */
    int32_t p_t;                    /* chunk length, 0 = decode only      */
    const int32_t *page_table;      /* device [num_seqs][max_pages_per_seq] */
    const int32_t *slots;           /* device [n_tokens]                  */
    /* Several chunks (§4.1: the scheduler may admit chunks of several
     * prompts under one token budget): n_prefills > 0 chunks in prefills
     * (a HOST array), used instead of prefill_seq_id / chunk_start / p_t,
     * which must then be -1 / 0 / 0.  At most MX_MAX_PREFILLS; their rows
     * follow the decode tokens chunk after chunk, so n_tokens = n_decodes +
     * the sum of their p_t.  0: the single chunk above (or none). */
    int32_t n_prefills;
    const mx_prefill *prefills;
} mx_iter_desc;

/* Per-layer tensors of one iteration (all DEVICE pointers). */
typedef struct {
    const void *q;  /* [n_tokens][Hq][128]  */
    const void *k;  /* [n_tokens][Hkv][128] */
    const void *v;  /* [n_tokens][Hkv][128] */
    void *k_pool;   /* [num_pages][Hkv][16][128] */
    void *v_pool;   /* [num_pages][Hkv][16][128] */
    void *out;      /* [n_tokens][Hq][128]  */
} mx_layer_bufs;

/* Create a context on CUDA device `device` (made current for the call) and
 * allocate its fixed workspace.  *out receives the context.  Errors:
 * MX_EINVAL (geometry), MX_EDEVICE (not an sm_100-family GPU), MX_ECUDA. */
int mx_create(mx_ctx **out, const mx_geom *geom, int device);

/* Free a context and its workspace (synchronises the device first).
 * NULL is accepted. */
int mx_destroy(mx_ctx *ctx);

/* KV append (§2.1 PagedAttention; §3.2 KV layout unchanged): for each token
 * t < n_tokens with slots[t] >= 0 and every KV head h, copy k[t][h][:] to
 * k_pool[slots[t] / 16][h][slots[t] % 16][:] and likewise for v.  slots is a
 * DEVICE array; the page table enters through it (slot =
 * page_table[seq][pos / 16] * 16 + pos % 16).  Each slot must appear at most
 * once.  Slots beyond the pool are skipped and flag MX_ERRBIT_SLOT.
 * Asynchronous on `stream`. */
int mx_kv_append(mx_ctx *ctx, const int32_t *slots, int32_t n_tokens,
                 const void *k, const void *v, void *k_pool, void *v_pool,
                 void *stream);

/* One layer of the mixed iteration in ONE persistent kernel launch: the KV
 * append of all n_decodes + p_t tokens plus causal paged GQA attention for
 * every query row and head, written to out as bf16.  Decode rows use a
 * split-KV flash-decode with a log-sum-exp merge; chunk rows use tcgen05
 * tensor-core tiles.  Asynchronous on `stream`.  Errors: MX_EINVAL /
 * MX_ECAPACITY (host validation, nothing launched), MX_ECUDA. */
int mx_mixed_attention(mx_ctx *ctx, const mx_iter_desc *desc,
                       const mx_layer_bufs *bufs, void *stream);

/* A whole iteration: the same schedule `desc` run through n_layers layers
 * (layers[l] holds layer l's tensors), one launch per layer, planned once,
 * in order: with MX_OPT_PDL 0 or 1 (the default), layer l+1 reads its
 * tensors only after layer l has completed, so layer l+1's q/k/v may be what
 * layer l wrote (its out, or data derived from it in place).  With
 * MX_OPT_PDL 2 consecutive layers overlap on the GPU and must be independent
 * (distinct tensors; no layer reads what another writes).
 * With device_us_out != NULL: records CUDA events before the first and after
 * the last launch, waits for the second, and stores the elapsed device time in
 * microseconds in *device_us_out (the L_t of Eq. 1 as completed on the
 * device); then reads and clears the device error word and returns
 * MX_ERANGE_PAGE / MX_ERANGE_SLOT / MX_ETIMEOUT if a kernel flagged one (the
 * time is still stored).  With device_us_out == NULL: only enqueues the
 * launches on `stream` and returns (errors via mx_sync_status). */
int mx_iteration(mx_ctx *ctx, const mx_iter_desc *desc, int32_t n_layers,
                 const mx_layer_bufs *layers, float *device_us_out,
                 void *stream);

/* mx_iteration replayed from a CUDA graph (the paper runs its iterations
 * under CUDA graphs, §4.1): the plan upload and the n_layers launches are
 * captured once into a graph, and each call only writes the new plan into
 * the context's replay slot and launches the graph, so the host cost per
 * call does not grow with n_layers.  The launches read the plan's counts
 * from device memory, and their TMA descriptors span the buffers'
 * capacity: each layer's q, k, v and out must hold max_tokens rows of the
 * context (rows past the call's tokens are read but do not affect the
 * results).  The graph is captured again when any of layers[0..n_layers),
 * desc's page_table or slots pointer, MX_OPT_GRID, MX_OPT_PDL,
 * MX_OPT_WAIT_LIMIT_US or MX_OPT_TEST_STALL_BLOCK differs from the last
 * capture (one graph is kept per value-ring depth, see MX_OPT_V_STAGES); the
 * capture happens inside this call, on a stream of the context, and is
 * not itself capturable.  A call waits until the previous replay has read
 * its plan.  Results are identical to mx_iteration's; device_us_out, the
 * error word and the return codes as for mx_iteration. */
int mx_iteration_graph(mx_ctx *ctx, const mx_iter_desc *desc, int32_t n_layers,
                       const mx_layer_bufs *layers, float *device_us_out,
                       void *stream);

/* Wait for `stream`, then read and clear the device error word. */
int mx_sync_status(mx_ctx *ctx, void *stream);

/* Copy a NUL-terminated description of the context's last failure into buf
 * (at most len bytes).  With ctx == NULL: why the calling thread's last
 * mx_create failed (empty after a successful one).  Returns the length
 * written, or MX_EINVAL (buf NULL or len <= 0). */
int mx_error_detail(mx_ctx *ctx, char *buf, int32_t len);

/* Tunables.  MX_OPT_SPLIT_KEYS: keys per decode split (multiple of 128,
 * 0 = automatic).  MX_OPT_GRID: persistent grid size (0 = number of SMs).
 * MX_OPT_PREFILL_PIECE_TILES: at most this many 128-key tiles per prefill
 * work item; longer causal tiles are split into pieces merged by
 * log-sum-exp (0 = automatic, 65535 = never split).  A prompt's first query
 * tile at chunk_start < 16 is never split (its rows of at most 16 keys are
 * recomputed exactly from the tiles the item holds); the size doubles while
 * the pieces' partials would not fit the context's workspace. */
#define MX_OPT_SPLIT_KEYS 1
#define MX_OPT_GRID 2
#define MX_OPT_PREFILL_PIECE_TILES 3
/* MX_OPT_PDL: how the layer launches of mx_iteration follow each other.
 * 1 (default): programmatic dependent launch hides the launch latency; each
 * CTA of layer l+1 waits (griddepcontrol.wait) until layer l has completed
 * and its writes are visible before it reads anything: the order of a model
 * whose layer l+1 attention reads what layer l produced.  2: the layers are
 * independent problems; layer l+1's CTAs start on the SMs layer l frees,
 * filling layer l's tail (needs a grid of every SM, else behaves as 1).
 * 0: ordinary stream order.  Consecutive launches use three workspace sets
 * in turn. */
#define MX_OPT_PDL 4
/* MX_OPT_WAIT_LIMIT_US: bound on every in-kernel wait, in microseconds
 * (0 = the default, one second); a wait that reaches it ends the launch with
 * MX_ETIMEOUT.  MX_OPT_TEST_STALL_BLOCK (fault injection, 0 = off): with
 * value b > 0, block b - 1 of every later launch claims its first work item
 * and then waits on a barrier that nothing arrives at, so the launch reports
 * MX_ETIMEOUT after the wait limit with that item undone.  After any
 * reported error the context clears its counters and stays usable. */
#define MX_OPT_WAIT_LIMIT_US 5
#define MX_OPT_TEST_STALL_BLOCK 6
/* MX_OPT_V_STAGES: depth of the value-tile ring of prefill items, 2 or 3
 * (0 = automatic: 3 when the launch's prefill tensor work in flops is at
 * least 150 times its decode key/value bytes, else 2).  Three stages hide
 * the value loads of long prefill items but take 224 KiB of shared memory
 * per SM instead of 192, and the smaller L1 slows decode-heavy launches.
 * Results are the same either way. */
#define MX_OPT_V_STAGES 7
/* MX_OPT_DECODE_CTAS: how many CTAs of a launch with both prefill and decode
 * items start on the decode items (the others start on the prefill items,
 * and each CTA turns to the other kind once its own runs out), so that
 * decode splits stream from HBM on some SMs while prefill tiles occupy the
 * tensor cores of the rest.  0 = automatic (the decode's share of the
 * launch's time at the HBM and tensor rates), -1 = none (every CTA takes
 * prefill items first), k = the first k CTAs (at most 65535).  Results are
 * the same for every value. */
#define MX_OPT_DECODE_CTAS 8
int mx_set_option(mx_ctx *ctx, int32_t option, int64_t value);

/* Number of work items and decode split length chosen for the last planned
 * call (for reporting). */
int mx_last_plan(mx_ctx *ctx, int32_t *n_items, int32_t *split_keys,
                 int32_t *n_prefill_items);

/* The work list of one layer launch, computed on the host without a device
 * (the planning step of mx_mixed_attention / mx_iteration, exposed so that
 * schedulers and tests can inspect it).  The paper schedules per iteration a
 * decode set D_t and a prefill chunk of p_t tokens (§2.1, Eq. 1); one launch
 * splits that work into items in two queues that its persistent CTAs claim
 * from: prefill query tiles (128 rows x two query heads of one KV head, or
 * one head when num_q_heads == num_kv_heads; or a key piece of one),
 * heaviest first, and decode splits (one decode x one KV head x a key
 * range), longest first.  The first counts[4] CTAs start on the decode
 * queue, the others on the prefill queue; each turns to the other queue
 * when its own is empty (MX_OPT_DECODE_CTAS).
 *
 * geom and desc as for mx_create / mx_mixed_attention (desc's page_table and
 * slots are not read and may be NULL); num_sms: the SM count the launch will
 * use; split_keys_opt, piece_tiles_opt, pdl: the values of MX_OPT_SPLIT_KEYS,
 * MX_OPT_PREFILL_PIECE_TILES and MX_OPT_PDL (0, 0 and 1 are the defaults).
 * Outputs (host arrays owned by the caller):
 *   items    int32 [max_items][4], n_items records in claim order:
 *     prefill {f << 4 | (heads - 1) << 8, t | hq << 16, s | n_s << 16,
 *       partial slot base}: piece s of n_s of query tile t (rows
 *       [128 t, 128 t + 128) of prefill chunk f, in the order of
 *       desc->prefills, or 0 for the single chunk) of query heads hq ..
 *       hq + heads - 1 (heads 1 or 2); the tile's n_T =
 *       ceil(chunk_start_f / 128) + t + 1 key tiles (128 keys each) are split
 *       as [s n_T / n_s, (s + 1) n_T / n_s); head e of piece s writes partial
 *       slot base + e n_s + s when n_s > 1;
 *     decode {1 | h << 4 | s << 11 | (len / 16) << 23, decode index i,
 *       page-table row, cached tokens ctx}: split s of decode i, KV head h,
 *       keys [s len, min((s + 1) len, ctx + 1)); kind 2 instead of 1 for a
 *       decode of at most 64 keys (one split, computed exactly in fp32);
 *   decodes  int32 [n_decodes][4]: page-table row, ctx, number of splits,
 *     first partial slot (of head 0; head h uses base + h * splits);
 *   counts   int32 [5]: n_items, prefill items (items [0, prefill items)
 *     are the prefill queue, the rest the decode queue), split_keys,
 *     piece_tiles, CTAs that start on the decode queue (the automatic
 *     choice of MX_OPT_DECODE_CTAS for a grid of num_sms).
 * Returns MX_OK, MX_EINVAL (arguments, geometry, descriptor) or MX_ECAPACITY
 * (the work does not fit max_items or the context's partial workspace), with
 * a message in err_buf (up to err_len bytes) when err_buf is not NULL. */
int mx_plan_work(const mx_geom *geom, const mx_iter_desc *desc, int32_t num_sms,
                 int32_t split_keys_opt, int32_t piece_tiles_opt, int32_t pdl,
                 int32_t *items, int32_t max_items, int32_t *decodes,
                 int32_t *counts, char *err_buf, int32_t err_len);

/* For callers that cannot allocate device memory (a host framework whose
 * allocator owns the GPU, a plug-in with a fixed pre-reserved budget, a path
 * that must not risk an allocation's implicit synchronisation or OOM).  The
 * paper has no counterpart: this is a deployment variant of
 * mx_mixed_attention that needs no context, because mx_create allocates.
 *
 * Same operation, layouts and descriptor as mx_mixed_attention (geom gives
 * the geometry a context would hold; max_tokens / max_decodes are ignored),
 * for at most one prefill chunk (desc->n_prefills must be 0).
 * Its scratch (work list, split partials, counters, error word) is one fixed
 * 4.11 MiB device array built into the library, which every GPU that loads
 * the library holds until the process exits.  Limits: n_decodes <= 256,
 * at most 4096 work items (prefill tiles = ceil(p_t / 128) * Hq, plus decode
 * splits), at most 1024 split partials, num_kv_heads <= 16; a request beyond
 * them returns MX_ECAPACITY and enqueues nothing.
 *
 * The call allocates nothing (no cudaMalloc/cudaFree, no allocating library
 * routine).  The first call on a device does a one-time set-up (it resolves
 * the array's device address and the kernel attributes), so make that first
 * call before any stream capture.  Each call zeroes the counters it needs,
 * uploads its work list, launches, waits for `stream`, and reads the error
 * word, so it returns MX_ERANGE_PAGE / MX_ERANGE_SLOT / MX_ETIMEOUT like
 * mx_iteration.  All calls on a GPU share the one array: calls whose GPU work
 * overlaps (other streams, other host threads) race and must be serialised
 * by the caller.  On failure a message is written to err_buf (up to err_len
 * bytes) when err_buf is not NULL. */
int mx_mixed_attention_noalloc(const mx_geom *geom, const mx_iter_desc *desc,
                               const mx_layer_bufs *bufs, void *stream,
                               char *err_buf, int32_t err_len);

/* ------------------------------------------------------------------------
 * The rest of a Qwen3 decoder layer around mx_mixed_attention (the
 * whole-model setting of the paper's measurements, §4.1; it sets the share
 * of L_prefill in Eq. 1's L_t).  Context-free: device pointers to row-major
 * bf16 tensors (16-byte aligned unless stated), asynchronous on `stream`.
 * Return MX_OK, MX_EINVAL (arguments; nothing launched) or MX_ECUDA. */

/* y[r] = x[r] / sqrt(mean(x[r]^2) + eps) * w for rows x [rows][dim], w
 * [dim] (dim a multiple of 8); y may be x. */
int mx_rms_norm(const void *x, const void *w, void *y, int32_t rows,
                int32_t dim, float eps, void *stream);

/* From the fused projection qkv [n_tokens][num_q_heads + 2 num_kv_heads][128]
 * (q heads, then k heads, then v heads): q [n_tokens][num_q_heads][128] and
 * k [n_tokens][num_kv_heads][128] = the rotary embedding at the token's
 * position (positions [n_tokens], int32) of the head's RMSNorm over its 128
 * elements (weights q_norm / k_norm [128]); rotate-half pairing, element i
 * with i + 64 at frequency theta^(-i/64); v [n_tokens][num_kv_heads][128] =
 * the v heads.  The outputs are the attention inputs (mx_layer_bufs q, k,
 * v); pointers 8-byte aligned. */
int mx_qk_norm_rope(const void *qkv, const void *q_norm, const void *k_norm,
                    const int32_t *positions, void *q, void *k, void *v,
                    int32_t n_tokens, int32_t num_q_heads,
                    int32_t num_kv_heads, float theta, float eps,
                    void *stream);

/* SwiGLU gate: y[r][j] = silu(gu[r][j]) * gu[r][d_ffn + j] for gate_up
 * [rows][2 d_ffn] (gate, then up), y [rows][d_ffn], d_ffn a multiple of 8. */
int mx_silu_mul(const void *gate_up, void *y, int32_t rows, int32_t d_ffn,
                void *stream);

/* c [m][n] = a [m][k] b [k][n] (+ c when accumulate = 1, e.g. a residual
 * add), bf16 in and out, fp32 accumulation (a cuBLAS GEMM). */
int mx_gemm(const void *a, const void *b, void *c, int32_t m, int32_t n,
            int32_t k, int32_t accumulate, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* MIXATTN_H */
