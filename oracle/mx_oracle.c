/*
 * Reference oracle for the mixed prefill/decode iteration — TEST
 * INFRASTRUCTURE ONLY.  Plain, slow, float64 C.  Only the test suite,
 * __graft_entry__.smoke() and bench.py's CPU-baseline leg load this file's
 * library; the product path never does.  It shares no code, header or
 * constant with the CUDA library.
 *
 * What it computes follows the paper's problem statement:
 *  - §2.1 (Eq. 1 and the paragraph before it): one scheduler iteration t
 *    carries the set D_t of decoding requests (one new token each) and p_t
 *    prompt tokens admitted for prefill; every decoder waits for the whole
 *    iteration.
 *  - §2.1 (PagedAttention, chunked prefill): the KV cache is paged and a long
 *    prompt is prefilled chunk by chunk, so chunk row j of a chunk starting at
 *    position chunk_start sits at absolute position chunk_start + j.
 *  - §3.2: attention backend, precision (BF16) and KV layout are unchanged by
 *    the controller, i.e. the computation is ordinary causal softmax
 *    attention, and §4.3/§5.1 require outputs to agree exactly with and
 *    without chunking.
 *
 * Readings where the paper is silent:
 *  - softmax scale 1/sqrt(head_dim);
 *  - GQA: query head h reads KV head h / (Hq/Hkv);
 *  - a decode with ctx cached tokens attends ctx + 1 keys (its own new key);
 *  - chunk row j attends keys [0, chunk_start + j] (bottom-right causal);
 *  - the append is applied before attention, so new keys are read back from
 *    the pages they were written to.
 *
 * Every floating-point step is the textbook definition: scores in float64,
 * a max-subtracted exponential, a plain sum, a division.  No blocking, no
 * online softmax, no reordering.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define ORC_OK 0
#define ORC_EINVAL (-1)
#define ORC_ERANGE (-2)

/* bf16 bit pattern -> exact double (bf16 is the top half of an IEEE float) */
static double bf16_bits_to_double(uint16_t b)
{
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * KV append (§2.1 PagedAttention; §3.2 "KV layout unchanged"): token t's key
 * and value for every KV head go to physical slot slots[t], i.e. page
 * slots[t] / page_size, offset slots[t] % page_size.  slot < 0 means "skip".
 * Pools are [num_pages][hkv][page_size][head_dim] bf16 bit patterns; k and v
 * are [n_tokens][hkv][head_dim].  A pure byte copy.
 */
int oracle_kv_append(uint16_t *k_pool, uint16_t *v_pool, int64_t num_pages,
                     int hkv, int page_size, int head_dim,
                     const int32_t *slots, int n_tokens,
                     const uint16_t *k, const uint16_t *v)
{
    if (!k_pool || !v_pool || !slots || (n_tokens > 0 && (!k || !v)))
        return ORC_EINVAL;
    for (int t = 0; t < n_tokens; ++t) {
        int64_t slot = slots[t];
        if (slot < 0)
            continue;
        int64_t page = slot / page_size, off = slot % page_size;
        if (page >= num_pages)
            return ORC_ERANGE;
        for (int h = 0; h < hkv; ++h) {
            size_t dst = (((size_t)page * hkv + h) * page_size + off) * head_dim;
            size_t src = ((size_t)t * hkv + h) * head_dim;
            memcpy(k_pool + dst, k + src, sizeof(uint16_t) * head_dim);
            memcpy(v_pool + dst, v + src, sizeof(uint16_t) * head_dim);
        }
    }
    return ORC_OK;
}

/*
 * Softmax attention of one query vector over the first n_keys logical
 * positions of one sequence, gathered through its page-table row in logical
 * order.  Writes out[head_dim] and the natural-log sum-exp of the scaled
 * scores.  scores[] is caller scratch of n_keys doubles.
 */
static int attend_one(const uint16_t *qv, int n_keys, const int32_t *pt_row,
                      int max_pages, int64_t num_pages, int kvh, int hkv,
                      int page_size, int head_dim, const uint16_t *k_pool,
                      const uint16_t *v_pool, double *scores, double *out,
                      double *lse)
{
    const double scale = 1.0 / sqrt((double)head_dim);
    double m = -INFINITY;
    for (int kp = 0; kp < n_keys; ++kp) {
        int lp = kp / page_size;
        if (lp >= max_pages)
            return ORC_ERANGE;
        int64_t page = pt_row[lp];
        if (page < 0 || page >= num_pages)
            return ORC_ERANGE;
        const uint16_t *kr = k_pool +
            (((size_t)page * hkv + kvh) * page_size + kp % page_size) * head_dim;
        double s = 0.0;
        for (int d = 0; d < head_dim; ++d)
            s += bf16_bits_to_double(qv[d]) * bf16_bits_to_double(kr[d]);
        s *= scale;
        scores[kp] = s;
        if (s > m)
            m = s;
    }
    double denom = 0.0;
    for (int kp = 0; kp < n_keys; ++kp) {
        scores[kp] = exp(scores[kp] - m);
        denom += scores[kp];
    }
    for (int d = 0; d < head_dim; ++d)
        out[d] = 0.0;
    for (int kp = 0; kp < n_keys; ++kp) {
        int64_t page = pt_row[kp / page_size];
        const uint16_t *vr = v_pool +
            (((size_t)page * hkv + kvh) * page_size + kp % page_size) * head_dim;
        double w = scores[kp] / denom;
        for (int d = 0; d < head_dim; ++d)
            out[d] += w * bf16_bits_to_double(vr[d]);
    }
    *lse = m + log(denom);
    return ORC_OK;
}

/*
 * One layer of the mixed iteration (§2.1): |D_t| = n_decodes decode queries
 * and n_prefills prefill chunks; chunk j has p_ts[j] rows of sequence
 * prefill_seqs[j] starting at position chunk_starts[j] (one chunk is the
 * paper's setting; §4.1's scheduler may admit the chunks of several prompts
 * under one token budget, each still a chunk of its own sequence).  Token
 * order in q/k/v/slots: the decodes first, then chunk 0's rows, chunk 1's, ...
 *
 * Step 1 applies the append of all n_decodes + p_t tokens to the pools (which
 * the caller passes as its own host copies; they are modified).  Step 2
 * computes attention for the requested token rows (rows == NULL: all rows)
 * and every query head, writing out[r][hq][head_dim] and lse[r][hq].
 *
 * scratch must hold max_keys doubles per OpenMP thread, where max_keys is the
 * largest n_keys of any requested row; the caller sizes it.
 */
int oracle_mixed_attention(int hq, int hkv, int head_dim, int page_size,
                           int64_t num_pages, int max_pages,
                           const int32_t *decode_seq_ids,
                           const int32_t *decode_ctx_lens, int n_decodes,
                           const int32_t *prefill_seqs, const int32_t *chunk_starts,
                           const int32_t *p_ts, int n_prefills,
                           const int32_t *page_table, const int32_t *slots,
                           const uint16_t *q, const uint16_t *k,
                           const uint16_t *v, uint16_t *k_pool,
                           uint16_t *v_pool, const int32_t *rows, int n_rows,
                           double *out, double *lse, double *scratch,
                           int64_t scratch_per_thread)
{
    if (hq <= 0 || hkv <= 0 || hq % hkv != 0 || head_dim <= 0 ||
        page_size <= 0 || n_decodes < 0 || n_prefills < 0)
        return ORC_EINVAL;
    int n_tok = n_decodes;
    for (int j = 0; j < n_prefills; ++j) {
        if (p_ts[j] < 0 || chunk_starts[j] < 0)
            return ORC_EINVAL;
        n_tok += p_ts[j];
    }
    int rc = oracle_kv_append(k_pool, v_pool, num_pages, hkv, page_size,
                              head_dim, slots, n_tok, k, v);
    if (rc != ORC_OK)
        return rc;
    int n_rep = hq / hkv;
    int nr = rows ? n_rows : n_tok;
    int err = ORC_OK;
#pragma omp parallel for schedule(dynamic) reduction(min : err)
    for (int64_t w = 0; w < (int64_t)nr * hq; ++w) {
        int ri = (int)(w / hq), h = (int)(w % hq);
        int r = rows ? rows[ri] : ri;
        int seq, n_keys;
        if (r < 0 || r >= n_tok) {
            err = ORC_EINVAL;
            continue;
        }
        if (r < n_decodes) {
            seq = decode_seq_ids[r];
            n_keys = decode_ctx_lens[r] + 1;
        } else {
            /* the chunk holding token r, and r's row within it */
            int j = 0, row = r - n_decodes;
            while (row >= p_ts[j]) {
                row -= p_ts[j];
                ++j;
            }
            seq = prefill_seqs[j];
            n_keys = chunk_starts[j] + row + 1;
        }
        if (n_keys > scratch_per_thread) {
            err = ORC_EINVAL;
            continue;
        }
#ifdef _OPENMP
        extern int omp_get_thread_num(void);
        double *sc = scratch + (int64_t)omp_get_thread_num() * scratch_per_thread;
#else
        double *sc = scratch;
#endif
        int e = attend_one(q + ((size_t)r * hq + h) * head_dim, n_keys,
                           page_table + (size_t)seq * max_pages, max_pages,
                           num_pages, h / n_rep, hkv, page_size, head_dim,
                           k_pool, v_pool, sc,
                           out + ((size_t)ri * hq + h) * head_dim,
                           lse + (size_t)ri * hq + h);
        if (e < err)
            err = e;
    }
    return err;
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}
