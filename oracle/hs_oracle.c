/*
 * hs_oracle.c -- float64 CPU oracle for checkpoint-aligned restore-and-resume.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library (paper_2609_15030_gb300)
 * links, loads or calls this file; only tests/, the smoke check and the CPU
 * baseline leg of bench.py do.  It shares no code, header or constant with
 * the CUDA path.
 *
 * Every routine is the plain definition, written for a reader to check by
 * eye against the paper:
 *   - oracle_align_prefix:     Section 2.2 (B = C*floor((N-1)/C) on a complete
 *                              hit; in general the largest available
 *                              checkpoint inside the strict-prefix query) and
 *                              Section 3.2 (the query excludes the last known
 *                              token), by brute-force scan.
 *   - oracle_align_prerepair:  the faulty pre-repair behaviour of Section 3.2
 *                              (B from the full prompt, credit p = N-1 on an
 *                              exact boundary); a negative fixture.
 *   - oracle_scatter_pages:    restoring the attention cache entries of
 *                              [0,B) page by page (Section 2.1, Section 5.2),
 *                              as memcpy.
 *   - oracle_gather_pages:     saving cache pages into a staging pool by block
 *                              table (the save path of Section 3.1 and the
 *                              D2H comparisons of Table 5), as memcpy.
 *   - oracle_scatter_slices / oracle_gather_slices: the same for one tensor-
 *                              parallel rank's bytes of every page row (Table 1:
 *                              TP=4; Section 5.2: per-rank transfers), as memcpy.
 *   - oracle_copy_slots:       restoring / snapshotting the recurrent state
 *                              (Section 1: state updated in place must be
 *                              restored, not recounted), as memcpy.
 *   - oracle_gla_head:         the gated linear-attention recurrence
 *                              S_t = diag(g_t) S_{t-1} + k_t v_t^T,
 *                              o_t = q_t S_t  (row vector times matrix),
 *                              g_t = exp(a_t), token by token in float64,
 *                              from the state of prefix [0,pos0)
 *                              (Section 2.2: a state for [0,B) continues
 *                              from B).  The paper names the FLA kernels but
 *                              never prints the recurrence; this form is the
 *                              one the library implements.  Checkpoints are
 *                              the state after a prefix whose length is a
 *                              multiple of C (Table 1: C = 1,792).
 *   - oracle_restore_bytes:    bytes moved by one restore (pages + states).
 *
 * Inputs are the exact quantised values the GPU consumes: bf16 bit patterns
 * widened to double, float32 log-gates widened to double.
 */
#include <stdint.h>
#include <string.h>
#include <math.h>

static double bf16_to_double(uint16_t b)
{
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Is b one of the n_avail available checkpoint positions? (linear search) */
static int is_available(int64_t b, const int64_t *avail, int32_t n_avail)
{
    if (b == 0)
        return 1;                 /* the empty prefix (zero state) always exists */
    for (int32_t i = 0; i < n_avail; ++i)
        if (avail[i] == b)
            return 1;
    return 0;
}

/*
 * Strict-prefix alignment by brute force.  The lookup query is the prompt
 * without its last token, further limited to the cached prefix hit_len, so
 * the chosen c satisfies c <= N-1 and c <= hit_len.  Scan b = N-1 .. 0 and
 * return the first b that is available and page aligned.
 * Returns 0, or -1 for invalid arguments.
 */
int oracle_align_prefix(int64_t N, int64_t hit_len, const int64_t *avail, int32_t n_avail,
                        int32_t page_size, int64_t *c_out, int64_t *n_pages_out,
                        int64_t *tail_out)
{
    if (N < 1 || hit_len < 0 || hit_len > N || page_size < 1 || n_avail < 0)
        return -1;
    int64_t c = 0;
    for (int64_t b = N - 1; b >= 0; --b) {
        if (b > hit_len)
            continue;
        if (b % page_size != 0)
            continue;
        if (!is_available(b, avail, n_avail))
            continue;
        c = b;
        break;
    }
    *c_out = c;
    *n_pages_out = c / page_size;
    *tail_out = N - c;
    return 0;
}

/*
 * The faulty pre-repair connector of Section 3.2: checkpoint selection used
 * the full prompt (B = C*floor(N/C)), while a later complete-prompt branch
 * credited the scheduler with one fewer token when B reached N.
 */
void oracle_align_prerepair(int64_t N, int64_t C, int64_t *B_out, int64_t *p_out)
{
    int64_t B = C * (N / C);
    *B_out = B;
    *p_out = (B == N) ? N - 1 : B;
}

/* cache_l[bt[j]] <- staging_l[j] for every layer l and page j < n_pages. */
void oracle_scatter_pages(const uint8_t *const *staging, uint8_t *const *cache, int32_t n_layers,
                          const int32_t *bt, int32_t n_pages, int64_t page_bytes)
{
    for (int32_t l = 0; l < n_layers; ++l)
        for (int32_t j = 0; j < n_pages; ++j)
            memcpy(cache[l] + (int64_t)bt[j] * page_bytes,
                   staging[l] + (int64_t)j * page_bytes, (size_t)page_bytes);
}

/* staging_l[j] <- cache_l[bt[j]] for every layer l and page j < n_pages. */
void oracle_gather_pages(const uint8_t *const *cache, uint8_t *const *staging, int32_t n_layers,
                         const int32_t *bt, int32_t n_pages, int64_t page_bytes)
{
    for (int32_t l = 0; l < n_layers; ++l)
        for (int32_t j = 0; j < n_pages; ++j)
            memcpy(staging[l] + (int64_t)j * page_bytes,
                   cache[l] + (int64_t)bt[j] * page_bytes, (size_t)page_bytes);
}

/* For every layer l, page j, row r < rows of row_bytes = page_bytes/rows:
 * bytes [col_off, col_off+col_bytes) of row r of cache_l[bt[j]] and the packed
 * staging row staging_l[(j*rows + r)*col_bytes ...]; gather != 0 copies cache to
 * staging, else staging to cache. */
void oracle_slices(int32_t gather, uint8_t *const *staging, uint8_t *const *cache, int32_t n_layers,
                   const int32_t *bt, int32_t n_pages, int64_t page_bytes, int32_t rows,
                   int64_t col_off, int64_t col_bytes)
{
    const int64_t row_bytes = page_bytes / rows;
    for (int32_t l = 0; l < n_layers; ++l)
        for (int32_t j = 0; j < n_pages; ++j)
            for (int32_t r = 0; r < rows; ++r) {
                uint8_t *c = cache[l] + (int64_t)bt[j] * page_bytes + r * row_bytes + col_off;
                uint8_t *s = staging[l] + ((int64_t)j * rows + r) * col_bytes;
                if (gather)
                    memcpy(s, c, (size_t)col_bytes);
                else
                    memcpy(c, s, (size_t)col_bytes);
            }
}

/* dst[i] <- src[i], n slots of floats_each float32 values. */
void oracle_copy_slots(const float *const *src, float *const *dst, int32_t n, int64_t floats_each)
{
    for (int32_t i = 0; i < n; ++i)
        memcpy(dst[i], src[i], (size_t)floats_each * sizeof(float));
}

/* Bytes moved by one restore: whole KV pages of every full-attention layer
 * plus one float32 state per linear layer and head. */
int64_t oracle_restore_bytes(int64_t n_full_layers, int64_t n_pages, int64_t page_bytes,
                             int64_t n_lin_layers, int64_t n_heads, int64_t d_k, int64_t d_v)
{
    return n_full_layers * n_pages * page_bytes + n_lin_layers * n_heads * d_k * d_v * 4;
}

/*
 * One head of one request, token by token.
 *   q, k : bf16 bits, token t at q + t*qk_stride, d_k values
 *   v    : bf16 bits, token t at v + t*v_stride,  d_v values
 *   a    : float32 log-gates, token t at a + t*a_stride, d_k values
 *   S    : double [d_k][d_v], in: state of prefix [0,pos0), out: of [0,pos0+n)
 *   o    : double, token t at o + t*o_stride, d_v values
 *   ckpts: if not NULL, receives S (double [d_k][d_v]) after every prefix
 *          length that is a positive multiple of C, in order.
 * Returns the number of checkpoints written.
 */
int64_t oracle_gla_head(int64_t n, int32_t d_k, int32_t d_v,
                        const uint16_t *q, const uint16_t *k, int64_t qk_stride,
                        const uint16_t *v, int64_t v_stride,
                        const float *a, int64_t a_stride,
                        double *S, double *o, int64_t o_stride,
                        int64_t pos0, int64_t C, double *ckpts)
{
    int64_t n_ck = 0;
    for (int64_t t = 0; t < n; ++t) {
        const uint16_t *qt = q + t * qk_stride;
        const uint16_t *kt = k + t * qk_stride;
        const uint16_t *vt = v + t * v_stride;
        const float *at = a + t * a_stride;
        /* S_t = diag(g_t) S_{t-1} + k_t v_t^T */
        for (int32_t i = 0; i < d_k; ++i) {
            double g = exp((double)at[i]);
            double ki = bf16_to_double(kt[i]);
            for (int32_t j = 0; j < d_v; ++j)
                S[i * d_v + j] = g * S[i * d_v + j] + ki * bf16_to_double(vt[j]);
        }
        /* o_t = q_t S_t */
        double *ot = o + t * o_stride;
        for (int32_t j = 0; j < d_v; ++j) {
            double acc = 0.0;
            for (int32_t i = 0; i < d_k; ++i)
                acc += bf16_to_double(qt[i]) * S[i * d_v + j];
            ot[j] = acc;
        }
        /* checkpoint: the state of prefix [0, pos0+t+1) when that length is a multiple of C */
        if (ckpts != NULL && C > 0 && (pos0 + t + 1) % C == 0) {
            memcpy(ckpts + n_ck * (int64_t)d_k * d_v, S, sizeof(double) * (size_t)d_k * d_v);
            ++n_ck;
        }
    }
    return n_ck;
}
