/*
 * hs.h -- checkpoint-aligned restore-and-resume for hybrid (full-attention +
 * linear-attention) language models on one GB300 (sm_103a).
 *
 * The calls follow one resumed request:
 *   1. hs_align_prefix                 strict-prefix lookup: pick the recurrent-state
 *                                      checkpoint c the scheduler may credit (host).
 *   2. hs_restore_kv_pages             scatter the cached KV pages of [0,c) from a device
 *                                      staging pool into the paged KV cache by block table.
 *   3. hs_restore_state                copy the float32 linear-attention state at c into the
 *                                      live state.
 *   4. hs_linattn_prefill_from_state   gated linear-attention prefill over the tail [c,N)
 *                                      from that state, emitting state checkpoints.
 *   5. hs_checkpoint_states            snapshot live states into checkpoint slots.
 *   6. hs_save_kv_pages                gather cache pages by block table into a staging
 *                                      pool (the save path; device or pinned host memory).
 *   hs_restore_kv_page_slices / hs_save_kv_page_slices: the same for one tensor-parallel
 *                                      rank's heads of every page.
 *
 * Conventions shared by every call
 *   - Every call returns hs_status.  HS_OK means the arguments passed host-side
 *     validation and the work was enqueued; it does not wait for the GPU.
 *   - The caller owns all memory.  The library never allocates or frees memory,
 *     never synchronises a stream and keeps no mutable global state.
 *   - "device" pointers point to GPU-visible memory of the current device; "host"
 *     pointers are read by the host before the call returns.
 *   - GPU work is enqueued on the caller's stream in argument order; calls on one
 *     stream execute in issue order.
 *   - Problems that only the GPU can see (a block id out of range, a misaligned
 *     pointer read from a device pointer array, a bounded wait that ran out) are
 *     reported through the optional device word d_err: the first kernel that
 *     detects one stores an HS_DEVERR_* code there if it still holds 0.  Kernels
 *     never clear it and never trap; the work item that failed is skipped.
 *     Pass NULL to skip reporting.
 *
 * Data types: "bf16" arrays hold bfloat16 bit patterns (uint16_t); float is IEEE
 * binary32.
 */
#ifndef HS_H
#define HS_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum hs_status {
    HS_OK = 0,
    HS_ERR_INVALID_ARG = 1,   /* null pointer, negative or inconsistent size, unsorted list */
    HS_ERR_MISALIGNED = 2,    /* pointer or byte size not a multiple of 16 bytes */
    HS_ERR_UNSUPPORTED = 3,   /* shape outside what the kernels implement (see each call) */
    HS_ERR_CUDA = 4,          /* a CUDA runtime call or launch failed */
    HS_ERR_DEVICE_CHECK = 5,  /* reserved for callers that fold d_err into a status */
    HS_ERR_TOO_LARGE = 6      /* the call needs more than the library's fixed workspace
                                 (HS_NOALLOC_SCRATCH_BYTES) holds */
} hs_status;

/* codes a kernel may store into d_err */
#define HS_DEVERR_NONE 0
#define HS_DEVERR_BLOCK_OOB 1     /* block_table entry < 0 or >= num_blocks */
#define HS_DEVERR_MISALIGNED 2    /* a pointer read from a device pointer array is not 16-byte aligned */
#define HS_DEVERR_NULL 3          /* a pointer read from a device pointer array is NULL */
#define HS_DEVERR_TIMEOUT 4       /* a bounded wait inside a kernel ran out */

/* Largest batch accepted by hs_linattn_prefill_from_state. */
#define HS_MAX_BATCH 384
/* Chunk length of the prefill; checkpoint intervals are multiples of it. */
#define HS_CHUNK 64
/* Segments (the part of a call inside one chunk) of at most this many tokens are
 * computed token by token, with the same arithmetic in every kernel. */
#define HS_SHORT_SEGMENT 8

/* Human-readable name of a status; never NULL. */
const char *hs_status_string(hs_status s);

/* Library version, major*10000 + minor*100 + patch. */
int32_t hs_version(void);

/*
 * hs_align_prefix -- strict-prefix checkpoint alignment (host only, no GPU).
 *
 * Paper: Section 2.2 (a state for prefix [0,B) continues from B, so the
 * scheduler credits p = B; on a complete hit with every checkpoint cached,
 * B = C*floor((N-1)/C)), Section 3.2 (the lookup query excludes the last known
 * token, so a complete hit never credits N) and Table 4 / Figure 2.
 *
 * Chooses c = the largest b with b <= N-1, b <= hit_len, b % page_size == 0 and b
 * either 0 (the empty prefix, always available) or listed in avail_ckpts.
 *   N            prompt length in tokens, >= 1
 *   hit_len      tokens of the prompt found in the external cache, 0 <= hit_len <= N
 *   avail_ckpts  host, n_avail checkpoint positions (prefix lengths) held in the
 *                cache, strictly increasing, each >= 0; entries above N are
 *                ignored; may be NULL when n_avail == 0
 *   page_size    KV page size in tokens, >= 1
 *   c_out        host: the aligned checkpoint c (the scheduler credit p = c)
 *   n_pages_out  host: c / page_size, the KV pages to restore per full layer
 *   tail_out     host: N - c >= 1, tokens to recompute
 * Errors: HS_ERR_INVALID_ARG (sizes, NULL outputs, unsorted or negative list).
 */
hs_status hs_align_prefix(int64_t N, int64_t hit_len, const int64_t *avail_ckpts, int32_t n_avail,
                          int32_t page_size, int64_t *c_out, int64_t *n_pages_out,
                          int64_t *tail_out);

/*
 * hs_restore_kv_pages -- scatter cached KV pages into the paged KV cache.
 *
 * Paper: Section 2.1 (attention cache entries travel with the checkpointed
 * state), Section 5.2 (restored bytes per rank follow the chosen B) and
 * Table 5 (H2D page transfers into poisoned destinations).
 *
 * For every layer l < n_layers and page j < n_pages:
 *     cache_layers[l] + block_table[j]*page_bytes  <-  staging_layers[l] + j*page_bytes
 * (page_bytes bytes).  Bytes of the cache outside the listed blocks are not
 * written.
 *   staging_layers  device array of n_layers pointers, each to n_pages*page_bytes
 *                   bytes laid out page after page; device memory, or pinned host memory
 *                   the device can address (the pages are then read over the host link)
 *   cache_layers    device array of n_layers device pointers, each to
 *                   num_blocks*page_bytes bytes (one layer's paged cache)
 *   block_table     device, n_pages int32 block ids; ids must be distinct (two equal
 *                   ids race); an id outside [0,num_blocks) sets
 *                   HS_DEVERR_BLOCK_OOB and that page is skipped
 *   page_bytes      > 0, multiple of 16
 * Every pointer in the arrays must be 16-byte aligned (else HS_DEVERR_MISALIGNED
 * and the layer is skipped).  n_layers == 0 or n_pages == 0 is a no-op.
 * Errors: HS_ERR_INVALID_ARG, HS_ERR_MISALIGNED (page_bytes), HS_ERR_CUDA.
 */
hs_status hs_restore_kv_pages(const void *const *staging_layers, void *const *cache_layers,
                              int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                              int64_t page_bytes, int64_t num_blocks, int32_t *d_err,
                              cudaStream_t stream);

/*
 * hs_restore_request -- hs_restore_kv_pages and hs_restore_state of one resumed
 * request in a single launch.
 *
 * Paper: Section 2.1 and Section 5.2 (the attention cache entries of [0,B) are
 * restored together with the recurrent state at B), Section 1 and Section 2.2.
 *
 * Same effect as hs_restore_kv_pages(staging_layers, cache_layers, n_layers,
 * block_table, n_pages, page_bytes, num_blocks) followed by
 * hs_restore_state(src_slots, dst_slots, n_slots, floats_each), with every slot
 * pointer 16-byte aligned (else HS_DEVERR_MISALIGNED and that slot is skipped)
 * and floats_each a multiple of 4.  The restored states are written so that a
 * prefill launched next finds them in L2.  Either part may be empty (n_layers or
 * n_pages == 0; n_slots or floats_each == 0).
 * Errors: HS_ERR_INVALID_ARG, HS_ERR_MISALIGNED (page_bytes % 16, floats_each % 4),
 * HS_ERR_CUDA.
 */
hs_status hs_restore_request(const void *const *staging_layers, void *const *cache_layers,
                             int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                             int64_t page_bytes, int64_t num_blocks, const float *const *src_slots,
                             float *const *dst_slots, int32_t n_slots, int64_t floats_each,
                             int32_t *d_err, cudaStream_t stream);

/*
 * hs_save_kv_pages -- gather KV pages of the paged cache into a staging pool (save).
 *
 * Paper: Section 3.1 (a save must have completed, not merely been submitted,
 * before dependent state is reused; the final regression delayed every save by
 * 500 ms and paired each dependent reuse with a wait on the actual save) and
 * Table 5 (D2H page comparisons, delayed-save wait pairs).
 *
 * For every layer l < n_layers and page j < n_pages:
 *     staging_layers[l] + j*page_bytes  <-  cache_layers[l] + block_table[j]*page_bytes
 * (page_bytes bytes), the inverse of hs_restore_kv_pages.  The call is
 * asynchronous: the pages are saved once the stream reaches the copy, so a
 * caller that will overwrite those cache blocks (or read the staging pool) from
 * other work must first wait for it, e.g. on a CUDA event recorded on `stream`
 * after this call.
 *   cache_layers    device array of n_layers device pointers, each to
 *                   num_blocks*page_bytes bytes (one layer's paged cache); read only
 *   staging_layers  device array of n_layers pointers, each to n_pages*page_bytes
 *                   bytes; device memory, or pinned host memory the device can
 *                   address (the pages are then written over the host link)
 *   block_table     device, n_pages int32 block ids, distinct; an id outside
 *                   [0,num_blocks) sets HS_DEVERR_BLOCK_OOB and that page is skipped
 *   page_bytes      > 0, multiple of 16
 * Every pointer in the arrays must be 16-byte aligned (else HS_DEVERR_MISALIGNED
 * and the layer is skipped).  n_layers == 0 or n_pages == 0 is a no-op.
 * Errors: HS_ERR_INVALID_ARG, HS_ERR_MISALIGNED (page_bytes), HS_ERR_CUDA.
 */
hs_status hs_save_kv_pages(const void *const *cache_layers, void *const *staging_layers,
                           int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                           int64_t page_bytes, int64_t num_blocks, int32_t *d_err,
                           cudaStream_t stream);

/*
 * hs_restore_kv_page_slices / hs_save_kv_page_slices -- one tensor-parallel rank's
 * slice of every KV page (restore: staging -> cache; save: cache -> staging).
 *
 * Paper: Table 1 (four-way tensor parallelism, FP8 KV setting) and Section 5.2
 * (restored bytes are counted per rank: each rank moves the pages of its own
 * heads).
 *
 * A page of page_bytes bytes is `rows` rows of row_bytes = page_bytes / rows bytes
 * (for the cache layout [2][page][kv head][head_dim]: rows = 2*page tokens, a row
 * = every KV head of one token); a rank owns bytes [col_off, col_off + col_bytes)
 * of every row (its KV heads).  The staging page holds the rank's rows back to
 * back, rows*col_bytes bytes, page after page.  For every layer l and page j:
 *     for r < rows:  cache_l[block_table[j]] + r*row_bytes + col_off   (col_bytes bytes)
 *                    <->  staging_l + (j*rows + r)*col_bytes
 * Bytes outside the slices are not written.  The element type is irrelevant (FP8
 * and BF16 pages are the same bytes to move).  rows = 1, col_off = 0,
 * col_bytes = page_bytes is hs_restore_kv_pages / hs_save_kv_pages.
 *   staging_layers, cache_layers, block_table, num_blocks, d_err: as for
 *                   hs_restore_kv_pages (staging may be pinned host memory)
 *   rows            >= 1, divides page_bytes
 *   col_off, col_bytes  col_off >= 0, col_bytes > 0, col_off + col_bytes <= row_bytes
 * Errors: HS_ERR_INVALID_ARG (sizes, slice outside the row), HS_ERR_MISALIGNED
 * (page_bytes, row_bytes, col_off or col_bytes not a multiple of 16), HS_ERR_CUDA.
 */
hs_status hs_restore_kv_page_slices(const void *const *staging_layers, void *const *cache_layers,
                                    int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                                    int64_t page_bytes, int32_t rows, int64_t col_off,
                                    int64_t col_bytes, int64_t num_blocks, int32_t *d_err,
                                    cudaStream_t stream);
hs_status hs_save_kv_page_slices(const void *const *cache_layers, void *const *staging_layers,
                                 int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                                 int64_t page_bytes, int32_t rows, int64_t col_off,
                                 int64_t col_bytes, int64_t num_blocks, int32_t *d_err,
                                 cudaStream_t stream);

/*
 * hs_restore_state -- restore recurrent states from checkpoint slots.
 *
 * Paper: Section 1 (a state updated in place cannot be rebuilt by reducing a
 * token count; it must be restored for the credited prefix) and Section 2.2.
 *
 * dst_slots[i][0..floats_each) <- src_slots[i][0..floats_each) for i < n, bit-exact.
 *   src_slots  device array of n device pointers (checkpoint slots; only read)
 *   dst_slots  device array of n device pointers (live states)
 * Slots may have any 4-byte alignment (16-byte aligned slots take the vector
 * path); NULL entries set HS_DEVERR_NULL and are skipped; slots must not overlap.
 * Errors: HS_ERR_INVALID_ARG, HS_ERR_CUDA.
 */
hs_status hs_restore_state(const float *const *src_slots, float *const *dst_slots, int32_t n,
                           int64_t floats_each, int32_t *d_err, cudaStream_t stream);

/*
 * hs_checkpoint_states -- snapshot live recurrent states into checkpoint slots.
 *
 * Paper: Table 1 (state checkpoints every C tokens) and Section 6 (a stored
 * checkpoint is an immutable payload).  Same contract as hs_restore_state with
 * src = live states and dst = checkpoint slots; restore never writes slots.
 */
hs_status hs_checkpoint_states(const float *const *live_states, float *const *ckpt_slots,
                               int32_t n, int64_t floats_each, int32_t *d_err,
                               cudaStream_t stream);

/* Which kernel hs_linattn_prefill_from_state runs. */
typedef enum hs_linattn_kernel {
    HS_LINATTN_AUTO = 0,       /* chunked tensor-core kernel when some n_tokens exceeds
                                  HS_SHORT_SEGMENT; the single-token kernel when every
                                  n_tokens is at most 1 (decode steps); else the recurrent
                                  kernel.  All three compute segments of at most
                                  HS_SHORT_SEGMENT tokens identically, so AUTO never changes
                                  results */
    HS_LINATTN_RECURRENT = 1,  /* per-token recurrence, CUDA cores */
    HS_LINATTN_CHUNKED_TC = 2, /* chunked form on tcgen05 tensor cores (d_k == d_v, 64 or
                                  128; at 64 the M = 128 products leave half their TMEM lanes
                                  unused) */
    HS_LINATTN_SINGLE_TOKEN = 3 /* one decode step per problem, state in registers, no
                                  shared memory (HS_ERR_UNSUPPORTED if some n_tokens > 1) */
} hs_linattn_kernel;

typedef struct hs_linattn_shape {
    int32_t batch;         /* independent problems: requests, or (request, layer) pairs */
    int32_t n_heads;       /* heads per problem */
    int32_t d_k;           /* key/query width: 64 or 128 */
    int32_t d_v;           /* value width: equal to d_k */
    int64_t max_tokens;    /* token extent T of q/k/v/log_g/o per problem (>= every n_tokens) */
    int32_t kernel;        /* hs_linattn_kernel */
    int32_t reserved;      /* must be 0 */
} hs_linattn_shape;

/*
 * hs_linattn_prefill_from_state -- gated linear-attention prefill from a
 * restored state.
 *
 * Paper: Section 2.2 (continue from the state of [0,B) over the suffix
 * [B,N)), Section 4.1 and Table 2 (matched checkpoint schedule), Section 4.2 /
 * Table 3 (fixed kernel configuration).  The paper runs its linear layers on
 * the FLA kernels without printing their recurrence; this call implements
 *     S_t = diag(g_t) S_{t-1} + k_t v_t^T,   o_t = q_t S_t,   g_t = exp(a_t)
 * with a_t <= 0 the per-dimension log-gates (a very negative a, e.g. -1e4,
 * is a zero gate).
 *
 * For problem b, token t < n_tokens[b] of q/k/v/log_g/o is absolute position
 * pos0[b] + t.  state[b] holds on entry the state of prefix [0,pos0[b]) and on
 * return that of [0,pos0[b]+n_tokens[b]).  Work is split into segments at the
 * multiples of HS_CHUNK on the absolute position grid and every segment is a
 * fixed function of its inputs and its incoming state, so resuming at a
 * multiple of HS_CHUNK reproduces a full recomputation bit for bit (with AUTO,
 * or with the same explicit kernel in both runs).
 *
 *   shp        host; batch in [0, HS_MAX_BATCH]; d_k == d_v in {64,128}
 *   q, k       device bf16 [batch][max_tokens][n_heads][d_k]
 *   v          device bf16 [batch][max_tokens][n_heads][d_v]
 *   log_g      device float [batch][max_tokens][n_heads][d_k]
 *   o          device float [batch][max_tokens][n_heads][d_v]; rows t >= n_tokens[b]
 *              are not written
 *              max_tokens is the token stride between problems; only rows
 *              t < n_tokens[b] of each problem are read or written, so views that start
 *              mid-sequence (pointer offset by whole tokens) are valid as long as those
 *              rows exist.
 *   state      device float [batch][n_heads][d_k][d_v], row index = key dimension
 *   pos0       host int64 [batch], >= 0
 *   n_tokens   host int32 [batch], 0 <= n_tokens[b] <= max_tokens
 *   ckpt_interval  C: 0 (no checkpoints) or a positive multiple of HS_CHUNK
 *   ckpt_slots device array of device pointers or NULL (no checkpoints written).
 *              Problem b emits one checkpoint for every multiple m*C in
 *              (pos0[b], pos0[b]+n_tokens[b]]: the state of prefix [0,m*C), float
 *              [n_heads][d_k][d_v].  Slots are listed problem by problem, in
 *              position order; hs_linattn_num_checkpoints gives the count.  Each
 *              slot must be 16-byte aligned (else HS_DEVERR_MISALIGNED, not written).
 *   d_err      optional device int32 (see conventions)
 * Accuracy: the recurrent and single-token kernels compute in float32 token by
 * token.  The tensor-core kernel runs a chunk on fp16 operands (11 significant
 * bits, float32 accumulation and state) when its log-gates are <= 0, its total
 * log2-decay stays >= -10 in every key dimension and every operand provably fits
 * fp16; any other chunk runs on tf32 operands with the intra-chunk scores computed
 * in float32.  On both paths a token's own score A_ii = q_i . k_i is summed in
 * float32 from the bf16 inputs, so operand rounding enters only through the
 * products of different tokens and through the state.  Per output element,
 * with eps = 2^-11 and Q~ = q 2^Lam, K~ = k 2^-Lam the decayed operands of the
 * chunk, the error is at most about
 *   2 eps (sum_d |Q~_id| |S_de| + sum_{j<i} |v_je| sum_d |Q~_id K~_jd|)
 *     + eps sum_{j<=i} |A_ij| |v_je|
 * plus the error the state carries in from earlier chunks (the same form).
 * This stays below 2e-3 of the head's largest output whenever those sums of
 * magnitudes are within about 1,000 times of it: over 3,000 seeded stress calls
 * (tails up to 600 tokens, v scaled by 2^17, q and k by 64, gates of -30, -1.2,
 * -1e4 and +0.02, states up to 2^16) the largest max-normalised error was 5.6e-4.
 * All of q, k, v, log_g, o, state must be 16-byte aligned.  q/k/v/log_g are only
 * read; o, state and the slots must not overlap the inputs or each other.
 * Token rows are 32-bit: b*max_tokens + n_tokens[b] must stay below 2^31.
 * Errors: HS_ERR_INVALID_ARG, HS_ERR_MISALIGNED, HS_ERR_UNSUPPORTED (d_k/d_v,
 * ckpt_interval not a multiple of HS_CHUNK, batch > HS_MAX_BATCH, rows beyond
 * 2^31), HS_ERR_CUDA.
 */
hs_status hs_linattn_prefill_from_state(const hs_linattn_shape *shp, const uint16_t *q,
                                        const uint16_t *k, const uint16_t *v, const float *log_g,
                                        float *o, float *state, const int64_t *pos0,
                                        const int32_t *n_tokens, int32_t ckpt_interval,
                                        float *const *ckpt_slots, int32_t *d_err,
                                        cudaStream_t stream);

/*
 * hs_linattn_prefill_packed -- hs_linattn_prefill_from_state over a packed
 * (unpadded) token layout: the tails of a batch of requests, each with its own
 * resume point, back to back in one launch, as an engine batches them (the
 * paper's engine schedules the resumed tail of every request, Section 2.2).
 *
 * Identical to hs_linattn_prefill_from_state (same arithmetic, same bits)
 * except where each problem's tokens live: token t of problem b is row
 * cu_rows[b] + t of q, k, v, log_g and o, which are [rows][n_heads][d]; the
 * shape's max_tokens is not used.
 *   cu_rows  host int64 [batch + 1], 0 <= cu_rows[b] <= cu_rows[b+1] and
 *            n_tokens[b] <= cu_rows[b+1] - cu_rows[b] (the usual cumulative
 *            sequence lengths have equality); rows must stay below 2^31
 * Errors: as hs_linattn_prefill_from_state; HS_ERR_INVALID_ARG also for a NULL
 * or non-monotone cu_rows or a problem longer than its rows.
 */
hs_status hs_linattn_prefill_packed(const hs_linattn_shape *shp, const uint16_t *q,
                                    const uint16_t *k, const uint16_t *v, const float *log_g,
                                    float *o, float *state, const int64_t *pos0,
                                    const int32_t *n_tokens, const int64_t *cu_rows,
                                    int32_t ckpt_interval, float *const *ckpt_slots,
                                    int32_t *d_err, cudaStream_t stream);

/*
 * hs_linattn_prefill_scan -- the prefill of hs_linattn_prefill_from_state for calls
 * with few problems: the segments of each problem's tail run in parallel.
 *
 * Paper: as hs_linattn_prefill_from_state (Section 2.2, Section 4.1 and Table 2).
 * The recurrence is linear in the state, so over a segment [s,e) of the absolute
 * 64-token grid S_e = diag(G) S_s + dS with G = exp(sum of the segment's log-gates)
 * and dS the segment's state from the zero state.  Three launches: a segment-state
 * kernel computes every (segment, head)'s dS and G at once (tf32 tensor-core
 * products), an elementwise scan chains S_{n+1} = G_n S_n + dS_n per (problem, head)
 * and writes the checkpoints and the final state, and the tensor-core prefill kernel
 * runs every segment again from its start state S_n for the outputs (consecutive
 * segments grouped so that the launch fills the SMs; each segment still starts from its
 * own S_n, so the grouping changes no result).  A call with one problem of 16 heads
 * then spreads (segments x 16) units of work over the GPU instead of 16 chains; for
 * calls whose (problem, head) pairs already fill the SMs it is slower than
 * hs_linattn_prefill_from_state, which reads and writes fewer bytes.
 *
 * Results: the outputs, final states and checkpoints of the same recurrence, within
 * the same accuracy as hs_linattn_prefill_from_state (the two are not bit-identical:
 * here the state enters each segment through the scan's fma instead of the tensor-
 * core accumulation).  Every step depends only on the segment's inputs and the state
 * it starts from, so resuming at a multiple of HS_CHUNK with this call reproduces a
 * full recomputation with this call bit for bit.
 *
 * Arguments as hs_linattn_prefill_from_state (shp->kernel AUTO or CHUNKED_TC: the
 * segments run on the tensor-core kernel), plus
 *   workspace        device memory the call uses between its launches, 16-byte
 *                    aligned, at least hs_linattn_scan_workspace_bytes bytes: two float
 *                    states per segment (2 x segments x n_heads x d_k x d_v x 4 bytes);
 *                    its contents on entry are ignored and on return undefined
 *   workspace_bytes  its size
 * The rows t >= n_tokens[b] of o are not written.  The workspace must not overlap
 * any other argument, and concurrent calls need their own workspaces.
 * Errors: as hs_linattn_prefill_from_state; HS_ERR_INVALID_ARG also for a NULL or
 * too small workspace, HS_ERR_MISALIGNED for a misaligned one, HS_ERR_UNSUPPORTED
 * for another kernel choice.
 */
hs_status hs_linattn_prefill_scan(const hs_linattn_shape *shp, const uint16_t *q,
                                  const uint16_t *k, const uint16_t *v, const float *log_g,
                                  float *o, float *state, const int64_t *pos0,
                                  const int32_t *n_tokens, int32_t ckpt_interval,
                                  float *const *ckpt_slots, void *workspace,
                                  int64_t workspace_bytes, int32_t *d_err, cudaStream_t stream);

/*
 * hs_linattn_scan_workspace_bytes -- the workspace hs_linattn_prefill_scan needs for
 * these arguments (host only): 2 x segments x n_heads x d_k x d_v x 4 bytes, with
 * segments = sum over b of ceil((pos0[b] + n_tokens[b]) / 64) - floor(pos0[b] / 64)
 * for n_tokens[b] > 0.  Errors: the shape and argument checks of the call.
 */
hs_status hs_linattn_scan_workspace_bytes(const hs_linattn_shape *shp, const int64_t *pos0,
                                          const int32_t *n_tokens, int64_t *bytes_out);

/* Size of the fixed device workspace of hs_linattn_prefill_scan_noalloc (16 MiB per device):
 * room for 2 x 8 segments x 16 heads x 128 x 128 floats, e.g. one 512-token tail of 16
 * heads at d = 128 that starts on the 64-token grid. */
#define HS_NOALLOC_SCRATCH_BYTES (16u << 20)

/*
 * hs_linattn_prefill_scan_noalloc -- hs_linattn_prefill_scan for callers that cannot
 * allocate device memory when they resume a request.
 *
 * The paper has no counterpart: it is a calling convention of this library.  Some callers
 * have no device memory to give out at that point: a serving engine commonly reserves
 * nearly all free HBM for its KV-cache block pool at start-up and allocates only from its
 * own pools afterwards, and its scheduler loop cannot take the device-wide synchronisation
 * that cudaMalloc or cudaFree may cause.  This call takes the workspace from a fixed array
 * of HS_NOALLOC_SCRATCH_BYTES bytes that the library keeps on each device, and calls no
 * allocating routine.
 *
 * Arguments, results and errors: as hs_linattn_prefill_scan without workspace and
 * workspace_bytes, plus HS_ERR_TOO_LARGE when hs_linattn_scan_workspace_bytes for these
 * arguments exceeds HS_NOALLOC_SCRATCH_BYTES (checked on the host before any CUDA call), and
 * HS_ERR_CUDA when the set-up below fails.
 * Set-up: the first call on a device that has tokens to compute looks up the array's
 * address there (cudaGetSymbolAddress, with the current device, which loads the array if
 * the library's module is loaded lazily) and caches it; make that first call before any
 * stream capture.  The stream must belong to the current device.
 * Sharing: every call on a device uses the same array and finds the previous call's data
 * in it; nothing has to be cleared, since a call writes every word it reads first.  Calls
 * that can run at the same time on the GPU (two streams, or host threads without an order
 * between their calls) corrupt each other's workspace: serialise them.
 */
hs_status hs_linattn_prefill_scan_noalloc(const hs_linattn_shape *shp, const uint16_t *q,
                                          const uint16_t *k, const uint16_t *v,
                                          const float *log_g, float *o, float *state,
                                          const int64_t *pos0, const int32_t *n_tokens,
                                          int32_t ckpt_interval, float *const *ckpt_slots,
                                          int32_t *d_err, cudaStream_t stream);

/*
 * hs_linattn_num_checkpoints -- number of checkpoint slots the prefill above
 * writes for these arguments (host only): the sum over b of
 * floor((pos0[b]+n_tokens[b])/C) - floor(pos0[b]/C), 0 when C == 0.
 */
hs_status hs_linattn_num_checkpoints(int32_t batch, const int64_t *pos0, const int32_t *n_tokens,
                                     int32_t ckpt_interval, int64_t *total_out);

#ifdef __cplusplus
}
#endif

#endif /* HS_H */
