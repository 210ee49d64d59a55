// C-ABI entry points of libhs: host-side validation, then one launch per call.
// Validation happens before any CUDA runtime call, so argument errors are
// reported without touching the GPU.
#include <algorithm>
#include <cstring>

#include "gla_dstate.cuh"
#include "hs_internal.cuh"
#include "hs_test.h"

namespace {

inline bool misaligned16(const void *p)
{
    return (reinterpret_cast<uintptr_t>(p) & 15u) != 0;
}

inline hs_status cuda_status(cudaError_t e)
{
    return e == cudaSuccess ? HS_OK : HS_ERR_CUDA;
}

// the current device's SM count, queried once per device
std::atomic<int> g_sm_count[64];

hs_status sm_count(int *out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return HS_ERR_CUDA;
    if (dev >= 0 && dev < 64 && (*out = g_sm_count[dev].load(std::memory_order_relaxed)) > 0)
        return HS_OK;
    if (cudaDeviceGetAttribute(out, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return HS_ERR_CUDA;
    if (dev >= 0 && dev < 64)
        g_sm_count[dev].store(*out, std::memory_order_relaxed);
    return HS_OK;
}

hs_status copy_slots(const float *const *src, float *const *dst, int32_t n, int64_t floats_each,
                     int32_t *d_err, cudaStream_t stream)
{
    if (n < 0 || floats_each < 0)
        return HS_ERR_INVALID_ARG;
    if (n == 0 || floats_each == 0)
        return HS_OK;
    if (src == nullptr || dst == nullptr)
        return HS_ERR_INVALID_ARG;
    int sms = 0;
    hs_status st = sm_count(&sms);
    if (st != HS_OK)
        return st;
    return cuda_status(hs::launch_slot_copy(src, dst, n, floats_each, d_err, sms, stream));
}

}  // namespace

extern "C" {

const char *hs_status_string(hs_status s)
{
    switch (s) {
    case HS_OK: return "HS_OK";
    case HS_ERR_INVALID_ARG: return "HS_ERR_INVALID_ARG: invalid argument";
    case HS_ERR_MISALIGNED: return "HS_ERR_MISALIGNED: pointer or size not 16-byte aligned";
    case HS_ERR_UNSUPPORTED: return "HS_ERR_UNSUPPORTED: shape not implemented";
    case HS_ERR_CUDA: return "HS_ERR_CUDA: CUDA runtime call or launch failed";
    case HS_ERR_DEVICE_CHECK: return "HS_ERR_DEVICE_CHECK: a kernel reported an error";
    case HS_ERR_TOO_LARGE:
        return "HS_ERR_TOO_LARGE: the call needs more than the library's fixed workspace";
    }
    return "unknown hs_status";
}

int32_t hs_version(void)
{
    return 100;  // 0.1.0
}

hs_status hs_align_prefix(int64_t N, int64_t hit_len, const int64_t *avail_ckpts, int32_t n_avail,
                          int32_t page_size, int64_t *c_out, int64_t *n_pages_out,
                          int64_t *tail_out)
{
    if (N < 1 || hit_len < 0 || hit_len > N || page_size < 1 || n_avail < 0)
        return HS_ERR_INVALID_ARG;
    if (c_out == nullptr || n_pages_out == nullptr || tail_out == nullptr)
        return HS_ERR_INVALID_ARG;
    if (n_avail > 0 && avail_ckpts == nullptr)
        return HS_ERR_INVALID_ARG;
    for (int32_t i = 0; i < n_avail; ++i) {
        if (avail_ckpts[i] < 0 || (i > 0 && avail_ckpts[i] <= avail_ckpts[i - 1]))
            return HS_ERR_INVALID_ARG;
    }
    // strict prefix: the query excludes the last prompt token and stops at the hit
    const int64_t bound = (N - 1 < hit_len) ? N - 1 : hit_len;
    // largest listed position <= bound (binary search), then walk down to a page boundary
    int32_t lo = 0, hi = n_avail;  // first index with value > bound
    while (lo < hi) {
        const int32_t mid = lo + (hi - lo) / 2;
        if (avail_ckpts[mid] <= bound)
            lo = mid + 1;
        else
            hi = mid;
    }
    int64_t c = 0;
    for (int32_t i = lo - 1; i >= 0; --i) {
        if (avail_ckpts[i] % page_size == 0) {
            c = avail_ckpts[i];
            break;
        }
    }
    *c_out = c;
    *n_pages_out = c / page_size;
    *tail_out = N - c;
    return HS_OK;
}

hs_status hs_restore_kv_pages(const void *const *staging_layers, void *const *cache_layers,
                              int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                              int64_t page_bytes, int64_t num_blocks, int32_t *d_err,
                              cudaStream_t stream)
{
    if (n_layers < 0 || n_pages < 0 || page_bytes <= 0 || num_blocks < 0)
        return HS_ERR_INVALID_ARG;
    if (page_bytes % 16 != 0)
        return HS_ERR_MISALIGNED;
    if (n_layers == 0 || n_pages == 0)
        return HS_OK;
    if (staging_layers == nullptr || cache_layers == nullptr || block_table == nullptr)
        return HS_ERR_INVALID_ARG;
    if ((int64_t)n_pages > num_blocks)
        return HS_ERR_INVALID_ARG;  // block ids must be distinct
    int sms = 0;
    hs_status st = sm_count(&sms);
    if (st != HS_OK)
        return st;
    return cuda_status(hs::launch_kv_scatter(staging_layers, cache_layers, n_layers, block_table,
                                             n_pages, page_bytes, num_blocks, d_err, sms, stream));
}

hs_status hs_save_kv_pages(const void *const *cache_layers, void *const *staging_layers,
                           int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                           int64_t page_bytes, int64_t num_blocks, int32_t *d_err,
                           cudaStream_t stream)
{
    if (n_layers < 0 || n_pages < 0 || page_bytes <= 0 || num_blocks < 0)
        return HS_ERR_INVALID_ARG;
    if (page_bytes % 16 != 0)
        return HS_ERR_MISALIGNED;
    if (n_layers == 0 || n_pages == 0)
        return HS_OK;
    if (staging_layers == nullptr || cache_layers == nullptr || block_table == nullptr)
        return HS_ERR_INVALID_ARG;
    if ((int64_t)n_pages > num_blocks)
        return HS_ERR_INVALID_ARG;  // a request's pages occupy distinct blocks
    int sms = 0;
    hs_status st = sm_count(&sms);
    if (st != HS_OK)
        return st;
    return cuda_status(hs::launch_kv_gather(cache_layers, staging_layers, n_layers, block_table,
                                            n_pages, page_bytes, num_blocks, d_err, sms, stream));
}

static hs_status kv_slices(bool gather, const void *const *from, void *const *to, int32_t n_layers,
                           const int32_t *block_table, int32_t n_pages, int64_t page_bytes,
                           int32_t rows, int64_t col_off, int64_t col_bytes, int64_t num_blocks,
                           int32_t *d_err, cudaStream_t stream)
{
    if (n_layers < 0 || n_pages < 0 || page_bytes <= 0 || num_blocks < 0 || rows <= 0 ||
        col_off < 0 || col_bytes <= 0)
        return HS_ERR_INVALID_ARG;
    if (page_bytes % rows != 0 || col_off + col_bytes > page_bytes / rows)
        return HS_ERR_INVALID_ARG;
    if (page_bytes % 16 != 0 || (page_bytes / rows) % 16 != 0 || col_off % 16 != 0 ||
        col_bytes % 16 != 0)
        return HS_ERR_MISALIGNED;
    if ((int64_t)rows * (col_bytes / 16) > INT32_MAX)
        return HS_ERR_UNSUPPORTED;   // one page slice is at most 2^31 16-byte vectors
    if (n_layers == 0 || n_pages == 0)
        return HS_OK;
    if (from == nullptr || to == nullptr || block_table == nullptr)
        return HS_ERR_INVALID_ARG;
    if ((int64_t)n_pages > num_blocks)
        return HS_ERR_INVALID_ARG;  // a request's pages occupy distinct blocks
    int sms = 0;
    hs_status st = sm_count(&sms);
    if (st != HS_OK)
        return st;
    return cuda_status(hs::launch_kv_slices(gather, from, to, n_layers, block_table, n_pages,
                                            page_bytes, rows, col_off, col_bytes, num_blocks, d_err,
                                            sms, stream));
}

hs_status hs_restore_kv_page_slices(const void *const *staging_layers, void *const *cache_layers,
                                    int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                                    int64_t page_bytes, int32_t rows, int64_t col_off,
                                    int64_t col_bytes, int64_t num_blocks, int32_t *d_err,
                                    cudaStream_t stream)
{
    return kv_slices(false, staging_layers, cache_layers, n_layers, block_table, n_pages,
                     page_bytes, rows, col_off, col_bytes, num_blocks, d_err, stream);
}

hs_status hs_save_kv_page_slices(const void *const *cache_layers, void *const *staging_layers,
                                 int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                                 int64_t page_bytes, int32_t rows, int64_t col_off,
                                 int64_t col_bytes, int64_t num_blocks, int32_t *d_err,
                                 cudaStream_t stream)
{
    return kv_slices(true, cache_layers, staging_layers, n_layers, block_table, n_pages,
                     page_bytes, rows, col_off, col_bytes, num_blocks, d_err, stream);
}

hs_status hs_restore_request(const void *const *staging_layers, void *const *cache_layers,
                             int32_t n_layers, const int32_t *block_table, int32_t n_pages,
                             int64_t page_bytes, int64_t num_blocks, const float *const *src_slots,
                             float *const *dst_slots, int32_t n_slots, int64_t floats_each,
                             int32_t *d_err, cudaStream_t stream)
{
    if (n_layers < 0 || n_pages < 0 || page_bytes <= 0 || num_blocks < 0 || n_slots < 0 ||
        floats_each < 0)
        return HS_ERR_INVALID_ARG;
    if (page_bytes % 16 != 0 || floats_each % 4 != 0)
        return HS_ERR_MISALIGNED;
    const bool kv = n_layers > 0 && n_pages > 0;
    const bool st = n_slots > 0 && floats_each > 0;
    if (kv && (staging_layers == nullptr || cache_layers == nullptr || block_table == nullptr))
        return HS_ERR_INVALID_ARG;
    if (kv && (int64_t)n_pages > num_blocks)
        return HS_ERR_INVALID_ARG;  // a request's pages occupy distinct blocks
    if (st && (src_slots == nullptr || dst_slots == nullptr))
        return HS_ERR_INVALID_ARG;
    if (!kv && !st)
        return HS_OK;
    int sms = 0;
    hs_status status = sm_count(&sms);
    if (status != HS_OK)
        return status;
    return cuda_status(hs::launch_restore_request(
        staging_layers, cache_layers, kv ? n_layers : 0, block_table, kv ? n_pages : 0, page_bytes,
        num_blocks, src_slots, dst_slots, st ? n_slots : 0, st ? floats_each : 0, d_err, sms,
        stream));
}

hs_status hs_restore_state(const float *const *src_slots, float *const *dst_slots, int32_t n,
                           int64_t floats_each, int32_t *d_err, cudaStream_t stream)
{
    return copy_slots(src_slots, dst_slots, n, floats_each, d_err, stream);
}

hs_status hs_checkpoint_states(const float *const *live_states, float *const *ckpt_slots,
                               int32_t n, int64_t floats_each, int32_t *d_err,
                               cudaStream_t stream)
{
    return copy_slots(live_states, ckpt_slots, n, floats_each, d_err, stream);
}

hs_status hs_linattn_num_checkpoints(int32_t batch, const int64_t *pos0, const int32_t *n_tokens,
                                     int32_t ckpt_interval, int64_t *total_out)
{
    if (batch < 0 || ckpt_interval < 0 || total_out == nullptr)
        return HS_ERR_INVALID_ARG;
    if (batch > 0 && (pos0 == nullptr || n_tokens == nullptr))
        return HS_ERR_INVALID_ARG;
    int64_t total = 0;
    for (int32_t b = 0; b < batch; ++b) {
        if (pos0[b] < 0 || n_tokens[b] < 0)
            return HS_ERR_INVALID_ARG;
        if (ckpt_interval > 0 && n_tokens[b] > 0)
            total += (pos0[b] + n_tokens[b]) / ckpt_interval - pos0[b] / ckpt_interval;
    }
    *total_out = total;
    return HS_OK;
}

// The prefill of both token layouts: cu_rows == nullptr is the padded layout (problem b's
// token t at row b*max_tokens + t), else problem b's token t is at row cu_rows[b] + t.
static hs_status prefill(const hs_linattn_shape *shp, const uint16_t *q, const uint16_t *k,
                         const uint16_t *v, const float *log_g, float *o, float *state,
                         const int64_t *pos0, const int32_t *n_tokens, const int64_t *cu_rows,
                         int32_t ckpt_interval, float *const *ckpt_slots, int32_t *d_err,
                         cudaStream_t stream, bool stall_for_test = false)
{
    if (shp == nullptr)
        return HS_ERR_INVALID_ARG;
    const hs_linattn_shape s = *shp;
    if (s.batch < 0 || s.n_heads < 1 || s.max_tokens < 0 || s.reserved != 0)
        return HS_ERR_INVALID_ARG;
    if (s.kernel != HS_LINATTN_AUTO && s.kernel != HS_LINATTN_RECURRENT &&
        s.kernel != HS_LINATTN_CHUNKED_TC && s.kernel != HS_LINATTN_SINGLE_TOKEN)
        return HS_ERR_INVALID_ARG;
    if (s.d_k != s.d_v || (s.d_k != 64 && s.d_k != 128))
        return HS_ERR_UNSUPPORTED;
    if (stall_for_test && s.kernel != HS_LINATTN_CHUNKED_TC)
        return HS_ERR_UNSUPPORTED;   // the hook exists in the tensor-core kernel only
    if (s.batch > HS_MAX_BATCH)
        return HS_ERR_UNSUPPORTED;
    if (ckpt_interval < 0)
        return HS_ERR_INVALID_ARG;
    if (ckpt_interval % HS_CHUNK != 0)
        return HS_ERR_UNSUPPORTED;
    if (s.batch == 0)
        return HS_OK;
    if (pos0 == nullptr || n_tokens == nullptr || state == nullptr)
        return HS_ERR_INVALID_ARG;
    bool any_tokens = false;
    for (int32_t b = 0; b < s.batch; ++b) {
        if (pos0[b] < 0 || n_tokens[b] < 0)
            return HS_ERR_INVALID_ARG;
        if (pos0[b] > ((int64_t)1 << 40))
            return HS_ERR_INVALID_ARG;
        if (cu_rows == nullptr) {
            if ((int64_t)n_tokens[b] > s.max_tokens)
                return HS_ERR_INVALID_ARG;
        } else if (cu_rows[b] < 0 || cu_rows[b + 1] < cu_rows[b] ||
                   (int64_t)n_tokens[b] > cu_rows[b + 1] - cu_rows[b]) {
            return HS_ERR_INVALID_ARG;
        }
        any_tokens = any_tokens || n_tokens[b] > 0;
    }
    if (!any_tokens)
        return HS_OK;
    if (q == nullptr || k == nullptr || v == nullptr || log_g == nullptr || o == nullptr)
        return HS_ERR_INVALID_ARG;
    if (misaligned16(q) || misaligned16(k) || misaligned16(v) || misaligned16(log_g) ||
        misaligned16(o) || misaligned16(state))
        return HS_ERR_MISALIGNED;

    hs::GlaParams p;
    std::memset(&p, 0, sizeof p);
    p.q = q;
    p.k = k;
    p.v = v;
    p.log_g = log_g;
    p.o = o;
    p.state = state;
    p.ckpt_slots = (ckpt_interval > 0) ? ckpt_slots : nullptr;
    p.d_err = d_err;
    p.batch = s.batch;
    p.n_heads = s.n_heads;
    p.ckpt_interval = (p.ckpt_slots != nullptr) ? ckpt_interval : 0;
    p.stall_for_test = stall_for_test ? 1 : 0;
    int64_t base = 0;
    for (int32_t b = 0; b < s.batch; ++b) {
        const int64_t r0 = cu_rows ? cu_rows[b] : (int64_t)b * s.max_tokens;
        if (r0 + n_tokens[b] > INT32_MAX)
            return HS_ERR_UNSUPPORTED;   // token rows are 32-bit
        p.pos0[b] = pos0[b];
        p.n_tokens[b] = n_tokens[b];
        p.row0[b] = (int32_t)r0;
        p.ck_base[b] = (int32_t)base;
        if (p.ckpt_interval > 0 && n_tokens[b] > 0)
            base += (pos0[b] + n_tokens[b]) / p.ckpt_interval - pos0[b] / p.ckpt_interval;
    }
    if (base > INT32_MAX)
        return HS_ERR_INVALID_ARG;

    const bool tc_ok = hs::gla_chunked_tc_supported(s.d_k);
    if (s.kernel == HS_LINATTN_CHUNKED_TC && !tc_ok)
        return HS_ERR_UNSUPPORTED;
    int32_t max_n = 0;
    for (int32_t b = 0; b < s.batch; ++b)
        max_n = n_tokens[b] > max_n ? n_tokens[b] : max_n;
    if (s.kernel == HS_LINATTN_SINGLE_TOKEN && max_n > 1)
        return HS_ERR_UNSUPPORTED;
    // AUTO: decode steps (one token per problem) take the single-token kernel, other calls
    // whose tails are all short the recurrent kernel; both compute such segments bit for
    // bit like the chunked kernel does, so the choice never changes results; everything
    // else takes the tensor-core kernel
    const bool use_tc = s.kernel == HS_LINATTN_CHUNKED_TC ||
                        (s.kernel == HS_LINATTN_AUTO && tc_ok && max_n > HS_SHORT_SEGMENT);
    if (use_tc)
        return cuda_status(hs::launch_gla_chunked_tc(p, s.d_k, stream));
    if (s.kernel == HS_LINATTN_SINGLE_TOKEN || (s.kernel == HS_LINATTN_AUTO && max_n == 1))
        return cuda_status(hs::launch_gla_decode(p, s.d_k, stream));
    return cuda_status(hs::launch_gla_recurrent(p, s.d_k, stream));
}

hs_status hs_linattn_prefill_from_state(const hs_linattn_shape *shp, const uint16_t *q,
                                        const uint16_t *k, const uint16_t *v, const float *log_g,
                                        float *o, float *state, const int64_t *pos0,
                                        const int32_t *n_tokens, int32_t ckpt_interval,
                                        float *const *ckpt_slots, int32_t *d_err,
                                        cudaStream_t stream)
{
    return prefill(shp, q, k, v, log_g, o, state, pos0, n_tokens, nullptr, ckpt_interval,
                   ckpt_slots, d_err, stream);
}

hs_status hs_test_prefill_stalled(const hs_linattn_shape *shp, const uint16_t *q,
                                  const uint16_t *k, const uint16_t *v, const float *log_g,
                                  float *o, float *state, const int64_t *pos0,
                                  const int32_t *n_tokens, int32_t ckpt_interval,
                                  float *const *ckpt_slots, int32_t *d_err, cudaStream_t stream)
{
    return prefill(shp, q, k, v, log_g, o, state, pos0, n_tokens, nullptr, ckpt_interval,
                   ckpt_slots, d_err, stream, true);
}

// ---- the segment-parallel prefill: every segment from the zero state, a state scan, every
// segment from its start state ----

// segments of [pos0, pos0 + n) on the HS_CHUNK grid
static int64_t n_segments(int64_t pos0, int64_t n)
{
    return n > 0 ? (pos0 + n + HS_CHUNK - 1) / HS_CHUNK - pos0 / HS_CHUNK : 0;
}

// the checks of hs_linattn_prefill_from_state that do not touch device memory, and the
// number of segments; HS_OK with *n_seg = 0 when there is nothing to compute
static hs_status scan_check(const hs_linattn_shape *shp, const int64_t *pos0,
                            const int32_t *n_tokens, int64_t *n_seg)
{
    if (shp == nullptr || n_seg == nullptr)
        return HS_ERR_INVALID_ARG;
    const hs_linattn_shape s = *shp;
    if (s.batch < 0 || s.n_heads < 1 || s.max_tokens < 0 || s.reserved != 0)
        return HS_ERR_INVALID_ARG;
    if (s.kernel != HS_LINATTN_AUTO && s.kernel != HS_LINATTN_CHUNKED_TC)
        return s.kernel >= HS_LINATTN_AUTO && s.kernel <= HS_LINATTN_SINGLE_TOKEN
                   ? HS_ERR_UNSUPPORTED : HS_ERR_INVALID_ARG;
    if (s.d_k != s.d_v || (s.d_k != 64 && s.d_k != 128))
        return HS_ERR_UNSUPPORTED;
    if (s.batch > HS_MAX_BATCH)
        return HS_ERR_UNSUPPORTED;
    *n_seg = 0;
    if (s.batch > 0 && (pos0 == nullptr || n_tokens == nullptr))
        return HS_ERR_INVALID_ARG;
    int64_t total = 0;
    for (int32_t b = 0; b < s.batch; ++b) {
        if (pos0[b] < 0 || n_tokens[b] < 0 || pos0[b] > ((int64_t)1 << 40) ||
            (int64_t)n_tokens[b] > s.max_tokens)
            return HS_ERR_INVALID_ARG;
        if ((int64_t)b * s.max_tokens + n_tokens[b] > INT32_MAX)
            return HS_ERR_UNSUPPORTED;   // token rows are 32-bit
        total += n_segments(pos0[b], n_tokens[b]);
    }
    if (total * s.n_heads > INT32_MAX)
        return HS_ERR_UNSUPPORTED;   // (segment, head) units are 32-bit
    *n_seg = total;
    return HS_OK;
}

hs_status hs_linattn_scan_workspace_bytes(const hs_linattn_shape *shp, const int64_t *pos0,
                                          const int32_t *n_tokens, int64_t *bytes_out)
{
    if (bytes_out == nullptr)
        return HS_ERR_INVALID_ARG;
    int64_t n_seg = 0;
    const hs_status st = scan_check(shp, pos0, n_tokens, &n_seg);
    if (st != HS_OK)
        return st;
    *bytes_out = 2 * n_seg * shp->n_heads * (int64_t)shp->d_k * shp->d_v * 4;
    return HS_OK;
}

hs_status hs_linattn_prefill_scan(const hs_linattn_shape *shp, const uint16_t *q,
                                  const uint16_t *k, const uint16_t *v, const float *log_g,
                                  float *o, float *state, const int64_t *pos0,
                                  const int32_t *n_tokens, int32_t ckpt_interval,
                                  float *const *ckpt_slots, void *workspace,
                                  int64_t workspace_bytes, int32_t *d_err, cudaStream_t stream)
{
    int64_t n_seg = 0;
    hs_status st = scan_check(shp, pos0, n_tokens, &n_seg);
    if (st != HS_OK)
        return st;
    const hs_linattn_shape s = *shp;
    if (ckpt_interval < 0)
        return HS_ERR_INVALID_ARG;
    if (ckpt_interval % HS_CHUNK != 0)
        return HS_ERR_UNSUPPORTED;
    if (n_seg == 0)
        return HS_OK;
    if (q == nullptr || k == nullptr || v == nullptr || log_g == nullptr || o == nullptr ||
        state == nullptr || workspace == nullptr)
        return HS_ERR_INVALID_ARG;
    if (misaligned16(q) || misaligned16(k) || misaligned16(v) || misaligned16(log_g) ||
        misaligned16(o) || misaligned16(state) || misaligned16(workspace))
        return HS_ERR_MISALIGNED;
    const int64_t D = s.d_k;
    const int64_t per = (int64_t)s.n_heads * D * D;     // floats of one segment's state
    if (workspace_bytes < 2 * n_seg * per * 4)
        return HS_ERR_INVALID_ARG;
    float *ws_dS = static_cast<float *>(workspace);
    float *ws_Sn = ws_dS + n_seg * per;

    // the scan's parameters (the original problems) and the segments' first rows
    hs::ScanParams sp;
    std::memset(&sp, 0, sizeof sp);
    sp.state = state;
    sp.dS = ws_dS;
    sp.Sn = ws_Sn;
    sp.ckpt_slots = (ckpt_interval > 0) ? ckpt_slots : nullptr;
    sp.d_err = d_err;
    sp.batch = s.batch;
    sp.n_heads = s.n_heads;
    sp.ckpt_interval = (sp.ckpt_slots != nullptr) ? ckpt_interval : 0;
    int64_t seg = 0, ck = 0;
    for (int32_t b = 0; b < s.batch; ++b) {
        sp.pos0[b] = pos0[b];
        sp.n_tokens[b] = n_tokens[b];
        sp.row0[b] = (int32_t)((int64_t)b * s.max_tokens);
        sp.ck_base[b] = (int32_t)ck;
        sp.seg_base[b] = (int32_t)seg;
        seg += n_segments(pos0[b], n_tokens[b]);
        if (sp.ckpt_interval > 0 && n_tokens[b] > 0)
            ck += (pos0[b] + n_tokens[b]) / sp.ckpt_interval - pos0[b] / sp.ckpt_interval;
    }
    if (ck > INT32_MAX)
        return HS_ERR_INVALID_ARG;

    // every segment's state from the zero state (dS)
    hs::DStateParams dp;
    std::memset(&dp, 0, sizeof dp);
    dp.k = k;
    dp.v = v;
    dp.log_g = log_g;
    dp.dS = ws_dS;
    dp.Sn = ws_Sn;
    dp.d_err = d_err;
    dp.batch = s.batch;
    dp.n_heads = s.n_heads;
    dp.n_units = (int32_t)(n_seg * s.n_heads);
    for (int32_t b = 0; b < s.batch; ++b) {
        dp.pos0[b] = sp.pos0[b];
        dp.n_tokens[b] = sp.n_tokens[b];
        dp.row0[b] = sp.row0[b];
        dp.seg_base[b] = sp.seg_base[b];
    }
    int sms = 0;
    if ((st = sm_count(&sms)) != HS_OK)
        return st;
    const int grid = (int)std::min<int64_t>(dp.n_units, 2 * (int64_t)sms);
    if ((st = cuda_status(hs::launch_gla_dstate(dp, (int)D, grid, stream))) != HS_OK)
        return st;

    // the scan: start states, checkpoints, final state
    if ((st = cuda_status(hs::launch_gla_scan(sp, (int)D, stream))) != HS_OK)
        return st;

    // the tensor-core kernel over every segment from its start state Sn, writing the outputs
    // and no state.  Consecutive segments of a problem are grouped into spans, one CTA per
    // (span, head), about one CTA per SM in all; each segment restarts from its own start
    // state, so the grouping changes no result.  At most HS_MAX_BATCH spans per launch.
    const int64_t per_span = std::max<int64_t>(1, (n_seg * s.n_heads + sms - 1) / sms);
    hs::GlaParams p;
    int32_t j = 0;
    auto reset = [&]() {
        std::memset(&p, 0, sizeof p);
        p.q = q;
        p.k = k;
        p.v = v;
        p.log_g = log_g;
        p.o = o;
        p.state = ws_Sn;
        p.d_err = d_err;
        p.n_heads = s.n_heads;
        p.no_state_out = 1;
    };
    auto flush = [&]() -> hs_status {
        if (j == 0)
            return HS_OK;
        p.batch = j;
        const hs_status r = cuda_status(hs::launch_gla_chunked_tc_restart(p, (int)D, stream));
        j = 0;
        reset();
        return r;
    };
    reset();
    for (int32_t b = 0; b < s.batch; ++b) {
        const int64_t end = pos0[b] + n_tokens[b];
        int64_t seg_i = sp.seg_base[b];
        for (int64_t at = pos0[b]; at < end;) {
            // a span of up to per_span segments from `at`
            int64_t e = at, n = 0;
            while (e < end && n < per_span) {
                e = std::min<int64_t>(end, (e / HS_CHUNK + 1) * HS_CHUNK);
                ++n;
            }
            p.pos0[j] = at;
            p.n_tokens[j] = (int32_t)(e - at);
            p.row0[j] = (int32_t)((int64_t)b * s.max_tokens + (at - pos0[b]));
            p.ck_base[j] = (int32_t)seg_i;
            seg_i += n;
            at = e;
            if (++j == HS_MAX_BATCH && (st = flush()) != HS_OK)
                return st;
        }
    }
    return flush();
}

hs_status hs_linattn_prefill_packed(const hs_linattn_shape *shp, const uint16_t *q,
                                    const uint16_t *k, const uint16_t *v, const float *log_g,
                                    float *o, float *state, const int64_t *pos0,
                                    const int32_t *n_tokens, const int64_t *cu_rows,
                                    int32_t ckpt_interval, float *const *ckpt_slots,
                                    int32_t *d_err, cudaStream_t stream)
{
    if (shp != nullptr && shp->batch > 0 && cu_rows == nullptr)
        return HS_ERR_INVALID_ARG;
    return prefill(shp, q, k, v, log_g, o, state, pos0, n_tokens, cu_rows, ckpt_interval,
                   ckpt_slots, d_err, stream);
}

}  // extern "C"
