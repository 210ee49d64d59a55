// Block-table scatter of KV pages from a staging pool into the paged KV cache
// (restoring the attention cache entries of the credited prefix, Section 2.1
// and Section 5.2 of the paper), and the inverse gather of cache pages into a
// staging pool (the save path whose completion Section 3.1 and Table 5 check).
// Staging may be device memory or pinned host memory read or written over
// NVLink-C2C.
//
// Pure HBM copy: every page is a contiguous run of page_bytes bytes on both
// sides, so each CTA moves whole pages with 16-byte vector loads and stores.
// Loads bypass L1 and stores are streaming (evict-first): neither side is
// reused by this kernel.  Several 16-byte loads are in flight per thread
// before the first store so that the copy is limited by bandwidth, not by
// load latency.  The grid is a whole number of waves over the SMs and
// strides over (layer, page) units with pages of one layer adjacent, so
// reads from the staging pool are sequential.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 8;

__device__ __forceinline__ uint4 ld_stream(const uint4 *p)
{
    return __ldcs(p);
}

__device__ __forceinline__ void st_stream(uint4 *p, const uint4 &v)
{
    __stcs(p, v);
}

// Page j of every layer moves between staging slot j and cache block bt[j]:
// cache <- staging when kGather is false, staging <- cache when it is true.
template <bool kGather>
__device__ __forceinline__ void kv_pages(const void *const *staging, void *const *cache_w,
                                         const void *const *cache_r, int32_t n_layers,
                                         const int32_t *bt, int32_t n_pages, int64_t page_vecs,
                                         int64_t num_blocks, int32_t *d_err, void *const *staging_w)
{
    pdl_wait_and_release();
    const int64_t units = (int64_t)n_layers * n_pages;
    for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
        const int32_t l = (int32_t)(u / n_pages);
        const int32_t j = (int32_t)(u - (int64_t)l * n_pages);
        const uint4 *src = static_cast<const uint4 *>(kGather ? cache_r[l] : staging[l]);
        uint4 *dst = static_cast<uint4 *>(kGather ? staging_w[l] : cache_w[l]);
        const int32_t blk = bt[j];
        if (src == nullptr || dst == nullptr) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_NULL);
            continue;
        }
        if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) != 0) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_MISALIGNED);
            continue;
        }
        if (blk < 0 || (int64_t)blk >= num_blocks) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_BLOCK_OOB);
            continue;
        }
        src += (int64_t)(kGather ? blk : j) * page_vecs;
        dst += (int64_t)(kGather ? j : blk) * page_vecs;
        for (int64_t base = threadIdx.x; base < page_vecs; base += (int64_t)kThreads * kUnroll) {
            uint4 r[kUnroll];
#pragma unroll
            for (int x = 0; x < kUnroll; ++x) {
                const int64_t i = base + (int64_t)x * kThreads;
                if (i < page_vecs)
                    r[x] = ld_stream(src + i);
            }
#pragma unroll
            for (int x = 0; x < kUnroll; ++x) {
                const int64_t i = base + (int64_t)x * kThreads;
                if (i < page_vecs)
                    st_stream(dst + i, r[x]);
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads)
kv_scatter_kernel(const void *const *staging, void *const *cache, int32_t n_layers,
                  const int32_t *bt, int32_t n_pages, int64_t page_vecs, int64_t num_blocks,
                  int32_t *d_err)
{
    kv_pages<false>(staging, cache, nullptr, n_layers, bt, n_pages, page_vecs, num_blocks, d_err,
                    nullptr);
}

__global__ void __launch_bounds__(kThreads)
kv_gather_kernel(const void *const *cache, void *const *staging, int32_t n_layers,
                 const int32_t *bt, int32_t n_pages, int64_t page_vecs, int64_t num_blocks,
                 int32_t *d_err)
{
    kv_pages<true>(nullptr, nullptr, cache, n_layers, bt, n_pages, page_vecs, num_blocks, d_err,
                   staging);
}

// Page slices: every page is `rows` rows of row_bytes; the transfer covers bytes
// [col_off, col_off + col_bytes) of each row (one tensor-parallel rank's heads).
// The staging page holds the rows' slices back to back (rows * col_bytes bytes).
// cache <- staging when kGather is false, staging <- cache when it is true.
template <bool kGather>
__global__ void __launch_bounds__(kThreads)
kv_slices_kernel(const void *const *from, void *const *to, int32_t n_layers, const int32_t *bt,
                 int32_t n_pages, int64_t page_bytes, int32_t rows, int64_t row_bytes,
                 int64_t col_off, int32_t col_vecs, int64_t num_blocks, int32_t *d_err)
{
    pdl_wait_and_release();
    const int64_t units = (int64_t)n_layers * n_pages;
    const int32_t vecs = rows * col_vecs;                      // 16-byte vectors per page slice
    for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
        const int32_t l = (int32_t)(u / n_pages);
        const int32_t j = (int32_t)(u - (int64_t)l * n_pages);
        const uint8_t *src = static_cast<const uint8_t *>(from[l]);
        uint8_t *dst = static_cast<uint8_t *>(to[l]);
        const int32_t blk = bt[j];
        if (src == nullptr || dst == nullptr) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_NULL);
            continue;
        }
        if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) != 0) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_MISALIGNED);
            continue;
        }
        if (blk < 0 || (int64_t)blk >= num_blocks) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_BLOCK_OOB);
            continue;
        }
        const uint8_t *cache_page = (kGather ? src : dst) + (int64_t)blk * page_bytes + col_off;
        const int64_t stage_page = (int64_t)j * vecs * 16;
        for (int32_t base = threadIdx.x; base < vecs; base += kThreads * kUnroll) {
            uint4 r[kUnroll];
            int64_t coff[kUnroll];     // byte offset of the vector in the cache page
#pragma unroll
            for (int x = 0; x < kUnroll; ++x) {
                const int32_t i = base + x * kThreads;
                const int32_t row = i / col_vecs;
                coff[x] = (int64_t)row * row_bytes + (int64_t)(i - row * col_vecs) * 16;
                if (i < vecs) {
                    const uint8_t *s = kGather ? cache_page + coff[x] : src + stage_page + (int64_t)i * 16;
                    r[x] = ld_stream(reinterpret_cast<const uint4 *>(s));
                }
            }
#pragma unroll
            for (int x = 0; x < kUnroll; ++x) {
                const int32_t i = base + x * kThreads;
                if (i < vecs) {
                    uint8_t *d = kGather ? dst + stage_page + (int64_t)i * 16
                                         : const_cast<uint8_t *>(cache_page) + coff[x];
                    st_stream(reinterpret_cast<uint4 *>(d), r[x]);
                }
            }
        }
    }
}

// 8 resident CTAs of 256 threads per SM; at most 4 waves, never more CTAs than units
int64_t kv_grid(int32_t n_layers, int32_t n_pages, int sm_count)
{
    const int64_t units = (int64_t)n_layers * n_pages;
    const int64_t grid = (int64_t)sm_count * 8 * 4;
    return grid > units ? units : grid;
}

}  // namespace

cudaError_t launch_kv_gather(const void *const *cache, void *const *staging, int32_t n_layers,
                             const int32_t *bt, int32_t n_pages, int64_t page_bytes,
                             int64_t num_blocks, int32_t *d_err, int sm_count, cudaStream_t s)
{
    const int64_t grid = kv_grid(n_layers, n_pages, sm_count);
    return launch_pdl(kv_gather_kernel, dim3((unsigned)grid), dim3(kThreads), 0, s, cache, staging,
                      n_layers, bt, n_pages, (int64_t)(page_bytes / 16), num_blocks, d_err);
}

cudaError_t launch_kv_slices(bool gather, const void *const *from, void *const *to, int32_t n_layers,
                             const int32_t *bt, int32_t n_pages, int64_t page_bytes, int32_t rows,
                             int64_t col_off, int64_t col_bytes, int64_t num_blocks, int32_t *d_err,
                             int sm_count, cudaStream_t s)
{
    const int64_t grid = kv_grid(n_layers, n_pages, sm_count);
    const int64_t row_bytes = page_bytes / rows;
    if (gather)
        return launch_pdl(kv_slices_kernel<true>, dim3((unsigned)grid), dim3(kThreads), 0, s, from,
                          to, n_layers, bt, n_pages, page_bytes, rows, row_bytes, col_off,
                          (int32_t)(col_bytes / 16), num_blocks, d_err);
    return launch_pdl(kv_slices_kernel<false>, dim3((unsigned)grid), dim3(kThreads), 0, s, from, to,
                      n_layers, bt, n_pages, page_bytes, rows, row_bytes, col_off,
                      (int32_t)(col_bytes / 16), num_blocks, d_err);
}

cudaError_t launch_kv_scatter(const void *const *staging, void *const *cache, int32_t n_layers,
                              const int32_t *bt, int32_t n_pages, int64_t page_bytes,
                              int64_t num_blocks, int32_t *d_err, int sm_count, cudaStream_t s)
{
    const int64_t grid = kv_grid(n_layers, n_pages, sm_count);
    return launch_pdl(kv_scatter_kernel, dim3((unsigned)grid), dim3(kThreads), 0, s, staging, cache,
                      n_layers, bt, n_pages, (int64_t)(page_bytes / 16), num_blocks, d_err);
}

}  // namespace hs
