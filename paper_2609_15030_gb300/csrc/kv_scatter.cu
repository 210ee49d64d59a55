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
// A slice is small (8 KiB for one FP8 rank of four), so the loads of a unit's block id
// and layer pointers, which its data loads depend on, cost about as much as its data:
// each CTA requests the next unit's while it moves the current one.  Slices of at most
// 2 x 256 vectors take the kU = 2 instantiation, 32 registers and 8 resident CTAs per SM
// (twice the bytes in flight), larger ones kU = 4.  Measured on 48 x 256 FP8 slices of 8 KiB
// (one box): 0.60 of the HBM copy peak before (each unit waiting for its own metadata, eight
// vectors per thread, 4 CTAs per SM), 0.62 with the metadata ahead, 0.72 with kU = 2 at 8 CTAs
// per SM; 16 and 32 KiB slices: 0.86 and 0.94 with kU = 4, 0.84 and 0.91 with kU = 2.
struct SliceUnit {
    const uint8_t *src;
    uint8_t *dst;
    int32_t j;     // page index (staging slot)
    int32_t blk;   // cache block
};

template <bool kGather, int kU, int kMinBlocks>
__global__ void __launch_bounds__(kThreads, kMinBlocks)
kv_slices_kernel(const void *const *from, void *const *to, int32_t n_layers, const int32_t *bt,
                 int32_t n_pages, int64_t page_bytes, int32_t rows, int64_t row_bytes,
                 int64_t col_off, int32_t col_vecs, int64_t num_blocks, int32_t *d_err)
{
    pdl_wait_and_release();
    const int64_t units = (int64_t)n_layers * n_pages;
    const int32_t vecs = rows * col_vecs;                      // 16-byte vectors per page slice
    auto unit = [&](int64_t u) -> SliceUnit {
        SliceUnit m;
        const int32_t l = (int32_t)(u / n_pages);
        m.j = (int32_t)(u - (int64_t)l * n_pages);
        m.src = static_cast<const uint8_t *>(from[l]);
        m.dst = static_cast<uint8_t *>(to[l]);
        m.blk = bt[m.j];
        return m;
    };
    int64_t u = blockIdx.x;
    SliceUnit cur;
    if (u < units)
        cur = unit(u);
    while (u < units) {
        const int64_t un = u + gridDim.x;
        SliceUnit nxt = cur;
        if (un < units)
            nxt = unit(un);   // in flight while this unit moves
        const uint8_t *src = cur.src;
        uint8_t *dst = cur.dst;
        bool ok = true;
        if (src == nullptr || dst == nullptr) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_NULL);
            ok = false;
        } else if (((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) != 0) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_MISALIGNED);
            ok = false;
        } else if (cur.blk < 0 || (int64_t)cur.blk >= num_blocks) {
            if (threadIdx.x == 0)
                report(d_err, HS_DEVERR_BLOCK_OOB);
            ok = false;
        }
        if (ok) {
            const uint8_t *cache_page = (kGather ? src : dst) + (int64_t)cur.blk * page_bytes + col_off;
            const int64_t stage_page = (int64_t)cur.j * vecs * 16;
            for (int32_t base = threadIdx.x; base < vecs; base += kThreads * kU) {
                uint4 r[kU];
                int64_t coff[kU];     // byte offset of the vector in the cache page
#pragma unroll
                for (int x = 0; x < kU; ++x) {
                    const int32_t i = base + x * kThreads;
                    const int32_t row = i / col_vecs;
                    coff[x] = (int64_t)row * row_bytes + (int64_t)(i - row * col_vecs) * 16;
                    if (i < vecs) {
                        const uint8_t *sp = kGather ? cache_page + coff[x] : src + stage_page + (int64_t)i * 16;
                        r[x] = ld_stream(reinterpret_cast<const uint4 *>(sp));
                    }
                }
#pragma unroll
                for (int x = 0; x < kU; ++x) {
                    const int32_t i = base + x * kThreads;
                    if (i < vecs) {
                        uint8_t *dp = kGather ? dst + stage_page + (int64_t)i * 16
                                              : const_cast<uint8_t *>(cache_page) + coff[x];
                        st_stream(reinterpret_cast<uint4 *>(dp), r[x]);
                    }
                }
            }
        }
        cur = nxt;
        u = un;
    }
}

// up to 8 resident CTAs of 256 threads per SM; at most 4 waves of 8, never more CTAs than units
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
    const int32_t col_vecs = (int32_t)(col_bytes / 16);
    const bool small = (int64_t)rows * col_vecs <= 2 * kThreads;
    auto kern = gather ? (small ? kv_slices_kernel<true, 2, 8> : kv_slices_kernel<true, 4, 1>)
                       : (small ? kv_slices_kernel<false, 2, 8> : kv_slices_kernel<false, 4, 1>);
    return launch_pdl(kern, dim3((unsigned)grid), dim3(kThreads), 0, s, from, to, n_layers, bt, n_pages,
                      page_bytes, rows, row_bytes, col_off, col_vecs, num_blocks, d_err);
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
