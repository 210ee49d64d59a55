// Restore of one resumed request in a single launch: the KV pages of the
// credited prefix scattered into the paged cache by block table (Section 2.1,
// Section 5.2 of the paper) and the float32 recurrent states copied from their
// checkpoint slots into the live states (Section 1, Section 2.2).
//
// The grid strides over one list of units: every state is split into 64 KiB
// pieces and every (layer, page) is one unit, state pieces first.  Each unit is
// a contiguous copy with eight 16-byte loads in flight per thread before the
// first store.  Sources are read with evict-first loads (neither the staging
// pool nor the checkpoint is reused here); KV pages are written with streaming
// stores, states with ordinary stores, so that the prefill that follows finds
// the live states in L2.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 8;
constexpr int64_t kPieceVecs = 4096;    // 64 KiB of a state per unit

template <bool kStream>
__device__ __forceinline__ void copy_vecs(const uint4 *src, uint4 *dst, int64_t nv)
{
    for (int64_t base = threadIdx.x; base < nv; base += (int64_t)kThreads * kUnroll) {
        uint4 r[kUnroll];
#pragma unroll
        for (int x = 0; x < kUnroll; ++x) {
            const int64_t i = base + (int64_t)x * kThreads;
            if (i < nv)
                r[x] = __ldcs(src + i);
        }
#pragma unroll
        for (int x = 0; x < kUnroll; ++x) {
            const int64_t i = base + (int64_t)x * kThreads;
            if (i < nv) {
                if (kStream)
                    __stcs(dst + i, r[x]);
                else
                    dst[i] = r[x];
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads)
restore_request_kernel(const void *const *staging, void *const *cache, int32_t n_layers,
                       const int32_t *bt, int32_t n_pages, int64_t page_vecs, int64_t num_blocks,
                       const float *const *src_slots, float *const *dst_slots, int32_t n_slots,
                       int64_t slot_vecs, int64_t pieces, int32_t *d_err)
{
    pdl_wait_and_release();
    const int64_t units_st = (int64_t)n_slots * pieces;
    const int64_t units = units_st + (int64_t)n_layers * n_pages;
    for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
        if (u < units_st) {
            const int32_t i = (int32_t)(u / pieces);
            const int64_t p = u - (int64_t)i * pieces;
            const float *s = src_slots[i];
            float *d = dst_slots[i];
            if (s == nullptr || d == nullptr) {
                if (threadIdx.x == 0 && p == 0)
                    report(d_err, HS_DEVERR_NULL);
                continue;
            }
            if (((reinterpret_cast<uintptr_t>(s) | reinterpret_cast<uintptr_t>(d)) & 15u) != 0) {
                if (threadIdx.x == 0 && p == 0)
                    report(d_err, HS_DEVERR_MISALIGNED);
                continue;
            }
            const int64_t lo = p * kPieceVecs;
            const int64_t nv = (slot_vecs - lo < kPieceVecs) ? slot_vecs - lo : kPieceVecs;
            copy_vecs<false>(reinterpret_cast<const uint4 *>(s) + lo, reinterpret_cast<uint4 *>(d) + lo,
                             nv);
            continue;
        }
        const int64_t w = u - units_st;
        const int32_t l = (int32_t)(w / n_pages);
        const int32_t j = (int32_t)(w - (int64_t)l * n_pages);
        const uint4 *src = static_cast<const uint4 *>(staging[l]);
        uint4 *dst = static_cast<uint4 *>(cache[l]);
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
        copy_vecs<true>(src + (int64_t)j * page_vecs, dst + (int64_t)blk * page_vecs, page_vecs);
    }
}

}  // namespace

cudaError_t launch_restore_request(const void *const *staging, void *const *cache, int32_t n_layers,
                                   const int32_t *bt, int32_t n_pages, int64_t page_bytes,
                                   int64_t num_blocks, const float *const *src_slots,
                                   float *const *dst_slots, int32_t n_slots, int64_t floats_each,
                                   int32_t *d_err, int sm_count, cudaStream_t s)
{
    const int64_t slot_vecs = floats_each / 4;
    const int64_t pieces = (slot_vecs + kPieceVecs - 1) / kPieceVecs;
    const int64_t units = (int64_t)n_slots * pieces + (int64_t)n_layers * n_pages;
    // 8 resident CTAs of 256 threads per SM; at most 4 waves, never more CTAs than units
    int64_t grid = (int64_t)sm_count * 8 * 4;
    if (grid > units)
        grid = units;
    if (grid == 0)
        return cudaSuccess;
    return launch_pdl(restore_request_kernel, dim3((unsigned)grid), dim3(kThreads), 0, s, staging,
                      cache, n_layers, bt, n_pages, page_bytes / 16, num_blocks, src_slots,
                      dst_slots, n_slots, slot_vecs, pieces, d_err);
}

}  // namespace hs
