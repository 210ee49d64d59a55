// Bit-exact copy of float32 recurrent states between live buffers and
// checkpoint slots: the state restore of Section 1 / Section 2.2 of the paper
// and the standalone checkpoint writer (Table 1: a checkpoint every C tokens).
//
// Each slot is split into 64 KiB pieces so that a handful of large states
// still spreads over every SM.  16-byte aligned slot pairs take 16-byte
// vector loads/stores, eight in flight per thread before the first store;
// any other pair falls back to 4-byte accesses.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kThreads = 256;
constexpr int64_t kPieceFloats = 16384;  // 64 KiB
constexpr int kUnroll = 8;

__global__ void __launch_bounds__(kThreads)
slot_copy_kernel(const float *const *src, float *const *dst, int32_t n, int64_t floats_each,
                 int64_t pieces, int32_t *d_err)
{
    pdl_wait_and_release();
    const int64_t units = (int64_t)n * pieces;
    for (int64_t u = blockIdx.x; u < units; u += gridDim.x) {
        const int32_t i = (int32_t)(u / pieces);
        const int64_t p = u - (int64_t)i * pieces;
        const float *s = src[i];
        float *d = dst[i];
        if (s == nullptr || d == nullptr) {
            if (threadIdx.x == 0 && p == 0)
                report(d_err, HS_DEVERR_NULL);
            continue;
        }
        const int64_t lo = p * kPieceFloats;
        int64_t hi = lo + kPieceFloats;
        if (hi > floats_each)
            hi = floats_each;
        const bool vec = (((reinterpret_cast<uintptr_t>(s) | reinterpret_cast<uintptr_t>(d)) & 15u) == 0)
                         && (floats_each % 4 == 0);
        if (vec) {
            const float4 *s4 = reinterpret_cast<const float4 *>(s + lo);
            float4 *d4 = reinterpret_cast<float4 *>(d + lo);
            const int64_t nv = (hi - lo) / 4;
            for (int64_t base = threadIdx.x; base < nv; base += (int64_t)kThreads * kUnroll) {
                float4 r[kUnroll];
#pragma unroll
                for (int x = 0; x < kUnroll; ++x) {
                    const int64_t e = base + (int64_t)x * kThreads;
                    if (e < nv)
                        r[x] = __ldcs(s4 + e);
                }
#pragma unroll
                for (int x = 0; x < kUnroll; ++x) {
                    const int64_t e = base + (int64_t)x * kThreads;
                    if (e < nv)
                        __stcs(d4 + e, r[x]);
                }
            }
        } else {
            for (int64_t e = lo + threadIdx.x; e < hi; e += kThreads)
                d[e] = s[e];
        }
    }
}

}  // namespace

cudaError_t launch_slot_copy(const float *const *src, float *const *dst, int32_t n,
                             int64_t floats_each, int32_t *d_err, int sm_count, cudaStream_t s)
{
    const int64_t pieces = (floats_each + kPieceFloats - 1) / kPieceFloats;
    const int64_t units = (int64_t)n * pieces;
    int64_t grid = (int64_t)sm_count * 8 * 2;
    if (grid > units)
        grid = units;
    return launch_pdl(slot_copy_kernel, dim3((unsigned)grid), dim3(kThreads), 0, s, src, dst, n,
                      floats_each, pieces, d_err);
}

}  // namespace hs
