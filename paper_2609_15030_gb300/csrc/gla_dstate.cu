// The first pass of the segment-parallel prefill (hs_linattn_prefill_scan): the state each
// segment of the 64-token absolute position grid reaches from the zero state,
//     dS = sum_j K^_j^T v_j,   K^_j = k_j 2^{Lam_last - Lam_j},
// with Lam the segment's cumulative log2-decay per key dim, so that 2^{Lam_last - Lam_j} is
// the decay from token j to the segment's end.  It is the exact path's state update of the
// tensor-core prefill applied to the zero state.
//
// One unit = one (segment, head).  All 256 threads stage the segment's k, v and log-gates
// in shared memory with cp.async (zeros past the segment's end, which leave the results
// unchanged); a CTA stages its next unit as soon as the current one's operands are built, so
// the copies overlap that unit's products and stores.  Then the 128 key-dim threads walk the 64 tokens backwards, keeping
// Lam_last - Lam_j as a running sum of the later tokens' log2-gates, and write K^ rounded to
// tf32 into a K-major operand (token = K), while the 128 value-dim threads put V^T into TMEM
// (bf16 values, exact in tf32); one thread issues dS^T = V^T K^ as eight M = 128, N = d,
// K = 8 tf32 products; the eight warps read dS^T back from TMEM and store it row by row
// (row = key dim), as the state layout wants.  Each key-dim thread also leaves the segment's
// decay of its row, G_d = 2^{Lam_last} (its final running sum), at element (d, 0) of the
// segment's start-state block, where the scan reads it before it writes the start state
// there.  A unit depends only on its segment's inputs, so resumed and full computations
// produce the same dS and G for a segment.
//
// Each CTA holds 256 TMEM columns (S^T in 0..d-1, V^T in 128..191) and 97 KiB of shared
// memory, so at most two CTAs share an SM and their TMEM allocations always fit.  The
// grid is persistent, each CTA walking units blockIdx.x, + gridDim.x, ...  The wait for the
// products is bounded (1 s): on timeout the CTA reports HS_DEVERR_TIMEOUT, waits once more
// (bounded) for its products, frees its TMEM and returns.
#include "gla_chunk_common.cuh"
#include "gla_dstate.cuh"

namespace hs {
namespace {

using namespace ptx;
using gck::bf16f;
using gck::ex2;
using gck::rna_tf32;
using gck::t_off;

constexpr int kThreads = 256;
constexpr int kChunk = 64;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kTmV = 128;                // V^T: column = token
// shared memory (from a 1024-byte aligned base): the K^ operand (d x 64 tf32) and the
// staged segment; 97 KiB with the alignment slack, so at most two CTAs fit on an SM
constexpr uint32_t OFF_OP = 0;                // K^ operand, K-major, 128-byte swizzle  32 KiB
constexpr uint32_t OFF_K = 32768;             // k  bf16 [64 tokens][d]                 16 KiB
constexpr uint32_t OFF_V = 49152;             // v  bf16 [64][d]                        16 KiB
constexpr uint32_t OFF_A = 65536;             // log-gates f32 [64][d]                  32 KiB
constexpr uint32_t kSmemBytes = 98304 + 1024;
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr float kLog2e = 1.4426950408889634f;

// 16 bytes global -> shared, asynchronous; the first `n` bytes copied, the rest zero-filled
__device__ __forceinline__ void cp_async16_zfill(void *smem_dst, const void *gmem_src, uint32_t n)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(
                     (uint32_t)__cvta_generic_to_shared(smem_dst)),
                 "l"(gmem_src), "r"(n)
                 : "memory");
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
gla_dstate_kernel(const __grid_constant__ DStateParams p)
{
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t s_bar;
    __shared__ uint32_t s_tmem;
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sb = smem_u32(smem);
    const uint32_t bar = smem_u32(&s_bar);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    if (warp == 0)
        tmem_alloc(smem_u32(&s_tmem), kTmemCols);
    pdl_wait_and_release();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = s_tmem;
    const int64_t tstride = (int64_t)p.n_heads * D;     // elements between consecutive tokens
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    constexpr uint32_t idesc = idesc_tf32(128, D, 0, 0);
    uint32_t ph = 0;
    bool aborted = false;

    // where unit u's segment lies: its (segment, head), token count and first element
    struct Unit {
        int g, h, L;
        int64_t base;
    };
    auto unit = [&](int64_t u) -> Unit {
        Unit r;
        r.g = (int)(u / p.n_heads);
        r.h = (int)(u - (int64_t)r.g * p.n_heads);
        // the problem holding segment g: the last b with seg_base[b] <= g (problems without
        // tokens hold no segment and share the next one's seg_base)
        int lo = 0, hi = p.batch - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (p.seg_base[mid] <= r.g)
                lo = mid;
            else
                hi = mid - 1;
        }
        const int64_t pos0 = p.pos0[lo];
        const int64_t chunk = pos0 / kChunk + (r.g - p.seg_base[lo]);
        const int64_t s = max(pos0, chunk * kChunk);
        r.L = (int)(min(pos0 + p.n_tokens[lo], (chunk + 1) * kChunk) - s);
        r.base = ((int64_t)p.row0[lo] + (s - pos0)) * tstride + (int64_t)r.h * D;
        return r;
    };
    // copy a unit's k, v (D/8 vectors per token) and log-gates (D/4) into the staging areas
    // (tokens j >= L zero-filled: no bytes read), as one cp.async group of this thread
    auto stage = [&](const Unit &w) {
        constexpr int VK = D / 8, VA = D / 4;
#pragma unroll
        for (int x = 0; x < 64 * VK / kThreads; ++x) {
            const int i = tid + x * kThreads, j = i / VK, c = i - j * VK;
            const int64_t off = w.base + (int64_t)min(j, w.L - 1) * tstride + c * 8;
            const uint32_t n = j < w.L ? 16u : 0u;
            cp_async16_zfill(smem + OFF_K + i * 16, p.k + off, n);
            cp_async16_zfill(smem + OFF_V + i * 16, p.v + off, n);
        }
#pragma unroll
        for (int x = 0; x < 64 * VA / kThreads; ++x) {
            const int i = tid + x * kThreads, j = i / VA, c = i - j * VA;
            const int64_t off = w.base + (int64_t)min(j, w.L - 1) * tstride + c * 4;
            cp_async16_zfill(smem + OFF_A + i * 16, p.log_g + off, j < w.L ? 16u : 0u);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };

    Unit w = unit(blockIdx.x);
    if ((int64_t)blockIdx.x < p.n_units)
        stage(w);
    for (int64_t u = blockIdx.x; u < p.n_units; u += gridDim.x) {
        const int g = w.g, h = w.h;
        asm volatile("cp.async.wait_all;" ::: "memory");
        __syncthreads();
        if (warp < 4) {
            const int d = tid;
            if (d < D) {
                const uint16_t *sk = reinterpret_cast<const uint16_t *>(smem + OFF_K) + d;
                const float *sa = reinterpret_cast<const float *>(smem + OFF_A) + d;
                float suf = 0.f;   // log2-decay from token j to the segment's end
#pragma unroll 16
                for (int j = kChunk - 1; j >= 0; --j) {
                    *reinterpret_cast<float *>(smem + OFF_OP + t_off(D, d, j)) =
                        rna_tf32(bf16f(sk[j * D]) * ex2(suf));
                    suf = fmaf(sa[j * D], kLog2e, suf);
                }
                p.Sn[((int64_t)g * p.n_heads + h) * D * D + (int64_t)d * D] = ex2(suf);
                fence_proxy_async_smem();
            }
        } else if ((warp & 3) * 32 < D) {
            const int e = (warp & 3) * 32 + lane;
            const uint16_t *sv = reinterpret_cast<const uint16_t *>(smem + OFF_V) + e;
#pragma unroll
            for (int c = 0; c < kChunk; c += 16) {
                uint32_t w[16];
#pragma unroll
                for (int x = 0; x < 16; ++x)
                    w[x] = (uint32_t)sv[(c + x) * D] << 16;
                tmem_st16(tmem + lrow + kTmV + c, w);
            }
            tmem_wait_st();
        }
        tc_fence_before();
        __syncthreads();   // the operands are built: the staging areas are free
        if (tid == 0) {
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < kChunk / 8; ++kk)
                mma_tf32_ts(tmem, tmem + kTmV + kk * 8,
                            sdesc_sw128(sb + OFF_OP + (kk >> 2) * (D * 128) + (kk & 3) * 32, 16, 1024),
                            idesc,
                            kk > 0);
            tc_commit(bar);
        }
        // the next unit's inputs arrive while this one's products and stores run
        if (u + gridDim.x < p.n_units) {
            w = unit(u + gridDim.x);
            stage(w);
        }
        aborted = __syncthreads_or(!mbar_wait_bounded(bar, ph, kTimeoutNs));
        if (aborted)
            break;
        ph ^= 1;
        tc_fence_after();
        if ((warp & 3) * 32 < D) {
            const int e = (warp & 3) * 32 + lane;
            float *dst = p.dS + ((int64_t)g * p.n_heads + h) * D * D + e;
#pragma unroll
            for (int c = 0; c < D / 2; c += 32) {
                const int d0 = (warp >> 2) * (D / 2) + c;
                float r[32];
                tmem_ld32(tmem + lrow + d0, r);
                tmem_wait_ld();
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    dst[(int64_t)(d0 + x) * D] = r[x];
            }
        }
        tc_fence_before();
        __syncthreads();   // TMEM and the operand are free for the next unit
    }
    if (aborted && tid == 0) {
        report(p.d_err, HS_DEVERR_TIMEOUT);
        mbar_wait_bounded(bar, ph, kTimeoutNs);   // the products in flight, before TMEM goes
    }
    asm volatile("cp.async.wait_all;" ::: "memory");   // a staged next unit, after an abort
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

template <int D>
cudaError_t launch_d(const DStateParams &p, int grid, cudaStream_t s)
{
    static std::atomic<uint64_t> smem_set{0};
    return launch_pdl_big_smem(gla_dstate_kernel<D>, dim3(grid), dim3(kThreads), kSmemBytes, s,
                               smem_set, p);
}

}  // namespace

cudaError_t launch_gla_dstate(const DStateParams &p, int d, int grid, cudaStream_t s)
{
    if (p.n_units <= 0 || grid <= 0)
        return cudaSuccess;
    if (d == 128)
        return launch_d<128>(p, grid, s);
    if (d == 64)
        return launch_d<64>(p, grid, s);
    return cudaErrorNotSupported;
}

}  // namespace hs
