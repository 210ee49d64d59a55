// Chunked gated linear attention on tcgen05 tensor cores (sm_103a).
//
// Recurrence (per head):  S_t = diag(g_t) S_{t-1} + k_t v_t^T,  o_t = q_t S_t,
// g_t = exp(a_t).  The paper runs its linear layers on FLA kernels without
// printing their recurrence; this is the form the library implements, in
// the chunked matrix form.  For a segment of L <= 64 tokens inside one
// 64-token chunk of the absolute position grid, with cumulative log2-decay
// Lam_i = log2(e) * sum_{s<=i} a_s (per key dimension):
//
//   Q~_i = q_i * 2^{Lam_i}            K~_j = k_j * 2^{-Lam_j}
//   A_ij = [j <= i] * Q~_i . K~_j     (= sum_d q_id k_jd 2^{Lam_id - Lam_jd})
//   o_i  = Q~_i S + sum_j A_ij v_j
//   S'   = diag(2^{Lam_last}) (S + K~^T V)
//
// One CTA owns one (problem, head) and walks its segments in order; the
// float32 state lives in tensor memory (TMEM) for the whole call, stored
// transposed (lane = value dim e, column = key dim d) so that it is directly
// the A operand of the inter-chunk product.  Per segment:
//   1. TMA stages q, k, v (bf16) and the log-gates (f32) of 64 tokens;
//   2. 256 threads build the tf32 operands in 128-byte-swizzled layouts: each
//      thread scans 32 tokens of one key dimension and the two halves of the
//      chunk are joined with warp shuffles;
//   3. one thread issues the MMAs:  D_A = Q~ K~^T;  D_O = S^T Q~^T (A operand
//      read from TMEM);  D_O += V^T A^T;  S^T += V^T K~  (all kind::tf32 with
//      K-major operands, fp32 accumulators in TMEM);
//   4. the causal mask is applied to D_A between the two groups, outputs are
//      streamed from D_O to global memory, and the state is scaled by
//      2^{Lam_last} column by column (TMEM -> registers -> TMEM); checkpoint
//      slots are written from the same registers.
// The next segment's TMA load is issued as soon as the staging buffers have
// been consumed, so it overlaps the MMAs and the epilogue.
//
// The factorised form needs 2^{-Lam_j} to stay finite: when some key
// dimension decays by more than 2^-64 inside one chunk (zero gates, for
// instance), that chunk computes A elementwise with 2^{Lam_i - Lam_j} <= 1
// and updates the state as diag(2^{Lam_last}) S + K^^T V with
// K^_j = k_j 2^{Lam_last - Lam_j}.  The choice depends only on the chunk's
// own inputs, as does every operation order, so a resumed run reproduces a
// full recomputation bit for bit when it starts on the chunk grid.
//
// Every wait on an mbarrier is bounded (1 s); on timeout the CTA reports
// HS_DEVERR_TIMEOUT, waits (bounded) for its own copies and MMAs in flight,
// frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "hs_internal.cuh"
#include "sm100_ptx.cuh"

namespace hs {
namespace {

using namespace ptx;

constexpr int D = 128;    // d_k = d_v
constexpr int CH = 64;    // chunk length (absolute grid)
constexpr int NT = 256;   // threads per CTA
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kFastMinLog2 = -64.0f;      // factorised form if every 2^{Lam_last} >= 2^-64
constexpr uint64_t kTimeoutNs = 1000000000ull;

// shared memory map (offsets from a 1024-byte aligned base).  Every tf32
// operand is K-major (kind::tf32 takes no transposed shared-memory operand),
// so the products that contract over tokens read V and K~ transposed.
constexpr uint32_t OFF_QT = 0;          // Q~   [64 tok i][128 d]  tf32, swizzled   32 KiB
constexpr uint32_t OFF_KT = 32768;      // K~   [64 tok j][128 d]                   32 KiB
constexpr uint32_t OFF_KTT = 65536;     // K~^T [128 d][64 tok j] (K^^T on the exact path)  32 KiB
constexpr uint32_t OFF_VT = 98304;      // V^T  [128 e][64 tok j]                   32 KiB
constexpr uint32_t OFF_A = 131072;      // A    [64 i][64 j]                        16 KiB
constexpr uint32_t OFF_SQ = 147456;     // staged q  bf16 [64][128]                16 KiB
constexpr uint32_t OFF_SK = 163840;     // staged k                                 16 KiB
constexpr uint32_t OFF_SV = 180224;     // staged v                                 16 KiB
constexpr uint32_t OFF_SG = 196608;     // staged log-gates f32 [64][128]           32 KiB
constexpr uint32_t OFF_GAM = 229376;    // 2^{Lam_last} per key dim                512 B
constexpr uint32_t OFF_BAR = 229888;    // 4 mbarriers
constexpr uint32_t OFF_MISC = 229920;   // TMEM base address, flags
constexpr uint32_t SMEM_BYTES = 229936 + 1024;
constexpr uint32_t STAGE_BYTES = 3 * 16384 + 32768;
constexpr uint32_t SLAB = 64 * 128;     // one 32-column slab of a 64-row operand
constexpr uint32_t SLAB_T = 128 * 128;  // one 32-column slab of a 128-row operand

constexpr uint32_t TMEM_COLS = 256;
constexpr uint32_t TM_S = 0;            // S^T   128 lanes x 128 cols
constexpr uint32_t TM_O = 128;          // D_O   128 lanes x 64 cols (lane e, col i)
constexpr uint32_t TM_A = 192;          // D_A   128 lanes x 64 cols (lanes 0..63 used)

constexpr uint32_t IDESC_N64 = idesc_tf32(128, 64, 0, 0);    // M=128, N=64, K-major x K-major
constexpr uint32_t IDESC_N128 = idesc_tf32(128, 128, 0, 0);  // M=128, N=128

struct TmaMaps {
    CUtensorMap q, k, v, g;
};

// Byte offset of element (row, col) of a row-major f32 operand stored as
// 32-column slabs (128-byte rows) in the 128-byte swizzled K-major canonical
// layout: 16-byte chunk c of row r sits at chunk position c ^ (r % 8).
// sw_off: 64-row operands; sw_off_t: 128-row operands.
__device__ __forceinline__ uint32_t sw_off(int row, int col)
{
    return (uint32_t)((col >> 5) * SLAB + row * 128 + ((((col & 31) >> 2) ^ (row & 7)) << 4) +
                      ((col & 3) << 2));
}

__device__ __forceinline__ uint32_t sw_chunk_t(int row, int col4)
{
    return (uint32_t)((col4 >> 3) * SLAB_T + row * 128 + (((col4 & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ float bf16f(uint16_t x)
{
    return __uint_as_float(((uint32_t)x) << 16);
}

__global__ void __launch_bounds__(NT, 1)
gla_chunked_tc_kernel(const __grid_constant__ GlaParams p, const __grid_constant__ TmaMaps maps)
{
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sb = smem_u32(smem);
    const uint16_t *sQ = reinterpret_cast<const uint16_t *>(smem + OFF_SQ);
    const uint16_t *sK = reinterpret_cast<const uint16_t *>(smem + OFF_SK);
    const uint16_t *sV = reinterpret_cast<const uint16_t *>(smem + OFF_SV);
    float *sG = reinterpret_cast<float *>(smem + OFF_SG);
    float *sGam = reinterpret_cast<float *>(smem + OFF_GAM);
    volatile uint32_t *sMisc = reinterpret_cast<volatile uint32_t *>(smem + OFF_MISC);
    const uint32_t bar_tma = sb + OFF_BAR, bar_a = sb + OFF_BAR + 8, bar_o = sb + OFF_BAR + 16,
                   bar_s = sb + OFF_BAR + 24;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int b = blockIdx.x / p.n_heads;
    const int h = blockIdx.x - b * p.n_heads;
    const int n = p.n_tokens[b];
    if (n <= 0)
        return;
    const int64_t pos0 = p.pos0[b];
    const int64_t end = pos0 + n;
    const int64_t tstride = (int64_t)p.n_heads * D;   // elements between consecutive tokens

    if (tid == 0) {
        mbar_init(bar_tma, 1);
        mbar_init(bar_a, 1);
        mbar_init(bar_o, 1);
        mbar_init(bar_s, 1);
        fence_mbar_init();
        sMisc[1] = 0;   // abort flag
    }
    if (warp == 0)
        tmem_alloc(sb + OFF_MISC, TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sMisc[0];
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = warp >> 2;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e

    // thread-0 bookkeeping of work in flight (for the abort path)
    bool tma_inflight = false;
    uint32_t ph_tma = 0, ph_a = 0, ph_o = 0, ph_s = 0;

    auto issue_tma = [&](int64_t tok_local) {
        const int32_t y = (int32_t)((int64_t)b * p.max_tokens + tok_local);
        const int32_t x = h * D;
        mbar_arrive_expect_tx(bar_tma, STAGE_BYTES);
        tma_load_2d(sb + OFF_SQ, &maps.q, x, y, bar_tma);
        tma_load_2d(sb + OFF_SK, &maps.k, x, y, bar_tma);
        tma_load_2d(sb + OFF_SV, &maps.v, x, y, bar_tma);
        tma_load_2d(sb + OFF_SG, &maps.g, x, y, bar_tma);
        tma_inflight = true;
    };
    if (tid == 0)
        issue_tma(0);

    // incoming state -> TMEM, transposed: S^T[e][d] = state[d][e]
    float *st_g = p.state + ((int64_t)b * p.n_heads + h) * D * D;
    {
        float r[32];
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 32) {
            const int d0 = colhalf * 64 + c0;
#pragma unroll
            for (int x = 0; x < 32; ++x)
                r[x] = st_g[(int64_t)(d0 + x) * D + e_own];
            tmem_st32(tmem + lrow + TM_S + d0, r);
        }
        tmem_wait_st();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    const int C = p.ckpt_interval;
    int64_t pos = pos0, tok = 0;
    bool aborted = false;
    while (pos < end) {
        const int64_t seg_end = min(end, (pos / CH + 1) * CH);
        const int L = (int)(seg_end - pos);
        const bool has_next = seg_end < end;
        const bool ckpt = (C > 0) && (seg_end % C == 0);

        // ---- 1. staged inputs
        if (tid == 0) {
            if (mbar_wait_bounded(bar_tma, ph_tma, kTimeoutNs))
                tma_inflight = false;
            else
                sMisc[1] = 1;
        }
        __syncthreads();
        if (sMisc[1]) {
            aborted = true;
            break;
        }
        ph_tma ^= 1;

        // ---- 2. operands: thread (d, half) scans tokens [32*half, 32*half+32) of key dim d
        const int d = 16 * warp + (lane & 15);
        const int half = lane >> 4;
        const int i0 = half * 32;
        float lam[32];
        float run = 0.f;
#pragma unroll
        for (int x = 0; x < 32; ++x) {
            const int i = i0 + x;
            const float a = (i < L) ? sG[i * D + d] : 0.f;
            run = fmaf(a, kLog2e, run);
            lam[x] = run;
        }
        const float tot_lo = __shfl_sync(0xffffffffu, run, lane & 15);
        const float tot_hi = __shfl_sync(0xffffffffu, run, (lane & 15) + 16);
        if (half) {
#pragma unroll
            for (int x = 0; x < 32; ++x)
                lam[x] = tot_lo + lam[x];
        }
        const float lam_last = tot_lo + tot_hi;
        if (half == 0)
            sGam[d] = exp2f(lam_last);
        const bool slow = __syncthreads_or(lam_last < kFastMinLog2) != 0;

#pragma unroll
        for (int x4 = 0; x4 < 32; x4 += 4) {
            float4 kt4, vt4;
            float *ktv = reinterpret_cast<float *>(&kt4), *vtv = reinterpret_cast<float *>(&vt4);
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int x = x4 + u;
                const int i = i0 + x;
                const bool valid = i < L;
                const float qv = valid ? bf16f(sQ[i * D + d]) : 0.f;
                const float kv = valid ? bf16f(sK[i * D + d]) : 0.f;
                const float l = lam[x];
                const uint32_t o = sw_off(i, d);
                *reinterpret_cast<float *>(smem + OFF_QT + o) = to_tf32(qv * exp2f(l));
                if (slow) {
                    ktv[u] = to_tf32(kv * exp2f(lam_last - l));   // K^ = k 2^{Lam_last - Lam}
                    sG[i * D + d] = l;    // cumulative log2-gates, in place, for the exact path
                } else {
                    const float kt = to_tf32(kv * exp2f(-l));
                    *reinterpret_cast<float *>(smem + OFF_KT + o) = kt;
                    ktv[u] = kt;
                }
                vtv[u] = valid ? bf16f(sV[i * D + d]) : 0.f;
            }
            const uint32_t ot = sw_chunk_t(d, (i0 + x4) >> 2);
            *reinterpret_cast<float4 *>(smem + OFF_KTT + ot) = kt4;
            *reinterpret_cast<float4 *>(smem + OFF_VT + ot) = vt4;
        }
        fence_proxy_async_smem();
        __syncthreads();

        // ---- 3a. first MMA group
        if (tid == 0) {
            tc_fence_after();
            if (!slow) {
#pragma unroll
                for (int kk = 0; kk < D / 8; ++kk) {
                    const uint32_t koff = (kk >> 2) * SLAB + (kk & 3) * 32;
                    mma_tf32_ss(tmem + TM_A, sdesc_sw128(sb + OFF_QT + koff, 16, 1024),
                                sdesc_sw128(sb + OFF_KT + koff, 16, 1024), IDESC_N64, kk > 0);
                }
                tc_commit(bar_a);
            }
#pragma unroll
            for (int kk = 0; kk < D / 8; ++kk) {
                const uint32_t koff = (kk >> 2) * SLAB + (kk & 3) * 32;
                mma_tf32_ts(tmem + TM_O, tmem + TM_S + kk * 8,
                            sdesc_sw128(sb + OFF_QT + koff, 16, 1024), IDESC_N64, kk > 0);
            }
            if (!slow && has_next)
                issue_tma(tok + L);
        }

        // ---- 3b. the masked intra-chunk matrix A -> shared memory (tf32, K-major)
        if (!slow) {
            if (tid == 0 && !mbar_wait_bounded(bar_a, ph_a, kTimeoutNs))
                sMisc[1] = 1;
            __syncthreads();
            if (sMisc[1]) {
                aborted = true;
                break;
            }
            ph_a ^= 1;
            tc_fence_after();
            if (warp < 2) {
                const int i = warp * 32 + lane;      // TMEM lane = query row
                float r[2][32];
                tmem_ld32(tmem + lrow + TM_A, r[0]);
                tmem_ld32(tmem + lrow + TM_A + 32, r[1]);
                tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    float4 w;
                    float *wv = reinterpret_cast<float *>(&w);
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int j = 4 * c + u;
                        wv[u] = (j <= i && i < L) ? to_tf32(r[j >> 5][j & 31]) : 0.f;
                    }
                    const uint32_t o = (c >> 3) * SLAB + i * 128 + (((c & 7) ^ (i & 7)) << 4);
                    *reinterpret_cast<float4 *>(smem + OFF_A + o) = w;
                }
            }
        } else {
            // exact elementwise path: A_ij = sum_d q_id k_jd 2^{Lam_id - Lam_jd}, j <= i < L
            for (int idx = tid; idx < CH * CH; idx += NT) {
                const int i = idx >> 6, j = idx & 63;
                float acc = 0.f;
                if (j <= i && i < L) {
                    for (int dd = 0; dd < D; ++dd)
                        acc = fmaf(bf16f(sQ[i * D + dd]) * bf16f(sK[j * D + dd]),
                                   exp2f(sG[i * D + dd] - sG[j * D + dd]), acc);
                }
                *reinterpret_cast<float *>(smem + OFF_A + sw_off(i, j)) = to_tf32(acc);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();

        // ---- 3c. second MMA group
        if (tid == 0) {
            tc_fence_after();
            if (slow && has_next)
                issue_tma(tok + L);
#pragma unroll
            for (int kk = 0; kk < CH / 8; ++kk) {
                const uint64_t va = sdesc_sw128(sb + OFF_VT + (kk >> 2) * SLAB_T + (kk & 3) * 32, 16, 1024);
                const uint32_t koff = (kk >> 2) * SLAB + (kk & 3) * 32;
                mma_tf32_ss(tmem + TM_O, va, sdesc_sw128(sb + OFF_A + koff, 16, 1024), IDESC_N64, 1);
            }
            if (!slow) {
#pragma unroll
                for (int kk = 0; kk < CH / 8; ++kk) {
                    const uint32_t koff = (kk >> 2) * SLAB_T + (kk & 3) * 32;
                    mma_tf32_ss(tmem + TM_S, sdesc_sw128(sb + OFF_VT + koff, 16, 1024),
                                sdesc_sw128(sb + OFF_KTT + koff, 16, 1024), IDESC_N128, 1);
                }
            }
            tc_commit(bar_o);
            if (!mbar_wait_bounded(bar_o, ph_o, kTimeoutNs))
                sMisc[1] = 1;
        }
        __syncthreads();
        if (sMisc[1]) {
            aborted = true;
            break;
        }
        ph_o ^= 1;
        tc_fence_after();

        // ---- 4a. outputs: lane e holds o[i][e] for 32 rows i
        {
            float r[32];
            const int ib = colhalf * 32;
            tmem_ld32(tmem + lrow + TM_O + ib, r);
            tmem_wait_ld();
            float *op = p.o + (((int64_t)b * p.max_tokens + tok) * p.n_heads + h) * D + e_own;
#pragma unroll
            for (int x = 0; x < 32; ++x)
                if (ib + x < L)
                    __stcs(op + (int64_t)(ib + x) * tstride, r[x]);
        }

        // ---- 4b. state decay (after the update on the factorised path, before it on the exact path)
        float *slot = nullptr;
        if (ckpt && p.ckpt_slots != nullptr) {
            const int64_t idx = p.ck_base[b] + (seg_end / C - pos0 / C - 1);
            slot = p.ckpt_slots[idx];
            if (slot == nullptr || (reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
                if (tid == 0)
                    report(p.d_err, slot == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
                slot = nullptr;
            } else {
                slot += (int64_t)h * D * D;
            }
        }
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 32) {
            const int d0 = colhalf * 64 + c0;
            float r[32];
            tmem_ld32(tmem + lrow + TM_S + d0, r);
            tmem_wait_ld();
#pragma unroll
            for (int x = 0; x < 32; ++x)
                r[x] *= sGam[d0 + x];
            tmem_st32(tmem + lrow + TM_S + d0, r);
            if (!slow && slot != nullptr) {
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    slot[(int64_t)(d0 + x) * D + e_own] = r[x];
            }
        }
        tmem_wait_st();
        if (slow) {
            tc_fence_before();
            __syncthreads();
            if (tid == 0) {
                tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < CH / 8; ++kk) {
                    const uint32_t koff = (kk >> 2) * SLAB_T + (kk & 3) * 32;
                    mma_tf32_ss(tmem + TM_S, sdesc_sw128(sb + OFF_VT + koff, 16, 1024),
                                sdesc_sw128(sb + OFF_KTT + koff, 16, 1024), IDESC_N128, 1);
                }
                tc_commit(bar_s);
                if (!mbar_wait_bounded(bar_s, ph_s, kTimeoutNs))
                    sMisc[1] = 1;
            }
            __syncthreads();
            if (sMisc[1]) {
                aborted = true;
                break;
            }
            ph_s ^= 1;
            tc_fence_after();
            if (slot != nullptr) {
#pragma unroll
                for (int c0 = 0; c0 < 64; c0 += 32) {
                    const int d0 = colhalf * 64 + c0;
                    float r[32];
                    tmem_ld32(tmem + lrow + TM_S + d0, r);
                    tmem_wait_ld();
#pragma unroll
                    for (int x = 0; x < 32; ++x)
                        slot[(int64_t)(d0 + x) * D + e_own] = r[x];
                }
            }
        }
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        pos = seg_end;
        tok += L;
    }

    if (!aborted) {
        // final state back to global memory, row = key dim
        float r[32];
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 32) {
            const int d0 = colhalf * 64 + c0;
            tmem_ld32(tmem + lrow + TM_S + d0, r);
            tmem_wait_ld();
#pragma unroll
            for (int x = 0; x < 32; ++x)
                st_g[(int64_t)(d0 + x) * D + e_own] = r[x];
        }
    } else if (tid == 0) {
        report(p.d_err, HS_DEVERR_TIMEOUT);
        // let this CTA's own copies and MMAs drain (bounded) before its memory goes away
        if (tma_inflight)
            mbar_wait_bounded(bar_tma, ph_tma, kTimeoutNs);
        tc_commit(bar_s);
        mbar_wait_bounded(bar_s, ph_s, kTimeoutNs);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    // resolved once per process from the driver; a pure function pointer
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (fn == nullptr) {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

bool encode_rows(CUtensorMap *m, CUtensorMapDataType dt, const void *base, uint64_t inner,
                 uint64_t rows, uint32_t elem)
{
    auto fn = encode_fn();
    if (fn == nullptr)
        return false;
    cuuint64_t gdim[2] = {inner, rows};
    cuuint64_t gstride[1] = {inner * elem};
    cuuint32_t box[2] = {(cuuint32_t)D, (cuuint32_t)CH};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, dt, 2, const_cast<void *>(base), gdim, gstride, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool gla_chunked_tc_supported(int d, int64_t batch, int64_t max_tokens)
{
    return d == D && batch * max_tokens < ((int64_t)1 << 31);
}

cudaError_t launch_gla_chunked_tc(const GlaParams &p, int d, cudaStream_t s)
{
    if (!gla_chunked_tc_supported(d, p.batch, p.max_tokens))
        return cudaErrorNotSupported;
    TmaMaps maps;
    const uint64_t inner = (uint64_t)p.n_heads * D;
    const uint64_t rows = (uint64_t)p.batch * (uint64_t)p.max_tokens;
    if (rows == 0)
        return cudaSuccess;
    if (!encode_rows(&maps.q, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, p.q, inner, rows, 2) ||
        !encode_rows(&maps.k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, p.k, inner, rows, 2) ||
        !encode_rows(&maps.v, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, p.v, inner, rows, 2) ||
        !encode_rows(&maps.g, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, p.log_g, inner, rows, 4))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(gla_chunked_tc_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
    if (e != cudaSuccess)
        return e;
    const unsigned grid = (unsigned)p.batch * (unsigned)p.n_heads;
    gla_chunked_tc_kernel<<<grid, NT, SMEM_BYTES, s>>>(p, maps);
    return cudaGetLastError();
}

}  // namespace hs
