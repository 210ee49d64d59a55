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
constexpr int kShort = 8; // segments of at most this many tokens run token by token
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
__device__ __forceinline__ uint32_t sw_off(int row, int col)
{
    return (uint32_t)((col >> 5) * SLAB + row * 128 + ((((col & 31) >> 2) ^ (row & 7)) << 4) +
                      ((col & 3) << 2));
}

// 16-byte chunk col4 (columns 4*col4 .. 4*col4+3) of row `row` of a 128-row operand
__device__ __forceinline__ uint32_t sw_chunk_t(int row, int col4)
{
    return (uint32_t)((col4 >> 3) * SLAB_T + row * 128 + (((col4 & 7) ^ (row & 7)) << 4));
}

__device__ __forceinline__ float bf16f(uint16_t x)
{
    return __uint_as_float(((uint32_t)x) << 16);
}

__device__ __forceinline__ float bf_lo(uint32_t w)
{
    return __uint_as_float(w << 16);
}

__device__ __forceinline__ float bf_hi(uint32_t w)
{
    return __uint_as_float(w & 0xFFFF0000u);
}

// 2^x, one MUFU op (relative error ~2^-22; inputs here lie in [-2^7, 2^7])
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// round to tf32 (nearest, ties away from zero) with integer ops; low 13 bits cleared
__device__ __forceinline__ float rna_tf32(float x)
{
    return __uint_as_float((__float_as_uint(x) + 0x1000u) & 0xFFFFE000u);
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
    pdl_wait_and_release();
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

    // operand-building map: thread owns key dims (dp, dp+1) of tokens [16*qr, 16*qr+16)
    const int qr = lane >> 3;
    const int dp = 2 * (warp * 8 + (lane & 7));
    uint32_t nat[8];       // byte offset of (row 16*qr + r, col dp) in a 64-row operand
    {
        const uint32_t base = (uint32_t)((dp >> 5) * SLAB + (16 * qr) * 128 + ((dp & 3) << 2));
        const int cd = (dp & 31) >> 2;
#pragma unroll
        for (int r = 0; r < 8; ++r)
            nat[r] = base + r * 128 + ((uint32_t)(cd ^ r) << 4);
    }
    uint32_t tr0[4], tr1[4];   // 16-byte chunk (tokens 16*qr + 4g ..) of rows dp, dp+1 of a 128-row operand
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        tr0[g] = sw_chunk_t(dp, 4 * qr + g);
        tr1[g] = sw_chunk_t(dp + 1, 4 * qr + g);
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
        float *slot = nullptr;     // checkpoint slot of this segment's end, if any
        if (C > 0 && seg_end % C == 0 && p.ckpt_slots != nullptr) {
            slot = p.ckpt_slots[p.ck_base[b] + (seg_end / C - pos0 / C - 1)];
            if (slot == nullptr || (reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
                if (tid == 0)
                    report(p.d_err, slot == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
                slot = nullptr;
            } else {
                slot += (int64_t)h * D * D;
            }
        }

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

        if (L <= kShort) {
            // ---- short segment: the per-token recurrence with the recurrent kernel's exact
            // operation order (fma chains over groups of 16 key rows, group partials summed
            // left to right), so both kernels agree bit for bit
            for (int idx = tid; idx < L * D; idx += NT)
                sG[idx] = expf(sG[idx]);
            __syncthreads();
            float S[64];
            tmem_ld32(tmem + lrow + TM_S + colhalf * 64, *reinterpret_cast<float(*)[32]>(&S[0]));
            tmem_ld32(tmem + lrow + TM_S + colhalf * 64 + 32, *reinterpret_cast<float(*)[32]>(&S[32]));
            tmem_wait_ld();
            float *part = reinterpret_cast<float *>(smem + OFF_QT);   // [kShort][8 groups][128]
            for (int i = 0; i < L; ++i) {
                const float ve = bf16f(sV[i * D + e_own]);
#pragma unroll
                for (int m = 0; m < 4; ++m) {
                    float acc = 0.f;
#pragma unroll
                    for (int r = 16 * m; r < 16 * m + 16; ++r) {
                        const int d = colhalf * 64 + r;
                        S[r] = fmaf(sG[i * D + d], S[r], bf16f(sK[i * D + d]) * ve);
                        acc = fmaf(bf16f(sQ[i * D + d]), S[r], acc);
                    }
                    part[(i * 8 + colhalf * 4 + m) * D + e_own] = acc;
                }
            }
            tmem_st32(tmem + lrow + TM_S + colhalf * 64, *reinterpret_cast<float(*)[32]>(&S[0]));
            tmem_st32(tmem + lrow + TM_S + colhalf * 64 + 32, *reinterpret_cast<float(*)[32]>(&S[32]));
            if (slot != nullptr) {
#pragma unroll
                for (int r = 0; r < 64; ++r)
                    slot[(int64_t)(colhalf * 64 + r) * D + e_own] = S[r];
            }
            tmem_wait_st();
            fence_proxy_async_smem();
            __syncthreads();
            if (tid == 0 && has_next)
                issue_tma(tok + L);
            float *ob = p.o + (((int64_t)b * p.max_tokens + tok) * p.n_heads + h) * D;
            for (int idx = tid; idx < L * D; idx += NT) {
                const int i = idx >> 7, e = idx & (D - 1);
                float sum = part[(i * 8) * D + e];
#pragma unroll
                for (int g = 1; g < 8; ++g)
                    sum += part[(i * 8 + g) * D + e];
                ob[(int64_t)i * tstride + e] = sum;
            }
            tc_fence_before();
            __syncthreads();
            tc_fence_after();
            pos = seg_end;
            tok += L;
            continue;
        }

        if (L < CH) {
            // zero the staged rows past the segment: every operand row >= L becomes 0
            for (int idx = tid; idx < (CH - L) * 80; idx += NT) {
                const int row = L + idx / 80, c = idx % 80;
                uint4 *dst;
                if (c < 16)
                    dst = reinterpret_cast<uint4 *>(smem + OFF_SQ + row * 256) + c;
                else if (c < 32)
                    dst = reinterpret_cast<uint4 *>(smem + OFF_SK + row * 256) + (c - 16);
                else if (c < 48)
                    dst = reinterpret_cast<uint4 *>(smem + OFF_SV + row * 256) + (c - 32);
                else
                    dst = reinterpret_cast<uint4 *>(smem + OFF_SG + row * 512) + (c - 48);
                *dst = make_uint4(0u, 0u, 0u, 0u);
            }
            __syncthreads();
        }

        // ---- 2. cumulative log2-gates: 16 tokens per thread, then a shuffle scan
        //         over the four token quarters that hold the same key dims
        float lam0[16], lam1[16];
        float run0 = 0.f, run1 = 0.f;
#pragma unroll
        for (int x = 0; x < 16; ++x) {
            const float2 a2 = *reinterpret_cast<const float2 *>(sG + (16 * qr + x) * D + dp);
            run0 = fmaf(a2.x, kLog2e, run0);
            run1 = fmaf(a2.y, kLog2e, run1);
            lam0[x] = run0;
            lam1[x] = run1;
        }
        float s0 = run0, s1 = run1;
        {
            const float y0 = __shfl_up_sync(0xffffffffu, s0, 8);
            const float y1 = __shfl_up_sync(0xffffffffu, s1, 8);
            if (qr >= 1) {
                s0 = s0 + y0;
                s1 = s1 + y1;
            }
        }
        {
            const float y0 = __shfl_up_sync(0xffffffffu, s0, 16);
            const float y1 = __shfl_up_sync(0xffffffffu, s1, 16);
            if (qr >= 2) {
                s0 = s0 + y0;
                s1 = s1 + y1;
            }
        }
        const float pre0 = __shfl_up_sync(0xffffffffu, s0, 8);   // tokens before this quarter
        const float pre1 = __shfl_up_sync(0xffffffffu, s1, 8);
        const float last0 = __shfl_sync(0xffffffffu, s0, (lane & 7) + 24);
        const float last1 = __shfl_sync(0xffffffffu, s1, (lane & 7) + 24);
        if (qr >= 1) {
#pragma unroll
            for (int x = 0; x < 16; ++x) {
                lam0[x] = pre0 + lam0[x];
                lam1[x] = pre1 + lam1[x];
            }
        }
        if (qr == 0)
            *reinterpret_cast<float2 *>(sGam + dp) = make_float2(ex2(last0), ex2(last1));
        const bool slow = __syncthreads_or(last0 < kFastMinLog2 || last1 < kFastMinLog2) != 0;

        // ---- operands (tf32, K-major, swizzled)
        if (!slow) {
#pragma unroll
            for (int g = 0; g < 4; ++g) {
                float4 kt0, kt1, vt0, vt1;
                float *k0 = &kt0.x, *k1 = &kt1.x, *v0 = &vt0.x, *v1 = &vt1.x;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int x = 4 * g + u;
                    const int i = 16 * qr + x;
                    const uint32_t q2 = *reinterpret_cast<const uint32_t *>(sQ + i * D + dp);
                    const uint32_t k2 = *reinterpret_cast<const uint32_t *>(sK + i * D + dp);
                    const uint32_t v2 = *reinterpret_cast<const uint32_t *>(sV + i * D + dp);
                    const uint32_t off = nat[x & 7] + (x >> 3) * 1024;
                    *reinterpret_cast<float2 *>(smem + OFF_QT + off) =
                        make_float2(rna_tf32(bf_lo(q2) * ex2(lam0[x])), rna_tf32(bf_hi(q2) * ex2(lam1[x])));
                    const float ka = rna_tf32(bf_lo(k2) * ex2(-lam0[x]));
                    const float kb = rna_tf32(bf_hi(k2) * ex2(-lam1[x]));
                    *reinterpret_cast<float2 *>(smem + OFF_KT + off) = make_float2(ka, kb);
                    k0[u] = ka;
                    k1[u] = kb;
                    v0[u] = bf_lo(v2);
                    v1[u] = bf_hi(v2);
                }
                *reinterpret_cast<float4 *>(smem + OFF_KTT + tr0[g]) = kt0;
                *reinterpret_cast<float4 *>(smem + OFF_KTT + tr1[g]) = kt1;
                *reinterpret_cast<float4 *>(smem + OFF_VT + tr0[g]) = vt0;
                *reinterpret_cast<float4 *>(smem + OFF_VT + tr1[g]) = vt1;
            }
        } else {
#pragma unroll 1
            for (int g = 0; g < 4; ++g) {
                float4 kt0, kt1, vt0, vt1;
                float *k0 = &kt0.x, *k1 = &kt1.x, *v0 = &vt0.x, *v1 = &vt1.x;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int x = 4 * g + u;
                    const int i = 16 * qr + x;
                    float la, lb;
                    // dynamic index into lam (exact path only)
#pragma unroll
                    for (int z = 0; z < 16; ++z)
                        if (z == x) {
                            la = lam0[z];
                            lb = lam1[z];
                        }
                    const uint32_t q2 = *reinterpret_cast<const uint32_t *>(sQ + i * D + dp);
                    const uint32_t k2 = *reinterpret_cast<const uint32_t *>(sK + i * D + dp);
                    const uint32_t v2 = *reinterpret_cast<const uint32_t *>(sV + i * D + dp);
                    *reinterpret_cast<float2 *>(smem + OFF_QT + sw_off(i, dp)) =
                        make_float2(rna_tf32(bf_lo(q2) * ex2(la)), rna_tf32(bf_hi(q2) * ex2(lb)));
                    k0[u] = rna_tf32(bf_lo(k2) * ex2(last0 - la));   // K^ = k 2^{Lam_last - Lam}
                    k1[u] = rna_tf32(bf_hi(k2) * ex2(last1 - lb));
                    v0[u] = bf_lo(v2);
                    v1[u] = bf_hi(v2);
                    *reinterpret_cast<float2 *>(sG + i * D + dp) = make_float2(la, lb);
                }
                *reinterpret_cast<float4 *>(smem + OFF_KTT + sw_chunk_t(dp, 4 * qr + g)) = kt0;
                *reinterpret_cast<float4 *>(smem + OFF_KTT + sw_chunk_t(dp + 1, 4 * qr + g)) = kt1;
                *reinterpret_cast<float4 *>(smem + OFF_VT + sw_chunk_t(dp, 4 * qr + g)) = vt0;
                *reinterpret_cast<float4 *>(smem + OFF_VT + sw_chunk_t(dp + 1, 4 * qr + g)) = vt1;
            }
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

        // ---- 3b. the causally masked intra-chunk matrix A -> shared memory
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
            if ((warp & 3) < 2) {
                const int i = (warp & 3) * 32 + lane;      // TMEM lane = query row
                const int jb = (warp >> 2) * 32;            // this warp's 32 key columns
                float r[32];
                tmem_ld32(tmem + lrow + TM_A + jb, r);
                tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < 8; ++c) {
                    float4 w;
                    float *wv = &w.x;
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        wv[u] = (jb + 4 * c + u <= i) ? rna_tf32(r[4 * c + u]) : 0.f;
                    const uint32_t o = (jb >> 5) * SLAB + i * 128 + ((uint32_t)(c ^ (i & 7)) << 4);
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
                                   ex2(sG[i * D + dd] - sG[j * D + dd]), acc);
                }
                *reinterpret_cast<float *>(smem + OFF_A + sw_off(i, j)) = rna_tf32(acc);
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
            float *op = p.o + (((int64_t)b * p.max_tokens + tok + ib) * p.n_heads + h) * D + e_own;
            if (L == CH) {
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    __stcs(op + (int64_t)x * tstride, r[x]);
            } else {
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    if (ib + x < L)
                        __stcs(op + (int64_t)x * tstride, r[x]);
            }
        }

        // ---- 4b. state decay (after the update on the factorised path, before it on the exact path)
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 32) {
            const int d0 = colhalf * 64 + c0;
            float r[32];
            tmem_ld32(tmem + lrow + TM_S + d0, r);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const float4 g4 = *reinterpret_cast<const float4 *>(sGam + d0 + 4 * c);
                r[4 * c] *= g4.x;
                r[4 * c + 1] *= g4.y;
                r[4 * c + 2] *= g4.z;
                r[4 * c + 3] *= g4.w;
            }
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
    return launch_pdl(gla_chunked_tc_kernel, dim3(grid), dim3(NT), SMEM_BYTES, s, p, maps);
}

}  // namespace hs
