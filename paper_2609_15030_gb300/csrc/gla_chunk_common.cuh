// Device pieces of the tensor-core prefill (gla_chunked_tc.cu): constants, the shared-memory
// and TMEM maps, the fast path's operand build, state pass, causal mask and output epilogue,
// the exact path's steps, the per-token short segments, and the MMA groups each path issues.
//
// Notation (per head, one segment of L <= 64 tokens inside one 64-token chunk of the
// absolute position grid, cumulative log2-decay Lam_i = log2(e) sum_{s<=i} a_s per key dim):
//   Q~_i = q_i 2^{Lam_i},  K~_j = k_j 2^{-Lam_j},  A_ij = [j <= i] Q~_i . K~_j,
//   o_i = Q~_i S + sum_j A_ij v_j,  S' = diag(2^{Lam_last}) (S + K~^T V)   (fast path)
//   S' = diag(2^{Lam_last}) S + K^^T V,  K^_j = k_j 2^{Lam_last - Lam_j}   (exact path)
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "hs_internal.cuh"
#include "sm100_ptx.cuh"

namespace hs {
namespace gck {

using namespace ptx;

constexpr int CH = 64;    // chunk length (absolute grid)
constexpr int NB = 256;   // operand builders (warps 0..7): cumulative gates, Q~, K~, K~^T, V^T
constexpr int NW = 256;   // state warps (warps 8..15): state passes, masks, epilogues
constexpr int NT = NB + NW;
constexpr int kLoader = 0;   // the first builder thread issues every TMA copy
constexpr int kIssuer = NB;  // the first state thread issues every MMA
constexpr int kShort = 8; // segments of at most this many tokens run token by token
constexpr float kLog2e = 1.4426950408889634f;
// exact path: log-gates below this are taken at this value.  2^(kGateFloor * log2 e) = 2^-144
// is flushed to 0 by ex2.approx.ftz, so such a gate still zeroes the state, while the
// cumulative log2-decay after it stays small enough (|Lam| of a few hundred, not ~1.4e4 for
// a gate of -1e4) for the differences Lam_i - Lam_j of later tokens to keep their precision.
constexpr float kGateFloor = -100.0f;
constexpr float kF16Lim = 32768.0f;         // fast-path fp16 operands stay below 2^15
// a decision taken mid-run bounds the state it starts from (the measured |S| of the previous
// segment's start plus that segment's largest update); the bound is scaled by this margin so
// that whenever it passes, the measured state (what a run resumed at that segment checks)
// passes too: rounding can put the computed state a few ulps above the exact-arithmetic bound
constexpr float kBoundMargin = 1.00390625f; // 1 + 2^-8
constexpr float kLamRange = 10.0f;          // fast path: a segment's total log2-decay >= -10, so
                                            // Q~ = q 2^Lam stays far from fp16's subnormals
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kPrefetch = 2;                // segments requested into L2 ahead of the staged one

// shared memory map (offsets from a 1024-byte aligned base), sized for the head width
// D = d_k = d_v = 128 (a D = 64 head uses the first part of each region).  Operands are
// K-major with the 128-byte swizzle.
constexpr uint32_t SET_BYTES = 57344;   // one fast operand set:
constexpr uint32_t S_QH = 0;            //   Q~  fp16 [64 tok i][D]                     16 KiB
constexpr uint32_t S_KH = 16384;        //   K~  fp16 [64 tok j][D]                     16 KiB
constexpr uint32_t S_AH = 32768;        //   A   fp16 [64 tok i][64 tok j]                8 KiB
                                        //   (16 KiB after it unused)
constexpr uint32_t X_QT = 0;            // exact path (over both sets): Q~ tf32 [64][D]         32 KiB
constexpr uint32_t X_LAM = 32768;       //   Lam f32 [64 tok][D], row-major                     32 KiB
constexpr uint32_t X_B2 = 65536;        //   [A ; K^^T] tf32 [64 i + D][64 tok j]               48 KiB
constexpr uint32_t OFF_SQ = 114688;     // staged q  bf16 [64][D]                  16 KiB
constexpr uint32_t OFF_SK = 131072;     // staged k                                 16 KiB
constexpr uint32_t OFF_SV = 147456;     // staged v                                 16 KiB
constexpr uint32_t OFF_SG = 163840;     // staged log-gates f32 [64][D]             32 KiB
constexpr uint32_t OFF_GAM = 196608;    // 2^{Lam_last} per key dim, four slots by chunk number   2 KiB
constexpr uint32_t OFF_TOT = 198656;    // partial log2-decay totals [token groups][D]        2 KiB
constexpr uint32_t OFF_RED = 200704;    // per warp [8][8]: builders max |q|, fast-path flag, max |k|,
                                        //   max |v| (0..3); state warps max |S| (4)
constexpr uint32_t OFF_BAR = 200960;    // 8 mbarriers
constexpr uint32_t OFF_MISC = 201024;   // TMEM base address, abort flag, decision, run result
constexpr uint32_t OFF_DG = 201088;     // diagonal of A in float32, two sets by segment parity:
                                        //   [set][key-dim half][64 tokens] partial sums  1 KiB
constexpr uint32_t SMEM_BYTES = 202112 + 1024;

// tensor memory: D_O alternates between two buffers by chunk parity, placed on
// either side of S^T so that [D_O0 | S^T] and [S^T | D_O1] are each one accumulator of
// N = 64 + D; even chunks order the (64 + D)-row operand as [A ; K~^T], odd ones as
// [K~^T ; A].  Every MMA has M = 128 (TMEM lanes = value dim e, or query row i for D_A):
// with D = 64 the lanes 64..127 of the state-side products are computed and never read.
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t TM_O0 = 0;           // D_O of even chunks (lane e, col i), 64 cols
constexpr uint32_t TM_S = 64;           // S^T  float32, 128 lanes x D cols
constexpr uint32_t TM_SH = 256;         // S^T fp16 copy, two key dims per column      D/2 cols
constexpr uint32_t TM_A0 = 320;         // D_A of even segments, 128 lanes x 64 cols (lanes 0..63 used)
constexpr uint32_t TM_V = 384;          // V^T: fast, fp16 pairs 2 x 32 cols; exact, f32 64 cols
constexpr uint32_t TM_A1 = 448;         // D_A of odd segments
// exact path (no fast-path data live): S^T as two tf32 parts for S^T Q~^T, hi in the D
// columns right of S^T (D_O1 and, for D = 128, the fp16 copy), lo in the D_A buffers (key
// dims 0..63, 64..127)
constexpr uint32_t TM_SLO0 = 320;
constexpr uint32_t TM_SLO1 = 448;

constexpr uint32_t IDF_N64 = idesc_f16(128, 64);
constexpr uint32_t IDT_N64 = idesc_tf32(128, 64, 0, 0);

// what depends on the head width D (64 or 128)
template <int D>
struct Geo {
    static_assert(D == 64 || D == 128, "head width");
    static constexpr int DP = D / 2;              // builder threads per token group (key-dim pairs)
    static constexpr int NQ = NB / DP;            // token groups of the build: 4 or 8
    static constexpr int TPG = CH / NQ;           // tokens per group: 16 or 8
    static constexpr int CW = D / 2;              // state columns per state thread: 64 or 32
    static constexpr int NG = D / 16;             // short segments: partial sums over 16 key rows
    static constexpr int ROWS = 64 + D;           // rows of the exact path's [A ; K^^T] operand
    static constexpr uint32_t O1 = TM_S + D;      // D_O of odd chunks, right of S^T
    static constexpr uint32_t SHI = TM_S + D;     // exact path: hi part of S^T
    static constexpr uint32_t IDF_ST = idesc_f16(128, D, 1);       // S^T += V^T K~ (K~ read MN-major)
    static constexpr uint32_t IDT_ST = idesc_tf32(128, D, 0, 0);   // exact: S^T += V^T K^
    static constexpr uint32_t STAGE = 3 * CH * D * 2 + CH * D * 4;  // staged q, k, v, log-gates
};

struct TmaMaps {
    CUtensorMap q, k, v, g;
};

// byte offset of 16-bit element (row, col) of a K-major operand with `rows` rows
// (64 columns = 128 bytes per row and slab)
__device__ __forceinline__ uint32_t h_off(int rows, int row, int col)
{
    return (uint32_t)((col >> 6) * rows * 128 + row * 128 + ((((col & 63) >> 3) ^ (row & 7)) << 4) +
                      ((col & 7) << 1));
}

// byte offset of 32-bit element (row, col) of a K-major operand (32 columns per slab)
__device__ __forceinline__ uint32_t t_off(int rows, int row, int col)
{
    return (uint32_t)((col >> 5) * rows * 128 + row * 128 + ((((col & 31) >> 2) ^ (row & 7)) << 4) +
                      ((col & 3) << 2));
}

// barriers among the builder warps (id 1) and among the state warps (id 2)
__device__ __forceinline__ void bar_builders()
{
    asm volatile("bar.sync 1, 256;" ::: "memory");
}

__device__ __forceinline__ void bar_staters()
{
    asm volatile("bar.sync 2, 256;" ::: "memory");
}

// named barrier `id` over 256 threads that also returns the OR of `pred` over them, so
// every thread of the group takes the same branch after it
__device__ __forceinline__ bool bar_or(int id, bool pred)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.or.pred q, %2, 256, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"((uint32_t)pred), "r"(id)
        : "memory");
    return r != 0;
}

__device__ __forceinline__ float warp_max(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// warp sums of eight per-lane values as a transposing butterfly: every lane returns the sum
// over the warp's 32 lanes of value x = (lane >> 2) & 7, added in the same order in every
// lane that holds it
__device__ __forceinline__ float warp_sum8(const float (&v)[8], int lane)
{
    const bool h4 = (lane & 16) != 0, h3 = (lane & 8) != 0, h2 = (lane & 4) != 0;
    float w[4], y[2];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float send = h4 ? v[j] : v[j + 4];
        w[j] = (h4 ? v[j + 4] : v[j]) + __shfl_xor_sync(0xffffffffu, send, 16);
    }
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const float send = h3 ? w[j] : w[j + 2];
        y[j] = (h3 ? w[j + 2] : w[j]) + __shfl_xor_sync(0xffffffffu, send, 8);
    }
    const float send = h2 ? y[0] : y[1];
    float z = (h2 ? y[1] : y[0]) + __shfl_xor_sync(0xffffffffu, send, 4);
    z += __shfl_xor_sync(0xffffffffu, z, 2);
    z += __shfl_xor_sync(0xffffffffu, z, 1);
    return z;
}

__device__ __forceinline__ float bf16f(uint16_t x)
{
    return __uint_as_float(((uint32_t)x) << 16);
}

// two floats -> fp16x2 (round to nearest even), the first in the low half
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi)
{
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// running elementwise maxima of |x| over fp16 / bf16 pairs (NaN propagates)
__device__ __forceinline__ __half2 hmax_abs(__half2 acc, uint32_t pair)
{
    return __hmax2_nan(acc, __habs2(*reinterpret_cast<const __half2 *>(&pair)));
}

__device__ __forceinline__ __nv_bfloat162 bmax_abs(__nv_bfloat162 acc, uint32_t pair)
{
    return __hmax2_nan(acc, __habs2(*reinterpret_cast<const __nv_bfloat162 *>(&pair)));
}

__device__ __forceinline__ float hmax_of(__half2 m)
{
    return fmaxf(__low2float(m), __high2float(m));
}

__device__ __forceinline__ float bmax_of(__nv_bfloat162 m)
{
    return fmaxf(__low2float(m), __high2float(m));
}

// 2^x, one MUFU op (relative error ~2^-22)
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


// zero the staged rows past a segment of L < 64 tokens (all threads, or the builder
// warps only)
template <int D>
__device__ __forceinline__ void zero_tail(uint8_t *smem, int L, bool builders_only)
{
    const int tid = threadIdx.x;
    constexpr int QV = D / 8, RV = 5 * D / 8;   // 16-byte vectors per q/k/v row, per token

    if (L < CH) {
        const int nthr = builders_only ? NB : NT;
        for (int idx = tid; idx < (CH - L) * RV; idx += nthr) {
            const int row = L + idx / RV, c = idx % RV;
            uint4 *dst;
            if (c < QV)
                dst = reinterpret_cast<uint4 *>(smem + OFF_SQ + row * 2 * D) + c;
            else if (c < 2 * QV)
                dst = reinterpret_cast<uint4 *>(smem + OFF_SK + row * 2 * D) + (c - QV);
            else if (c < 3 * QV)
                dst = reinterpret_cast<uint4 *>(smem + OFF_SV + row * 2 * D) + (c - 2 * QV);
            else
                dst = reinterpret_cast<uint4 *>(smem + OFF_SG + row * 4 * D) + (c - 3 * QV);
            *dst = make_uint4(0u, 0u, 0u, 0u);
        }
        if (builders_only)
            bar_builders();
        else
            __syncthreads();
    }
}


// ---- fast operands of a staged long segment into set `par` (builder warps).  Thread
// (dp, qt) owns key dims 2dp, 2dp+1 for the TPG tokens of group qt (16 tokens x 4 groups at
// D = 128, 8 x 8 at D = 64): it sums their log2-gates, then runs the cumulative sum again
// from the earlier groups' totals (shared memory; 2^{Lam_last} into gam slot `gslot`) while
// it writes Q~ and K~ (token-major, the d-contractions' operands) and K~^T (rows of
// [A ; K~^T]), fp16, with 4- and 16-byte stores.  Then thread (e, half) packs V^T into TMEM
// (zeros in the lanes e >= D).  Per warp: max |q|, |k|, |v| and whether every operand fits
// fp16 (for the guard).  The diagonal A_ii = q_i . k_i (no decay between a token and itself)
// is summed in float32 from the bf16 inputs, each warp's 64 key dims by a butterfly, into
// the set's diagonal partials: fp16 Q~ and K~ would round the terms of that dot product to
// 11 bits, which a token whose own q . k cancels cannot afford.
template <int D>
__device__ __forceinline__ void build_fast(uint8_t *smem, uint32_t tmem, int L, int par, int gslot)
{
    using G = Geo<D>;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool worker = warp < 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = warp >> 2;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e
    const int th = colhalf;
    const uint16_t *sQ = reinterpret_cast<const uint16_t *>(smem + OFF_SQ);
    const uint16_t *sK = reinterpret_cast<const uint16_t *>(smem + OFF_SK);
    const uint16_t *sV = reinterpret_cast<const uint16_t *>(smem + OFF_SV);
    const float *sG = reinterpret_cast<const float *>(smem + OFF_SG);
    float *sTot = reinterpret_cast<float *>(smem + OFF_TOT);
    float *sGam = reinterpret_cast<float *>(smem + OFF_GAM);
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);

    if (!worker)
        return;
    zero_tail<D>(smem, L, true);
    const int dp = tid % G::DP, qt = tid / G::DP;
    float amax = -INFINITY;
    {
        // group totals
        float r0 = 0.f, r1 = 0.f;
#pragma unroll
        for (int x = 0; x < G::TPG; ++x) {
            const float2 a = *reinterpret_cast<const float2 *>(sG + (G::TPG * qt + x) * D + 2 * dp);
            amax = fmaxf(amax, fmaxf(a.x, a.y));
            r0 = fmaf(a.x, kLog2e, r0);
            r1 = fmaf(a.y, kLog2e, r1);
        }
        *reinterpret_cast<float2 *>(sTot + qt * D + 2 * dp) = make_float2(r0, r1);
    }
    bar_builders();
    // the running sums start from the earlier groups' totals
    float run0 = 0.f, run1 = 0.f;
    bool lam_ok;
    {
        float t0 = 0.f, t1 = 0.f;
#pragma unroll
        for (int u = 0; u < G::NQ; ++u) {
            const float2 t = *reinterpret_cast<const float2 *>(sTot + u * D + 2 * dp);
            if (u < qt) {
                run0 += t.x;
                run1 += t.y;
            }
            t0 += t.x;
            t1 += t.y;
        }
        if (qt == 0)
            *reinterpret_cast<float2 *>(sGam + gslot * D + 2 * dp) = make_float2(ex2(t0), ex2(t1));
        lam_ok = t0 >= -kLamRange && t1 >= -kLamRange;
    }
    uint8_t *set = smem + par * SET_BYTES;
    __nv_bfloat162 bq = __float2bfloat162_rn(0.f), bk = bq;   // max |q|, |k|
    __half2 hq = __float2half2_rn(0.f), hk = hq;                 // max |Q~|, |K~| (fp16)
    // runs of 8 tokens; within a run, token pairs: Q~ and K~ as fp16 pairs of key dims
    float *sDg = reinterpret_cast<float *>(smem + OFF_DG) + par * 128 + (dp >> 5) * 64;
#pragma unroll 1
    for (int grp = 0; grp < G::TPG / 8; ++grp) {
        float pd[8];   // q . k over this thread's two key dims, tokens 8 grp + 0..7 of its group
#pragma unroll
        for (int u = 0; u < 4; ++u) {
#pragma unroll
            for (int t = 0; t < 2; ++t) {
                const int i = G::TPG * qt + 8 * grp + 2 * u + t;
                const float2 a = *reinterpret_cast<const float2 *>(sG + i * D + 2 * dp);
                run0 = fmaf(a.x, kLog2e, run0);
                run1 = fmaf(a.y, kLog2e, run1);
                const uint32_t q2 = *reinterpret_cast<const uint32_t *>(sQ + i * D + 2 * dp);
                const uint32_t k2 = *reinterpret_cast<const uint32_t *>(sK + i * D + 2 * dp);
                const float q0 = __uint_as_float(q2 << 16), q1 = __uint_as_float(q2 & 0xFFFF0000u);
                const float k0 = __uint_as_float(k2 << 16), k1 = __uint_as_float(k2 & 0xFFFF0000u);
                const uint32_t qp = pack_h2(q0 * ex2(run0), q1 * ex2(run1));
                const uint32_t kp = pack_h2(k0 * ex2(-run0), k1 * ex2(-run1));
                pd[2 * u + t] = fmaf(q1, k1, q0 * k0);
                *reinterpret_cast<uint32_t *>(set + S_QH + h_off(64, i, 2 * dp)) = qp;
                *reinterpret_cast<uint32_t *>(set + S_KH + h_off(64, i, 2 * dp)) = kp;
                bq = bmax_abs(bq, q2);
                bk = bmax_abs(bk, k2);
                hq = hmax_abs(hq, qp);
                hk = hmax_abs(hk, kp);
            }
        }
        const int j0 = G::TPG * qt + 8 * grp;
        const float dsum = warp_sum8(pd, lane);
        if ((lane & 3) == 0)
            sDg[j0 + ((lane >> 2) & 7)] = dsum;
    }
    // V^T: thread (e, half) packs tokens [32 half, 32 half + 32) of value dim e
    __nv_bfloat162 bv = __float2bfloat162_rn(0.f);
    {
        uint32_t vpk[16];
#pragma unroll
        for (int m = 0; m < 16; ++m) {
            const int i = 32 * th + 2 * m;
            uint32_t w = 0;
            if (e_own < D)
                w = (uint32_t)sV[i * D + e_own] | ((uint32_t)sV[(i + 1) * D + e_own] << 16);
            bv = bmax_abs(bv, w);
            vpk[m] = pack_h2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
        }
        tmem_st16(tmem + lrow + TM_V + 32 * par + 16 * th, vpk);
    }
    float mq = warp_max(bmax_of(bq));
    float mk = warp_max(bmax_of(bk));
    float mv = warp_max(bmax_of(bv));
    // non-increasing Lam (|Q~| <= |q|, |A| <= D max|q| max|k|), a total decay of at most
    // 2^-10 (Q~ of the segment's last tokens keeps its precision) and every fp16 operand below
    // 2^15; NaN fails
    bool ok = amax <= 0.f && lam_ok && hmax_of(hq) < kF16Lim && hmax_of(hk) < kF16Lim &&
              mv < kF16Lim;
    ok = __all_sync(0xffffffffu, ok);
    if (lane == 0) {
        sRed[warp * 8 + 0] = mq;
        sRed[warp * 8 + 1] = ok ? 1.f : 0.f;
        sRed[warp * 8 + 2] = mk;
        sRed[warp * 8 + 3] = mv;
    }
    tmem_wait_st();
}


// ---- state pass (state warps): decay by gam slot gpar (gpar < 0: none), checkpoint slot,
// fp16 copy of S^T for the next S^T Q~^T, and the largest |S|
template <int D>
__device__ __forceinline__ void state_pass(uint8_t *smem, uint32_t tmem, int gpar, float *slot, bool copy)
{
    constexpr int CW = Geo<D>::CW;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool worker = warp >= 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = (warp >> 2) & 1;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e
    const float *sGam = reinterpret_cast<const float *>(smem + OFF_GAM);
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);

    if (!worker)
        return;
    float m = 0.f;
    if (e_own < D) {
        const int db = colhalf * CW;
        float r[CW];
#pragma unroll
        for (int c0 = 0; c0 < CW; c0 += 32)
            tmem_ld32(tmem + lrow + TM_S + db + c0, *reinterpret_cast<float(*)[32]>(&r[c0]));
        tmem_wait_ld();
        if (gpar >= 0) {
            const float *gam = sGam + gpar * D + db;
#pragma unroll
            for (int c = 0; c < CW / 4; ++c) {
                const float4 g4 = *reinterpret_cast<const float4 *>(gam + 4 * c);
                r[4 * c] *= g4.x;
                r[4 * c + 1] *= g4.y;
                r[4 * c + 2] *= g4.z;
                r[4 * c + 3] *= g4.w;
            }
#pragma unroll
            for (int c0 = 0; c0 < CW; c0 += 32)
                tmem_st32(tmem + lrow + TM_S + db + c0, *reinterpret_cast<float(*)[32]>(&r[c0]));
        }
        if (slot != nullptr) {
#pragma unroll
            for (int x = 0; x < CW; ++x)
                slot[(int64_t)(db + x) * D + e_own] = r[x];
        }
        if (copy) {
            // the fp16 copy, two key dims per column; its largest magnitude (inf past fp16)
            __half2 hm = __float2half2_rn(0.f);
#pragma unroll
            for (int hh = 0; hh < CW / 32; ++hh) {
                uint32_t u[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) {
                    u[c] = pack_h2(r[32 * hh + 2 * c], r[32 * hh + 2 * c + 1]);
                    hm = hmax_abs(hm, u[c]);
                }
                tmem_st16(tmem + lrow + TM_SH + db / 2 + 16 * hh, u);
            }
            m = hmax_of(hm);
        } else {
#pragma unroll
            for (int x = 0; x < CW; ++x)
                m = fmaxf(m, fabsf(r[x]));
        }
        tmem_wait_st();
    }
    m = warp_max(m);
    if (lane == 0)
        sRed[(warp & 7) * 8 + 4] = m;
}


// ---- the causally masked intra-chunk matrix A (D_A) -> set par's A operand (state warps of
// TMEM lane quarters 0 and 1)
template <int D>
__device__ __forceinline__ void a_build(uint8_t *smem, uint32_t tmem, int par)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool worker = warp >= 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;

    if (!(worker && (warp & 3) < 2))
        return;
    const int i = (warp & 3) * 32 + lane;      // TMEM lane = query row
    const int jb = ((warp >> 2) & 1) * 32;      // this warp's 32 key columns
    float r[32];
    tmem_ld32(tmem + lrow + (par ? TM_A1 : TM_A0) + jb, r);
    // the diagonal from the builders' float32 partials (one per 64 key dims)
    const float *sDg = reinterpret_cast<const float *>(smem + OFF_DG) + par * 128;
    const float dg = (i >= jb && i < jb + 32) ? (D == 128 ? sDg[i] + sDg[64 + i] : sDg[i]) : 0.f;
    tmem_wait_ld();
    uint8_t *set = smem + par * SET_BYTES;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        uint32_t w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int j0 = jb + 8 * c + 2 * u;
            const float x0 = j0 == i ? dg : (j0 <= i ? r[8 * c + 2 * u] : 0.f);
            const float x1 = j0 + 1 == i ? dg : (j0 + 1 <= i ? r[8 * c + 2 * u + 1] : 0.f);
            w[u] = pack_h2(x0, x1);
        }
        *reinterpret_cast<uint4 *>(set + S_AH + h_off(64, i, jb + 8 * c)) =
            make_uint4(w[0], w[1], w[2], w[3]);
    }
}


// ---- output epilogue of a processed segment (state warps): D_O buffer `par` -> o (lane e,
// 32 rows per warp).  With `spare_issuer`, the warp of the MMA-issuing thread (warp 8) is
// left out while it issues, and warp 12 (the same TMEM lane quarter) writes both halves.
template <int D>
__device__ __forceinline__ void out_epilogue(uint32_t tmem, float *ob, int64_t tstride, int L, int par,
                                             bool spare_issuer)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool worker = warp >= 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = (warp >> 2) & 1;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e

    if (!worker || (spare_issuer && warp == 8) || e_own >= D)
        return;
    const int h0 = (spare_issuer && warp == 12) ? 0 : colhalf;
    const int h1 = (spare_issuer && warp == 12) ? 2 : colhalf + 1;
#pragma unroll 1
    for (int hh = h0; hh < h1; ++hh) {
        float r[32];
        const int ib = hh * 32;
        tmem_ld32(tmem + lrow + (par ? Geo<D>::O1 : TM_O0) + ib, r);
        tmem_wait_ld();
        float *op = ob + (int64_t)ib * tstride + e_own;
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
}


// ---- the state between global memory ([d][e], row = key dim) and TMEM (S^T, lane e) ----

// (state warps) load a state into TMEM and record its largest |S| (float32) for the guard
template <int D>
__device__ __forceinline__ void state_load(uint8_t *smem, uint32_t tmem, const float *src)
{
    constexpr int CW = Geo<D>::CW;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp < 8)
        return;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const int colhalf = (warp >> 2) & 1;
    const int e_own = (warp & 3) * 32 + lane;
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);
    float r[32];
    float m = 0.f;
    if (e_own < D) {
#pragma unroll
        for (int c0 = 0; c0 < CW; c0 += 32) {
            const int d0 = colhalf * CW + c0;
#pragma unroll
            for (int x = 0; x < 32; ++x) {
                r[x] = src[(int64_t)(d0 + x) * D + e_own];
                m = fmaxf(m, fabsf(r[x]));
            }
            tmem_st32(tmem + lrow + TM_S + d0, r);
        }
        tmem_wait_st();
    }
    m = warp_max(m);
    if (lane == 0)
        sRed[(warp & 7) * 8 + 4] = m;
}

// (state warps) store the state in TMEM to global memory
template <int D>
__device__ __forceinline__ void state_store(uint32_t tmem, float *dst)
{
    constexpr int CW = Geo<D>::CW;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int e_own = (warp & 3) * 32 + lane;
    if (warp < 8 || e_own >= D)
        return;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const int colhalf = (warp >> 2) & 1;
    float r[32];
#pragma unroll
    for (int c0 = 0; c0 < CW; c0 += 32) {
        const int d0 = colhalf * CW + c0;
        tmem_ld32(tmem + lrow + TM_S + d0, r);
        tmem_wait_ld();
#pragma unroll
        for (int x = 0; x < 32; ++x)
            dst[(int64_t)(d0 + x) * D + e_own] = r[x];
    }
}

// ---- exact path pieces (every thread of the 512-thread CTA takes part) ----

// cumulative log2-gates of a staged segment (key dim d over 32 tokens per state thread,
// token-major into X_LAM; gates below kGateFloor taken at the floor), Q~ = q 2^{Lam} (tf32,
// X_QT), K^^T = k 2^{Lam_last - Lam} (tf32, rows 64.. of X_B2), V^T float32 into TMEM and
// 2^{Lam_last} into gam slot gslot.  Ends with the operands visible to the tensor core.
template <int D>
__device__ __forceinline__ void exact_build(uint8_t *smem, uint32_t tmem, int L, int gslot)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = (warp & 3) * 32 + lane;
    const bool worker = warp >= 8 && d < D;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const int colhalf = (warp >> 2) & 1;
    const int th = colhalf;
    const uint16_t *sQ = reinterpret_cast<const uint16_t *>(smem + OFF_SQ);
    const uint16_t *sK = reinterpret_cast<const uint16_t *>(smem + OFF_SK);
    const uint16_t *sV = reinterpret_cast<const uint16_t *>(smem + OFF_SV);
    const float *sG = reinterpret_cast<const float *>(smem + OFF_SG);
    float *sTot = reinterpret_cast<float *>(smem + OFF_TOT);
    float *sGam = reinterpret_cast<float *>(smem + OFF_GAM);
    float *sLam = reinterpret_cast<float *>(smem + X_LAM);
    float last = 0.f, tot0 = 0.f;
    zero_tail<D>(smem, L, false);
    {
        float run = 0.f;
        if (worker) {
#pragma unroll 8
            for (int x = 0; x < 32; ++x) {
                run = fmaf(fmaxf(sG[(32 * th + x) * D + d], kGateFloor), kLog2e, run);
                sLam[(32 * th + x) * D + d] = run;
            }
            sTot[th * D + d] = run;
        }
        __syncthreads();
        if (worker) {
            tot0 = sTot[d];
            last = tot0 + sTot[D + d];   // Lam_last of key dim d
            if (!th)
                sGam[gslot * D + d] = ex2(last);
        }
    }
    if (worker) {
#pragma unroll 1
        for (int hh = 0; hh < 2; ++hh) {
            uint32_t vtr[16];
#pragma unroll
            for (int g = 0; g < 4; ++g) {
                float4 w;
                float *wv = &w.x;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int x = 16 * hh + 4 * g + u;
                    const int i = 32 * th + x;
                    float lam = sLam[i * D + d];
                    if (th) {
                        lam = tot0 + lam;
                        sLam[i * D + d] = lam;
                    }
                    *reinterpret_cast<float *>(smem + X_QT + t_off(64, i, d)) =
                        rna_tf32(bf16f(sQ[i * D + d]) * ex2(lam));
                    wv[u] = rna_tf32(bf16f(sK[i * D + d]) * ex2(last - lam));
                    vtr[4 * g + u] = __float_as_uint(bf16f(sV[i * D + d]));
                }
                *reinterpret_cast<float4 *>(smem + X_B2 + t_off(Geo<D>::ROWS, 64 + d, 32 * th + 16 * hh + 4 * g)) = w;
            }
            tmem_st16(tmem + lrow + TM_V + 32 * th + 16 * hh, vtr);
        }
        tmem_wait_st();
    }
}

// (state warps) the state as two tf32 parts for S^T Q~^T (an A operand from TMEM is read as
// tf32): hi = S with its low 13 mantissa bits cleared (exact in tf32), lo = S - hi (exact in
// fp32, at most 13 significant bits), so the product keeps the state to ~2^-20 instead of a
// 2^-10 truncation
template <int D>
__device__ __forceinline__ void exact_split_state(uint32_t tmem)
{
    constexpr int CW = Geo<D>::CW;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp < 8 || (warp & 3) * 32 + lane >= D)
        return;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const int colhalf = (warp >> 2) & 1;
#pragma unroll 1
    for (int c0 = 0; c0 < CW; c0 += 32) {
        const int d0 = colhalf * CW + c0;
        float r[32], lo[32];
        tmem_ld32(tmem + lrow + TM_S + d0, r);
        tmem_wait_ld();
#pragma unroll
        for (int x = 0; x < 32; ++x) {
            const float hi = __uint_as_float(__float_as_uint(r[x]) & 0xFFFFE000u);
            lo[x] = r[x] - hi;
            r[x] = hi;
        }
        tmem_st32(tmem + lrow + Geo<D>::SHI + d0, r);
        tmem_st32(tmem + lrow + (d0 < 64 ? TM_SLO0 + d0 : TM_SLO1 + (d0 - 64)), lo);
    }
    tmem_wait_st();
}

// (issuing thread) S^T Q~^T into D_O (TM_O0): the hi part, then the lo part
template <int D>
__device__ __forceinline__ void exact_issue_sq(uint32_t tmem, uint32_t sb)
{
#pragma unroll 1
    for (int kk = 0; kk < D / 8; ++kk) {
        const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
        mma_tf32_ts(tmem + TM_O0, tmem + Geo<D>::SHI + kk * 8, sdesc_sw128(sb + X_QT + koff, 16, 1024),
                    IDT_N64, kk > 0);
    }
#pragma unroll 1
    for (int kk = 0; kk < D / 8; ++kk) {
        const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
        const uint32_t lo = kk < 8 ? TM_SLO0 + kk * 8 : TM_SLO1 + (kk - 8) * 8;
        mma_tf32_ts(tmem + TM_O0, tmem + lo, sdesc_sw128(sb + X_QT + koff, 16, 1024), IDT_N64, 1);
    }
}

// (every thread) A_ij = sum_d q_id k_jd 2^{Lam_id - Lam_jd}, j <= i < L, elementwise, rounded
// to tf32 into rows 0..63 of X_B2
template <int D>
__device__ __forceinline__ void exact_scores(uint8_t *smem, int L)
{
    const int tid = threadIdx.x;
    const uint16_t *sQ = reinterpret_cast<const uint16_t *>(smem + OFF_SQ);
    const uint16_t *sK = reinterpret_cast<const uint16_t *>(smem + OFF_SK);
    const float *lg = reinterpret_cast<const float *>(smem + X_LAM);
    for (int idx = tid; idx < CH * CH; idx += NT) {
        const int i = idx >> 6, j = idx & 63;
        float acc = 0.f;
        if (j <= i && i < L) {
            for (int dd = 0; dd < D; ++dd)
                acc = fmaf(bf16f(sQ[i * D + dd]) * bf16f(sK[j * D + dd]),
                           ex2(lg[i * D + dd] - lg[j * D + dd]), acc);
        }
        *reinterpret_cast<float *>(smem + X_B2 + t_off(Geo<D>::ROWS, i, j)) = rna_tf32(acc);
    }
}

// (issuing thread) D_O += V^T A^T
template <int D>
__device__ __forceinline__ void exact_issue_av(uint32_t tmem, uint32_t sb)
{
#pragma unroll
    for (int kk = 0; kk < CH / 8; ++kk) {
        const uint32_t koff = (kk >> 2) * (Geo<D>::ROWS * 128) + (kk & 3) * 32;
        mma_tf32_ts(tmem + TM_O0, tmem + TM_V + kk * 8, sdesc_sw128(sb + X_B2 + koff, 16, 1024),
                    IDT_N64, 1);
    }
}

// (issuing thread) S^T += V^T K^ (the decay diag(2^{Lam_last}) S applied before)
template <int D>
__device__ __forceinline__ void exact_issue_state(uint32_t tmem, uint32_t sb)
{
#pragma unroll
    for (int kk = 0; kk < CH / 8; ++kk) {
        const uint32_t koff = (kk >> 2) * (Geo<D>::ROWS * 128) + (kk & 3) * 32 + 64 * 128;
        mma_tf32_ts(tmem + TM_S, tmem + TM_V + kk * 8, sdesc_sw128(sb + X_B2 + koff, 16, 1024),
                    Geo<D>::IDT_ST, 1);
    }
}

// ---- fast path MMA groups (issuing thread) ----

// D_A = Q~ K~^T of operand set `par` into its own buffer
template <int D>
__device__ __forceinline__ void fast_issue_scores(uint32_t tmem, uint32_t sb, int par)
{
    const uint32_t setb = sb + (uint32_t)par * SET_BYTES;
#pragma unroll 1
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
        mma_f16_ss(tmem + (par ? TM_A1 : TM_A0), sdesc_sw128(setb + S_QH + koff, 16, 1024),
                   sdesc_sw128(setb + S_KH + koff, 16, 1024), IDF_N64, kk > 0);
    }
}

// D_O = S^T Q~^T (A operand: the fp16 copy of S^T; the update product accumulates onto it)
template <int D>
__device__ __forceinline__ void fast_issue_sq(uint32_t tmem, uint32_t sb, int par)
{
    const uint32_t setb = sb + (uint32_t)par * SET_BYTES;
#pragma unroll 1
    for (int kk = 0; kk < D / 16; ++kk) {
        const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
        mma_f16_ts(tmem + (par ? Geo<D>::O1 : TM_O0), tmem + TM_SH + kk * 8,
                   sdesc_sw128(setb + S_QH + koff, 16, 1024), IDF_N64, kk > 0);
    }
}

// D_O += V^T A^T and S^T += V^T K~, 16 tokens per step.  K~ is stored token-major for D_A
// (K-major there, K = key dim); read with N = key dim contiguous it is the MN-major B operand
// of the state update: 64-dim blocks 8 KiB apart (leading byte offset), 8-token row groups
// 1 KiB apart (stride byte offset), 16 tokens = 2 KiB per step.
// (WITH_STATE false: D_O only, for launches that discard the state)
template <int D, bool WITH_STATE = true>
__device__ __forceinline__ void fast_issue_update(uint32_t tmem, uint32_t sb, int par)
{
    const uint32_t setb = sb + (uint32_t)par * SET_BYTES;
    const uint32_t vt = tmem + TM_V + 32 * par;
#pragma unroll 1
    for (int kk = 0; kk < CH / 16; ++kk) {
        mma_f16_ts(tmem + (par ? Geo<D>::O1 : TM_O0), vt + kk * 8,
                   sdesc_sw128(setb + S_AH + kk * 32, 16, 1024), IDF_N64, 1);
        if (WITH_STATE)
            mma_f16_ts(tmem + TM_S, vt + kk * 8, sdesc_sw128(setb + S_KH + kk * 2048, 8192, 1024),
                       Geo<D>::IDF_ST, 1);
    }
}

// ---- short segments (<= kShort tokens): the per-token recurrence with the recurrent kernel's
// exact operation order (fma chains over groups of 16 key rows, group partials summed left to
// right).  The state part (every thread; gates exponentiated in place, then the state warps
// update S in TMEM, write the slot and the largest |S|, and leave each token's group partials
// in the operand sets) ...
template <int D>
__device__ __forceinline__ void short_state(uint8_t *smem, uint32_t tmem, int L, float *slot)
{
    constexpr int CW = Geo<D>::CW, NG = Geo<D>::NG;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int e_own = (warp & 3) * 32 + lane;
    const bool worker = warp >= 8 && e_own < D;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;
    const int colhalf = (warp >> 2) & 1;
    const uint16_t *sQ = reinterpret_cast<const uint16_t *>(smem + OFF_SQ);
    const uint16_t *sK = reinterpret_cast<const uint16_t *>(smem + OFF_SK);
    const uint16_t *sV = reinterpret_cast<const uint16_t *>(smem + OFF_SV);
    float *sG = reinterpret_cast<float *>(smem + OFF_SG);
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);
    for (int idx = tid; idx < L * D; idx += NT)
        sG[idx] = expf(sG[idx]);
    __syncthreads();
    float *part = reinterpret_cast<float *>(smem);   // [kShort][D/16 groups][D] in the operand sets
    if (warp >= 8) {
        float m = 0.f;
        if (worker) {
            float S[CW];
#pragma unroll
            for (int c0 = 0; c0 < CW; c0 += 32)
                tmem_ld32(tmem + lrow + TM_S + colhalf * CW + c0, *reinterpret_cast<float(*)[32]>(&S[c0]));
            tmem_wait_ld();
            for (int i = 0; i < L; ++i) {
                const float ve = bf16f(sV[i * D + e_own]);
#pragma unroll
                for (int mm = 0; mm < CW / 16; ++mm) {
                    float acc = 0.f;
#pragma unroll
                    for (int r = 16 * mm; r < 16 * mm + 16; ++r) {
                        const int dd = colhalf * CW + r;
                        S[r] = fmaf(sG[i * D + dd], S[r], bf16f(sK[i * D + dd]) * ve);
                        acc = fmaf(bf16f(sQ[i * D + dd]), S[r], acc);
                    }
                    part[(i * NG + colhalf * (NG / 2) + mm) * D + e_own] = acc;
                }
            }
#pragma unroll
            for (int c0 = 0; c0 < CW; c0 += 32)
                tmem_st32(tmem + lrow + TM_S + colhalf * CW + c0, *reinterpret_cast<float(*)[32]>(&S[c0]));
#pragma unroll
            for (int r = 0; r < CW; ++r) {
                m = fmaxf(m, fabsf(S[r]));
                if (slot != nullptr)
                    slot[(int64_t)(colhalf * CW + r) * D + e_own] = S[r];
            }
            tmem_wait_st();
        }
        m = warp_max(m);
        if (lane == 0)
            sRed[(warp & 7) * 8 + 4] = m;
    }
    fence_proxy_async_smem();
    __syncthreads();
}

// ... and the outputs (every thread): each token's output is the left-to-right sum of its
// eight group partials
template <int D>
__device__ __forceinline__ void short_outputs(const uint8_t *smem, int L, float *ob, int64_t tstride)
{
    constexpr int NG = Geo<D>::NG;
    const float *part = reinterpret_cast<const float *>(smem);
    for (int idx = threadIdx.x; idx < L * D; idx += NT) {
        const int i = idx / D, e = idx % D;
        float sum = part[(i * NG) * D + e];
#pragma unroll
        for (int g = 1; g < NG; ++g)
            sum += part[(i * NG + g) * D + e];
        ob[(int64_t)i * tstride + e] = sum;
    }
}

// ---- tensor maps of the q / k / v / log-gate rows ([rows][n_heads * 128], one 64-row x
// 128-element box per head and segment) ----

inline PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
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

template <int D>
inline bool encode_rows(CUtensorMap *m, CUtensorMapDataType dt, const void *base, uint64_t inner,
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


}  // namespace gck
}  // namespace hs
