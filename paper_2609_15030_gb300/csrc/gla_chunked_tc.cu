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
// transposed (lane = value dim e, column = key dim d).
//
// Fast chunks run three kind::f16 MMA groups with fp16 operands and float32
// accumulators:  D_O = S^T Q~^T (A operand: an fp16 copy of S^T in TMEM),
// D_A = Q~ K~^T, then [D_O | S^T] += V^T [A ; K~^T]^T as one N=192 product
// (V^T in TMEM).  fp16 keeps the 10-bit mantissa of tf32 but halves the
// instructions (K = 16 per MMA).  The CTA's 16 warps form two groups in a
// pipeline over two alternating operand sets: while the eight state warps
// finish chunk c (the state pass, which applies the pending decay 2^{Lam_last},
// writes a due checkpoint and refreshes the fp16 copy of S^T; the causal mask;
// the output epilogue) the eight builder warps stage chunk c+1 and build its
// operands (cumulative decay scan, Q~, K~, K~^T, V^T).  The first builder thread
// issues the TMA copies and D_A, the first state thread the other MMAs.
//
// A chunk is fast only if every fp16 operand provably stays below 2^15 in
// magnitude (|q|, |v|, |K~|, the bound 128 max|q| max|k| on |A|, and a bound
// on |S| carried from the measured state) and its total decay factor
// 2^{Lam_last} stays >= 2^-10 in every key dim (so Q~ never nears fp16's
// subnormals).  Any other chunk (strong decay, huge values) runs the exact
// path: tf32 operands (the state split into two exact tf32 parts), the
// intra-chunk matrix computed elementwise in float32 with 2^{Lam_i - Lam_j} <= 1,
// and the state updated as
// diag(2^{Lam_last}) S + K^^T V with K^_j = k_j 2^{Lam_last - Lam_j}.  The
// choice depends only on the chunk's inputs and on the state it starts from,
// as does every operation order, so a resumed run reproduces a full
// recomputation bit for bit when it starts on the chunk grid.  Segments of at
// most 8 tokens run the per-token recurrence with the recurrent kernel's exact
// operation order.
//
// Every wait on an mbarrier is bounded (1 s) and is followed by a barrier that
// reduces the abort flag, so every thread of a group takes the same branch; on
// timeout the CTA reports HS_DEVERR_TIMEOUT, waits (bounded) for its own copies
// and MMAs in flight, frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "hs_internal.cuh"
#include "sm100_ptx.cuh"

namespace hs {
namespace {

using namespace ptx;

constexpr int D = 128;    // d_k = d_v
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

// shared memory map (offsets from a 1024-byte aligned base).  Operands are
// K-major with the 128-byte swizzle.
constexpr uint32_t SET_BYTES = 57344;   // one fast operand set:
constexpr uint32_t S_QH = 0;            //   Q~  fp16 [64 tok i][128 d]                 16 KiB
constexpr uint32_t S_KH = 16384;        //   K~  fp16 [64 tok j][128 d]                 16 KiB
constexpr uint32_t S_B2H = 32768;       //   [A ; K~^T] fp16 [64 i + 128 d][64 tok j]   24 KiB
constexpr uint32_t X_QT = 0;            // exact path (over both sets): Q~ tf32 [64][128]     32 KiB
constexpr uint32_t X_LAM = 32768;       //   Lam f32 [64 tok][128 d], row-major                 32 KiB
constexpr uint32_t X_B2 = 65536;        //   [A ; K^^T] tf32 [64 i + 128 d][64 tok j]           48 KiB
constexpr uint32_t OFF_SQ = 114688;     // staged q  bf16 [64][128]                16 KiB
constexpr uint32_t OFF_SK = 131072;     // staged k                                 16 KiB
constexpr uint32_t OFF_SV = 147456;     // staged v                                 16 KiB
constexpr uint32_t OFF_SG = 163840;     // staged log-gates f32 [64][128]           32 KiB
constexpr uint32_t OFF_GAM = 196608;    // 2^{Lam_last} per key dim, four slots by chunk number   2 KiB
constexpr uint32_t OFF_TOT = 198656;    // partial log2-decay totals [4 token quarters][128]  2 KiB
constexpr uint32_t OFF_RED = 200704;    // per warp [8][8]: builders max |q|, fast-path flag, max |k|,
                                        //   max |v| (0..3); state warps max |S| (4)
constexpr uint32_t OFF_BAR = 200960;    // 8 mbarriers
constexpr uint32_t OFF_MISC = 201024;   // TMEM base address, abort flag, decision, run result
constexpr uint32_t OFF_DG = 201088;     // diagonal of A in float32, two sets by segment parity:
                                        //   [set][key-dim half][64 tokens] partial sums  1 KiB
constexpr uint32_t SMEM_BYTES = 202112 + 1024;
constexpr uint32_t STAGE_BYTES = 3 * 16384 + 32768;

// tensor memory: D_O alternates between two buffers by chunk parity, placed on
// either side of S^T so that [D_O0 | S^T] and [S^T | D_O1] are each one N=192
// accumulator; even chunks order the 192-row operand as [A ; K~^T], odd ones
// as [K~^T ; A].
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t TM_O0 = 0;           // D_O of even chunks (lane e, col i), 64 cols
constexpr uint32_t TM_S = 64;           // S^T  float32, 128 lanes x 128 cols
constexpr uint32_t TM_O1 = 192;         // D_O of odd chunks
constexpr uint32_t TM_SH = 256;         // S^T fp16 copy, two key dims per column      64 cols
constexpr uint32_t TM_A0 = 320;         // D_A of even segments, 128 lanes x 64 cols (lanes 0..63 used)
constexpr uint32_t TM_V = 384;          // V^T: fast, fp16 pairs 2 x 32 cols; exact, f32 64 cols
constexpr uint32_t TM_A1 = 448;         // D_A of odd segments
// exact path (no fast-path data live): S^T as two tf32 parts for S^T Q~^T, hi in the 128
// columns of D_O1 and the fp16 copy, lo in the two D_A buffers (key dims 0..63, 64..127)
constexpr uint32_t TM_SHI = 192;
constexpr uint32_t TM_SLO0 = 320;
constexpr uint32_t TM_SLO1 = 448;

constexpr uint32_t IDF_N64 = idesc_f16(128, 64);
constexpr uint32_t IDF_N192 = idesc_f16(128, 192);
constexpr uint32_t IDT_N64 = idesc_tf32(128, 64, 0, 0);
constexpr uint32_t IDT_N128 = idesc_tf32(128, 128, 0, 0);

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
__device__ __forceinline__ void zero_tail(uint8_t *smem, int L, bool builders_only)
{
    const int tid = threadIdx.x;

    if (L < CH) {
        const int nthr = builders_only ? NB : NT;
        for (int idx = tid; idx < (CH - L) * 80; idx += nthr) {
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
        if (builders_only)
            bar_builders();
        else
            __syncthreads();
    }
}


// ---- fast operands of a staged long segment into set `par` (builder warps).  Thread
// (dp, qt) owns key dims 2dp, 2dp+1 for tokens [16 qt, 16 qt + 16): it sums their
// log2-gates, then runs the cumulative sum again from the earlier quarters' totals (shared
// memory; 2^{Lam_last} into gam slot `gslot`) while it writes Q~ and K~ (token-major, the
// d-contractions' operands) and K~^T (rows of [A ; K~^T]), fp16, with 4- and 16-byte
// stores.  Then thread (e, half) packs V^T into TMEM.  Per warp: max |q|, |k|, |v| and
// whether every operand fits fp16 (for the guard).  The diagonal A_ii = q_i . k_i (no decay
// between a token and itself) is summed in float32 from the bf16 inputs, each warp's 64 key
// dims by a butterfly, into the set's diagonal partials: fp16 Q~ and K~ would round the
// terms of that dot product to 11 bits, which a token whose own q . k cancels cannot afford.
__device__ __forceinline__ void build_fast(uint8_t *smem, uint32_t tmem, int L, int par, int gslot)
{
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
    zero_tail(smem, L, true);
    const int dp = tid & 63, qt = (tid >> 6) & 3;
    float amax = -INFINITY;
    {
        // quarter totals
        float r0 = 0.f, r1 = 0.f;
#pragma unroll
        for (int x = 0; x < 16; ++x) {
            const float2 a = *reinterpret_cast<const float2 *>(sG + (16 * qt + x) * D + 2 * dp);
            amax = fmaxf(amax, fmaxf(a.x, a.y));
            r0 = fmaf(a.x, kLog2e, r0);
            r1 = fmaf(a.y, kLog2e, r1);
        }
        *reinterpret_cast<float2 *>(sTot + qt * D + 2 * dp) = make_float2(r0, r1);
    }
    bar_builders();
    // the running sums start from the earlier quarters' totals
    float run0 = 0.f, run1 = 0.f;
    bool lam_ok;
    {
        float t0 = 0.f, t1 = 0.f;
#pragma unroll
        for (int u = 0; u < 4; ++u) {
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
    const int rowK = par ? 0 : 64;
    __nv_bfloat162 bq = __float2bfloat162_rn(0.f), bk = bq;   // max |q|, |k|
    __half2 hq = __float2half2_rn(0.f), hk = hq;                 // max |Q~|, |K~| (fp16)
    // two groups of 8 tokens; within a group, token pairs: Q~ and K~ as fp16 pairs of key
    // dims, K~^T rows 2dp and 2dp+1 as fp16 pairs of tokens (byte permutes of the K~ pairs)
    float *sDg = reinterpret_cast<float *>(smem + OFF_DG) + par * 128 + (warp & 1) * 64;
#pragma unroll 1
    for (int grp = 0; grp < 2; ++grp) {
        uint32_t kt0[4], kt1[4];
        float pd[8];   // q . k over this thread's two key dims, tokens 8 grp + 0..7 of its quarter
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            uint32_t kp[2];
#pragma unroll
            for (int t = 0; t < 2; ++t) {
                const int i = 16 * qt + 8 * grp + 2 * u + t;
                const float2 a = *reinterpret_cast<const float2 *>(sG + i * D + 2 * dp);
                run0 = fmaf(a.x, kLog2e, run0);
                run1 = fmaf(a.y, kLog2e, run1);
                const uint32_t q2 = *reinterpret_cast<const uint32_t *>(sQ + i * D + 2 * dp);
                const uint32_t k2 = *reinterpret_cast<const uint32_t *>(sK + i * D + 2 * dp);
                const float q0 = __uint_as_float(q2 << 16), q1 = __uint_as_float(q2 & 0xFFFF0000u);
                const float k0 = __uint_as_float(k2 << 16), k1 = __uint_as_float(k2 & 0xFFFF0000u);
                const uint32_t qp = pack_h2(q0 * ex2(run0), q1 * ex2(run1));
                kp[t] = pack_h2(k0 * ex2(-run0), k1 * ex2(-run1));
                pd[2 * u + t] = fmaf(q1, k1, q0 * k0);
                *reinterpret_cast<uint32_t *>(set + S_QH + h_off(64, i, 2 * dp)) = qp;
                *reinterpret_cast<uint32_t *>(set + S_KH + h_off(64, i, 2 * dp)) = kp[t];
                bq = bmax_abs(bq, q2);
                bk = bmax_abs(bk, k2);
                hq = hmax_abs(hq, qp);
                hk = hmax_abs(hk, kp[t]);
            }
            kt0[u] = __byte_perm(kp[0], kp[1], 0x5410);   // key dim 2dp: tokens (2u, 2u+1)
            kt1[u] = __byte_perm(kp[0], kp[1], 0x7632);   // key dim 2dp+1
        }
        const int j0 = 16 * qt + 8 * grp;
        {
            const float dsum = warp_sum8(pd, lane);
            if ((lane & 3) == 0)
                sDg[j0 + ((lane >> 2) & 7)] = dsum;
        }
        *reinterpret_cast<uint4 *>(set + S_B2H + h_off(192, rowK + 2 * dp, j0)) =
            make_uint4(kt0[0], kt0[1], kt0[2], kt0[3]);
        *reinterpret_cast<uint4 *>(set + S_B2H + h_off(192, rowK + 2 * dp + 1, j0)) =
            make_uint4(kt1[0], kt1[1], kt1[2], kt1[3]);
    }
    // V^T: thread (e, half) packs tokens [32 half, 32 half + 32) of value dim e
    __nv_bfloat162 bv = __float2bfloat162_rn(0.f);
    {
        uint32_t vpk[16];
#pragma unroll
        for (int m = 0; m < 16; ++m) {
            const int i = 32 * th + 2 * m;
            const uint32_t w = (uint32_t)sV[i * D + e_own] | ((uint32_t)sV[(i + 1) * D + e_own] << 16);
            bv = bmax_abs(bv, w);
            vpk[m] = pack_h2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
        }
        tmem_st16(tmem + lrow + TM_V + 32 * par + 16 * th, vpk);
    }
    float mq = warp_max(bmax_of(bq));
    float mk = warp_max(bmax_of(bk));
    float mv = warp_max(bmax_of(bv));
    // non-increasing Lam (|Q~| <= |q|, |A| <= 128 max|q| max|k|), a total decay of at most
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
__device__ __forceinline__ void state_pass(uint8_t *smem, uint32_t tmem, int gpar, float *slot, bool copy)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool worker = warp >= 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = (warp >> 2) & 1;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e
    const float *sGam = reinterpret_cast<const float *>(smem + OFF_GAM);
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);

    if (!worker)
        return;
    const int db = colhalf * 64;
    float r[64];
    tmem_ld32(tmem + lrow + TM_S + db, *reinterpret_cast<float(*)[32]>(&r[0]));
    tmem_ld32(tmem + lrow + TM_S + db + 32, *reinterpret_cast<float(*)[32]>(&r[32]));
    tmem_wait_ld();
    if (gpar >= 0) {
        const float *gam = sGam + gpar * D + db;
#pragma unroll
        for (int c = 0; c < 16; ++c) {
            const float4 g4 = *reinterpret_cast<const float4 *>(gam + 4 * c);
            r[4 * c] *= g4.x;
            r[4 * c + 1] *= g4.y;
            r[4 * c + 2] *= g4.z;
            r[4 * c + 3] *= g4.w;
        }
        tmem_st32(tmem + lrow + TM_S + db, *reinterpret_cast<float(*)[32]>(&r[0]));
        tmem_st32(tmem + lrow + TM_S + db + 32, *reinterpret_cast<float(*)[32]>(&r[32]));
    }
    if (slot != nullptr) {
#pragma unroll
        for (int x = 0; x < 64; ++x)
            slot[(int64_t)(db + x) * D + e_own] = r[x];
    }
    float m;
    if (copy) {
        // the fp16 copy, two key dims per column; its largest magnitude (inf past fp16)
        __half2 hm = __float2half2_rn(0.f);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
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
        m = 0.f;
#pragma unroll
        for (int x = 0; x < 64; ++x)
            m = fmaxf(m, fabsf(r[x]));
    }
    tmem_wait_st();
    m = warp_max(m);
    if (lane == 0)
        sRed[(warp & 7) * 8 + 4] = m;
}


// ---- the causally masked intra-chunk matrix A (D_A) -> rows rowA.. of set par's [A ; K~^T]
// (state warps of TMEM lane quarters 0 and 1)
__device__ __forceinline__ void a_build(uint8_t *smem, uint32_t tmem, int par)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool worker = warp >= 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;

    if (!(worker && (warp & 3) < 2))
        return;
    const int i = (warp & 3) * 32 + lane;      // TMEM lane = query row
    const int jb = ((warp >> 2) & 1) * 32;      // this warp's 32 key columns
    const int rowA = par ? 128 : 0;
    float r[32];
    tmem_ld32(tmem + lrow + (par ? TM_A1 : TM_A0) + jb, r);
    // the diagonal from the builders' float32 partials (the two key-dim halves)
    const float *sDg = reinterpret_cast<const float *>(smem + OFF_DG) + par * 128;
    const float dg = (i >= jb && i < jb + 32) ? sDg[i] + sDg[64 + i] : 0.f;
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
        *reinterpret_cast<uint4 *>(set + S_B2H + h_off(192, rowA + i, jb + 8 * c)) =
            make_uint4(w[0], w[1], w[2], w[3]);
    }
}


// ---- output epilogue of a processed segment (state warps): D_O buffer `par` -> o (lane e,
// 32 rows per warp).  With `spare_issuer`, the warp of the MMA-issuing thread (warp 8) is
// left out while it issues, and warp 12 (the same TMEM lane quarter) writes both halves.
__device__ __forceinline__ void out_epilogue(uint32_t tmem, float *ob, int64_t tstride, int L, int par,
                                             bool spare_issuer)
{
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool worker = warp >= 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = (warp >> 2) & 1;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e

    if (!worker || (spare_issuer && warp == 8))
        return;
    const int h0 = (spare_issuer && warp == 12) ? 0 : colhalf;
    const int h1 = (spare_issuer && warp == 12) ? 2 : colhalf + 1;
#pragma unroll 1
    for (int hh = h0; hh < h1; ++hh) {
        float r[32];
        const int ib = hh * 32;
        tmem_ld32(tmem + lrow + (par ? TM_O1 : TM_O0) + ib, r);
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
    float *sTot = reinterpret_cast<float *>(smem + OFF_TOT);
    float *sGam = reinterpret_cast<float *>(smem + OFF_GAM);
    float *sRed = reinterpret_cast<float *>(smem + OFF_RED);
    // [0] TMEM base, [1] abort flag, [2] decision on the latest built segment (1 = fast),
    // [3] run result (1 = the segment at [4..5] needs the exact path), [4..5] position
    // where the run stopped, [6..7] its local token index
    volatile uint32_t *sMisc = reinterpret_cast<volatile uint32_t *>(smem + OFF_MISC);
    volatile int64_t *sRun = reinterpret_cast<volatile int64_t *>(smem + OFF_MISC + 16);
    const uint32_t bar_tma = sb + OFF_BAR, bar_a = sb + OFF_BAR + 8, bar_o = sb + OFF_BAR + 16,
                   bar_s = sb + OFF_BAR + 24, bar_built = sb + OFF_BAR + 32,
                   bar_go = sb + OFF_BAR + 40, bar_ld = sb + OFF_BAR + 48,
                   bar_a1 = sb + OFF_BAR + 56;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int b = blockIdx.x / p.n_heads;
    const int h = blockIdx.x - b * p.n_heads;
    const int n = p.n_tokens[b];
    if (n <= 0)
        return;
    const int64_t pos0 = p.pos0[b];
    const int64_t end = pos0 + n;
    const int64_t tstride = (int64_t)p.n_heads * D;   // elements between consecutive tokens
    const int C = p.ckpt_interval;

    if (tid == 0) {
        mbar_init(bar_tma, 1);
        mbar_init(bar_a, 1);
        mbar_init(bar_o, 1);
        mbar_init(bar_s, 1);
        mbar_init(bar_built, 1);
        mbar_init(bar_go, 1);
        mbar_init(bar_ld, 1);
        mbar_init(bar_a1, 1);
        fence_mbar_init();
        sMisc[1] = 0;   // abort flag
    }
    if (warp == 0)
        tmem_alloc(sb + OFF_MISC, TMEM_COLS);
    if (tid == kLoader) {
        // the first segment's inputs into L2 while the previous kernel finishes: a
        // prefetch moves no data into this SM, and L2 holds the only copy any later write
        // updates, so it is safe even if that kernel writes those inputs
        const int32_t y = (int32_t)p.row0[b];
        tma_prefetch_2d(&maps.q, h * D, y);
        tma_prefetch_2d(&maps.k, h * D, y);
        tma_prefetch_2d(&maps.v, h * D, y);
        tma_prefetch_2d(&maps.g, h * D, y);
    }
    pdl_wait();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sMisc[0];
    const bool builder = warp < 8;
    const bool worker = !builder;                              // a state warp
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = (warp >> 2) & 1;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e
    // exact operand map: state thread owns key dim d = e_own for tokens [32*th, 32*th+32)
    const int d = e_own;
    const int th = colhalf;

    // bookkeeping of the loader (copies issued, one still in flight) and of the issuer,
    // for the waits and the abort path; every mbarrier is waited on by one thread only
    uint32_t n_tma = 0;
    bool tma_pending = false;
    uint32_t ph_tma = 0, ph_o = 0, ph_s = 0, ph_built = 0, ph_go = 0;
    uint32_t ph_a0 = 0, ph_a1 = 0;   // D_A products of even / odd segments (bar_a, bar_a1)
    bool aborted = false;

    // L2 prefetch of the 64 tokens from local position t (if any are this problem's)
    auto prefetch = [&](int64_t t) {
        if (t >= n)
            return;
        const int32_t y = (int32_t)((int64_t)p.row0[b] + t);
        const int32_t x = h * D;
        tma_prefetch_2d(&maps.q, x, y);
        tma_prefetch_2d(&maps.k, x, y);
        tma_prefetch_2d(&maps.v, x, y);
        tma_prefetch_2d(&maps.g, x, y);
    };
    // (loader) staged inputs of the segment at local position tok_local; segments after
    // the first start on the 64-token grid, so the segment kPrefetch ahead starts at
    // tok_local + 64 * kPrefetch and is requested into L2 now
    auto issue_tma = [&](int64_t tok_local) {
        const int32_t y = (int32_t)((int64_t)p.row0[b] + tok_local);
        const int32_t x = h * D;
        mbar_arrive_expect_tx(bar_tma, STAGE_BYTES);
        tma_load_2d(sb + OFF_SQ, &maps.q, x, y, bar_tma);
        tma_load_2d(sb + OFF_SK, &maps.k, x, y, bar_tma);
        tma_load_2d(sb + OFF_SV, &maps.v, x, y, bar_tma);
        tma_load_2d(sb + OFF_SG, &maps.g, x, y, bar_tma);
        ++n_tma;
        tma_pending = true;
        if (tok_local > 0)
            prefetch(tok_local + (int64_t)CH * kPrefetch);
    };
    // one thread (`who`) waits on an mbarrier; false (for every thread) if that wait ran
    // out or another thread raised the abort flag.  CTA-wide, or within the builder (id 1)
    // or state (id 2) warps; the barrier's OR reduction makes the answer uniform.
    auto wait_all = [&](int who, uint32_t bar, uint32_t &ph) -> bool {
        bool bad = false;
        if (tid == who)
            bad = !mbar_wait_bounded(bar, ph, kTimeoutNs);
        if (bad)
            sMisc[1] = 1;
        ph ^= 1;
        const bool stop = __syncthreads_or(bad || sMisc[1] != 0) != 0;
        tc_fence_after();
        if (stop)
            aborted = true;
        return !stop;
    };
    auto wait_tma = [&]() -> bool {
        tma_pending = false;
        return wait_all(kLoader, bar_tma, ph_tma);
    };
    auto wait_group = [&](int id, int who, uint32_t bar, uint32_t &ph) -> bool {
        bool bad = false;
        if (tid == who)
            bad = !mbar_wait_bounded(bar, ph, kTimeoutNs);
        if (bad)
            sMisc[1] = 1;
        ph ^= 1;
        const bool stop = bar_or(id, bad || sMisc[1] != 0);
        tc_fence_after();
        if (stop)
            aborted = true;
        return !stop;
    };
    // a group barrier that also reports the abort flag, uniformly
    auto sync_group = [&](int id) -> bool {
        const bool stop = bar_or(id, sMisc[1] != 0);
        if (stop)
            aborted = true;
        return !stop;
    };
    auto sync_all = [&]() -> bool {
        const bool stop = __syncthreads_or(sMisc[1] != 0) != 0;
        if (stop)
            aborted = true;
        return !stop;
    };
    auto seg_len = [&](int64_t at) -> int { return (int)(min(end, (at / CH + 1) * CH) - at); };
    auto is_long = [&](int64_t at) -> bool { return at < end && seg_len(at) > kShort; };
    auto ckpt_slot = [&](int64_t seg_end) -> float * {
        if (!(C > 0 && seg_end % C == 0 && p.ckpt_slots != nullptr))
            return nullptr;
        float *slot = p.ckpt_slots[p.ck_base[b] + (seg_end / C - pos0 / C - 1)];
        if (slot == nullptr || (reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
            if (tid == kIssuer)
                report(p.d_err, slot == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
            return nullptr;
        }
        return slot + (int64_t)h * D * D;
    };
    // largest |S| recorded by the last state pass (valid after the barrier that follows it)
    auto state_max = [&]() -> float {
        float m = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w)
            m = fmaxf(m, sRed[w * 8 + 4]);
        return m;
    };

    if (tid == kLoader)
        issue_tma(0);
    bool prefetched = false;   // (loader) the segments after the first requested into L2

    // incoming state -> TMEM (state warps), transposed: S^T[e][d] = state[d][e]; its
    // largest magnitude.  The builders meanwhile stage and build the first segment.
    float *st_g = p.state + ((int64_t)b * p.n_heads + h) * D * D;
    if (worker) {
        float r[32];
        float m = 0.f;
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 32) {
            const int d0 = colhalf * 64 + c0;
#pragma unroll
            for (int x = 0; x < 32; ++x) {
                r[x] = st_g[(int64_t)(d0 + x) * D + e_own];
                m = fmaxf(m, fabsf(r[x]));
            }
            tmem_st32(tmem + lrow + TM_S + d0, r);
        }
        tmem_wait_st();
        m = warp_max(m);
        if (lane == 0)
            sRed[(warp & 7) * 8 + 4] = m;
        tc_fence_before();
        bar_staters();
        tc_fence_after();
    }

    // ---- a short segment (<= kShort tokens, staged inputs already waited for, no decay
    // pending): the per-token recurrence with the recurrent kernel's exact operation order
    // (fma chains over groups of 16 key rows, group partials summed left to right)
    auto short_segment = [&](int64_t tok_s, int L, int64_t seg_end) {
        for (int idx = tid; idx < L * D; idx += NT)
            sG[idx] = expf(sG[idx]);
        __syncthreads();
        float *part = reinterpret_cast<float *>(smem);   // [kShort][8 groups][128] in the operand sets
        float *slot = ckpt_slot(seg_end);
        if (worker) {
            float S[64];
            tmem_ld32(tmem + lrow + TM_S + colhalf * 64, *reinterpret_cast<float(*)[32]>(&S[0]));
            tmem_ld32(tmem + lrow + TM_S + colhalf * 64 + 32, *reinterpret_cast<float(*)[32]>(&S[32]));
            tmem_wait_ld();
            for (int i = 0; i < L; ++i) {
                const float ve = bf16f(sV[i * D + e_own]);
#pragma unroll
                for (int m = 0; m < 4; ++m) {
                    float acc = 0.f;
#pragma unroll
                    for (int r = 16 * m; r < 16 * m + 16; ++r) {
                        const int dd = colhalf * 64 + r;
                        S[r] = fmaf(sG[i * D + dd], S[r], bf16f(sK[i * D + dd]) * ve);
                        acc = fmaf(bf16f(sQ[i * D + dd]), S[r], acc);
                    }
                    part[(i * 8 + colhalf * 4 + m) * D + e_own] = acc;
                }
            }
            tmem_st32(tmem + lrow + TM_S + colhalf * 64, *reinterpret_cast<float(*)[32]>(&S[0]));
            tmem_st32(tmem + lrow + TM_S + colhalf * 64 + 32, *reinterpret_cast<float(*)[32]>(&S[32]));
            float m = 0.f;
#pragma unroll
            for (int r = 0; r < 64; ++r) {
                m = fmaxf(m, fabsf(S[r]));
                if (slot != nullptr)
                    slot[(int64_t)(colhalf * 64 + r) * D + e_own] = S[r];
            }
            m = warp_max(m);
            if (lane == 0)
                sRed[(warp & 7) * 8 + 4] = m;
            tmem_wait_st();
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == kLoader && seg_end < end)
            issue_tma(tok_s + L);
        float *ob = p.o + (((int64_t)p.row0[b] + tok_s) * p.n_heads + h) * D;
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
    };

    // the guard of a built fast segment (state warps, after the wait for the builders): log-gates
    // <= 0, and every fp16 operand (Q~, K~, V, A, the fp16 copy of the state it starts from)
    // below 2^15 in magnitude.  Returns whether the segment's own inputs pass; `state_ok` says
    // whether the state (its measured magnitude, or a bound on it) passes too.
    float mk_new = 0.f, mv_new = 0.f;
    auto guard = [&](float s_mag, bool &state_ok) -> bool {
        float mq = 0.f, mk = 0.f, mv = 0.f;
        bool ok = true;
#pragma unroll
        for (int w = 0; w < 8; ++w) {
            mq = fmaxf(mq, sRed[w * 8 + 0]);
            ok = ok && sRed[w * 8 + 1] != 0.f;
            mk = fmaxf(mk, sRed[w * 8 + 2]);
            mv = fmaxf(mv, sRed[w * 8 + 3]);
        }
        mk_new = mk;
        mv_new = mv;
        state_ok = s_mag < kF16Lim;
        return ok && 128.0f * mq * mk < kF16Lim;
    };

    // ---- one exact segment, from staged inputs, no decay pending and no MMA in flight;
    // leaves the final state in TMEM, writes its outputs and checkpoint
    auto exact_segment = [&](int64_t tok_s, int L, int par, int gslot, int64_t seg_end) -> bool {
        // cumulative log2-gates: key dim d over 32 tokens per thread (token-major into
        // X_LAM, the elementwise A reads them there), halves joined through shared memory;
        // 2^{Lam_last} into gam slot gslot
        float *sLam = reinterpret_cast<float *>(smem + X_LAM);
        float last = 0.f, tot0 = 0.f;
        zero_tail(smem, L, false);
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
            // Q~ = q 2^{Lam} (tf32), K^^T = k 2^{Lam_last - Lam} (tf32, rows 64.. of X_B2),
            // V^T float32 into TMEM, 16 tokens at a time
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
                    *reinterpret_cast<float4 *>(smem + X_B2 + t_off(192, 64 + d, 32 * th + 16 * hh + 4 * g)) = w;
                }
                tmem_st16(tmem + lrow + TM_V + 32 * th + 16 * hh, vtr);
            }
            // the state as two tf32 parts for S^T Q~^T (an A operand from TMEM is read as
            // tf32): hi = S with its low 13 mantissa bits cleared (exact in tf32), lo = S - hi
            // (exact in fp32, at most 13 significant bits), so the product keeps the state to
            // ~2^-20 instead of a 2^-10 truncation
#pragma unroll 1
            for (int c0 = 0; c0 < 64; c0 += 32) {
                const int d0 = colhalf * 64 + c0;
                float r[32], lo[32];
                tmem_ld32(tmem + lrow + TM_S + d0, r);
                tmem_wait_ld();
#pragma unroll
                for (int x = 0; x < 32; ++x) {
                    const float hi = __uint_as_float(__float_as_uint(r[x]) & 0xFFFFE000u);
                    lo[x] = r[x] - hi;
                    r[x] = hi;
                }
                tmem_st32(tmem + lrow + TM_SHI + d0, r);
                tmem_st32(tmem + lrow + (d0 < 64 ? TM_SLO0 + d0 : TM_SLO1 + (d0 - 64)), lo);
            }
            tmem_wait_st();
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        const uint32_t tm_o = TM_O0;   // par is 0 here: D_O1's columns hold the split state
        if (tid == kIssuer) {
            // S^T Q~^T into D_O: the hi part, then the lo part
            tc_fence_after();
#pragma unroll 1
            for (int kk = 0; kk < D / 8; ++kk) {
                const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
                mma_tf32_ts(tmem + tm_o, tmem + TM_SHI + kk * 8, sdesc_sw128(sb + X_QT + koff, 16, 1024),
                            IDT_N64, kk > 0);
            }
#pragma unroll 1
            for (int kk = 0; kk < D / 8; ++kk) {
                const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
                const uint32_t lo = kk < 8 ? TM_SLO0 + kk * 8 : TM_SLO1 + (kk - 8) * 8;
                mma_tf32_ts(tmem + tm_o, tmem + lo, sdesc_sw128(sb + X_QT + koff, 16, 1024), IDT_N64, 1);
            }
        }
        // A_ij = sum_d q_id k_jd 2^{Lam_id - Lam_jd}, j <= i < L, elementwise
        {
            const float *lg = reinterpret_cast<const float *>(smem + X_LAM);
            for (int idx = tid; idx < CH * CH; idx += NT) {
                const int i = idx >> 6, j = idx & 63;
                float acc = 0.f;
                if (j <= i && i < L) {
                    for (int dd = 0; dd < D; ++dd)
                        acc = fmaf(bf16f(sQ[i * D + dd]) * bf16f(sK[j * D + dd]),
                                   ex2(lg[i * D + dd] - lg[j * D + dd]), acc);
                }
                *reinterpret_cast<float *>(smem + X_B2 + t_off(192, i, j)) = rna_tf32(acc);
            }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncthreads();
        if (tid == kIssuer) {
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < CH / 8; ++kk) {
                const uint32_t koff = (kk >> 2) * (192 * 128) + (kk & 3) * 32;
                mma_tf32_ts(tmem + tm_o, tmem + TM_V + kk * 8, sdesc_sw128(sb + X_B2 + koff, 16, 1024),
                            IDT_N64, 1);
            }
            tc_commit(bar_o);
        }
        if (!wait_all(kIssuer, bar_o, ph_o))
            return false;
        state_pass(smem, tmem, gslot, nullptr, false);          // S <- diag(2^{Lam_last}) S
        tc_fence_before();
        __syncthreads();
        if (tid == kIssuer) {
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < CH / 8; ++kk) {
                const uint32_t koff = (kk >> 2) * (192 * 128) + (kk & 3) * 32 + 64 * 128;
                mma_tf32_ts(tmem + TM_S, tmem + TM_V + kk * 8, sdesc_sw128(sb + X_B2 + koff, 16, 1024),
                            IDT_N128, 1);
            }
            tc_commit(bar_s);
        }
        if (!wait_all(kIssuer, bar_s, ph_s))
            return false;
        state_pass(smem, tmem, -1, ckpt_slot(seg_end), false);   // checkpoint and |S| of the final state
        out_epilogue(tmem, p.o + (((int64_t)p.row0[b] + tok_s) * p.n_heads + h) * D, tstride, L, par, false);
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        return true;
    };

    // ---- a run of long segments on the fast path, the two groups of warps in a pipeline:
    // the builders stage and build segment k+1 while the state warps finish segment k.
    // Handoffs (each mbarrier has one waiting thread and one arriving party):
    //   bar_built: builders -> state warps, segment k built (operands, V^T, guard maxima)
    //   bar_go:    state warps -> builders, the decision on segment k is made (sMisc[2]);
    //              when it is fast, it also means the operand set of segment k+1 is free
    //              (the products of segment k-1 are complete)
    // A run ends after the last long segment, before a segment whose own inputs the guard
    // sends to the exact path, or before a segment whose state bound fails: a decision inside a
    // run only has a bound on the state it starts from (that state is still being computed), so
    // such a segment starts a new run, whose first decision reads the measured state exactly as
    // a run resumed from a checkpoint at that segment does.  The groups then meet CTA-wide.
    // No MMA is in flight at either end.
    auto outp = [&](int64_t t) { return p.o + (((int64_t)p.row0[b] + t) * p.n_heads + h) * D; };
    int kseq = 0;   // long segments of the current run so far (slot of 2^{Lam_last}: kseq mod 4)
    auto builder_run = [&](int64_t rpos, int64_t rtok) {
        int par = 0;
        while (true) {
            const int L = seg_len(rpos);
            if (!wait_group(1, kLoader, bar_tma, ph_tma))
                return;
            tma_pending = false;
            if (tid == kLoader && !prefetched) {
                // once the first segment has landed (the state and the first segment are
                // not queued behind these): the next kPrefetch segments into L2
                prefetched = true;
                for (int j = 1; j <= kPrefetch; ++j)
                    prefetch(rtok + L + (int64_t)CH * (j - 1));
            }
            build_fast(smem, tmem, L, par, kseq & 3);
            fence_proxy_async_smem();
            tc_fence_before();
            if (!sync_group(1))
                return;
            const bool next_long = is_long(rpos + L);
            if (tid == kLoader) {
                mbar_arrive(bar_built);
                // the staged rows are consumed: stage the next segment (long or short) now;
                // an exact decision on this one reloads it
                if (rpos + L < end)
                    issue_tma(rtok + L);
                // D_A = Q~ K~^T of this segment, into its own buffer (the state warps wait on
                // bar_a / bar_a1 by parity before they read it)
                tc_fence_after();
                const uint32_t setb = sb + (uint32_t)par * SET_BYTES;
#pragma unroll 1
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
                    mma_f16_ss(tmem + (par ? TM_A1 : TM_A0), sdesc_sw128(setb + S_QH + koff, 16, 1024),
                               sdesc_sw128(setb + S_KH + koff, 16, 1024), IDF_N64, kk > 0);
                }
                tc_commit(par ? bar_a1 : bar_a);
            }
            if (!wait_group(1, kLoader, bar_go, ph_go))
                return;
            if (sMisc[2] == 0 || !next_long)
                return;
            rpos += L;
            rtok += L;
            par ^= 1;
            ++kseq;
        }
    };
    auto state_run = [&](int64_t rpos, int64_t rtok) {
        int par = 0;
        bool pend = false;
        uint32_t stop = 0;   // why the run ended: 0 done or short segment, 1 exact, 2 new run
        int pend_par = 0, pend_L = 0, pend_g = 0;
        int64_t pend_tok = 0, pend_end = 0;
        float mk_cur = 0.f, mv_cur = 0.f;
        if (!wait_group(2, kIssuer, bar_built, ph_built))
            return;
        // first segment of a run: the measured state (float32 maximum of the last state pass
        // or of the loaded state)
        bool state_ok;
        bool fast = guard(state_max(), state_ok) && state_ok;
        if (tid == kIssuer) {
            sMisc[2] = fast ? 1u : 0u;
            if (!fast)
                mbar_arrive(bar_go);
        }
        stop = fast ? 0u : 1u;
        // a segment sent to the exact path: its (unused) D_A product is drained first
        if (!fast && !wait_group(2, kIssuer, bar_a, ph_a0))
            return;
        while (fast) {
            const int L = seg_len(rpos);
            const int64_t seg_end = rpos + L;
            mk_cur = mk_new;
            mv_cur = mv_new;
            if (pend && !wait_group(2, kIssuer, bar_o, ph_o))
                return;
            // the products of the previous segment are complete: its operand set is free
            if (tid == kIssuer)
                mbar_arrive(bar_go);
            state_pass(smem, tmem, pend ? pend_g : -1, pend ? ckpt_slot(pend_end) : nullptr, true);
            tc_fence_before();
            if (!sync_group(2))
                return;
            const uint32_t setb = sb + (uint32_t)par * SET_BYTES;
            if (tid == kIssuer) {
                // D_O = S^T Q~^T (the N = 192 product below accumulates onto it in order)
                tc_fence_after();
#pragma unroll 1
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * 8192 + (kk & 3) * 32;
                    mma_f16_ts(tmem + (par ? TM_O1 : TM_O0), tmem + TM_SH + kk * 8,
                               sdesc_sw128(setb + S_QH + koff, 16, 1024), IDF_N64, kk > 0);
                }
            }
            if (pend)
                out_epilogue(tmem, outp(pend_tok), tstride, pend_L, pend_par, true);
            // D_A of this segment (issued by the builders' loader)
            if (!(par ? wait_group(2, kIssuer, bar_a1, ph_a1) : wait_group(2, kIssuer, bar_a, ph_a0)))
                return;
            a_build(smem, tmem, par);
            fence_proxy_async_smem();
            tc_fence_before();
            if (!sync_group(2))
                return;
            if (tid == kIssuer) {
                tc_fence_after();
                const uint32_t vt = tmem + TM_V + 32 * par;
#pragma unroll 1
                for (int kk = 0; kk < CH / 16; ++kk)
                    mma_f16_ts(tmem + (par ? TM_S : TM_O0), vt + kk * 8,
                               sdesc_sw128(setb + S_B2H + kk * 32, 16, 1024), IDF_N192, 1);
                tc_commit(bar_o);
            }
            pend = true;
            pend_par = par;
            pend_tok = rtok;
            pend_L = L;
            pend_end = seg_end;
            pend_g = kseq & 3;
            rpos = seg_end;
            rtok += L;
            par ^= 1;
            ++kseq;
            if (!is_long(rpos))
                break;
            // the builders' next segment, and the decision on it: the state it starts from is
            // bounded by the fp16 copy's largest |S| at this segment's start plus this segment's
            // largest update, 64 max|k| max|v| (the decay factors are <= 1)
            if (!wait_group(2, kIssuer, bar_built, ph_built))
                return;
            const bool inputs_ok =
                guard((state_max() + 64.0f * mk_cur * mv_cur) * kBoundMargin, state_ok);
            fast = inputs_ok && state_ok;
            if (tid == kIssuer) {
                sMisc[2] = fast ? 1u : 0u;
                if (!fast)
                    mbar_arrive(bar_go);
            }
            stop = fast ? 0u : (inputs_ok ? 2u : 1u);
            if (!fast && !(par ? wait_group(2, kIssuer, bar_a1, ph_a1) : wait_group(2, kIssuer, bar_a, ph_a0)))
                return;
        }
        if (pend) {
            if (!wait_group(2, kIssuer, bar_o, ph_o))
                return;
            state_pass(smem, tmem, pend_g, ckpt_slot(pend_end), false);
            out_epilogue(tmem, outp(pend_tok), tstride, pend_L, pend_par, false);
            tc_fence_before();
            if (!sync_group(2))
                return;
        }
        if (tid == kIssuer) {
            sMisc[3] = stop;
            sRun[0] = rpos;
            sRun[1] = rtok;
        }
    };

    // failure-detection hook (tests only): every thread joins one CTA-wide wait on an
    // mbarrier that nothing completes before the first decision (bar_go, phase 0); the
    // loader's bounded wait runs out and raises the abort flag, and the CTA leaves through
    // the abort path below
    if (p.stall_for_test) {
        uint32_t ph_stall = 0;
        wait_all(kLoader, bar_go, ph_stall);
    }

    int64_t pos = pos0, tok = 0;
    while (!aborted && pos < end) {
        const int L = seg_len(pos);
        if (L <= kShort) {
            // a leading or trailing short segment (its inputs are staged or in flight)
            if (!wait_tma())
                break;
            short_segment(tok, L, pos + L);
            pos += L;
            tok += L;
            continue;
        }
        if (builder)
            builder_run(pos, tok);
        else
            state_run(pos, tok);
        if (!sync_all())
            break;
        tc_fence_after();
        const uint32_t stop = sMisc[3];
        pos = sRun[0];
        tok = sRun[1];
        kseq = 0;
        if (stop != 0) {
            // the segment at pos takes the exact path (1) or starts a new run (2): restage its
            // inputs (the copy of the next segment may be in flight)
            const int Lx = seg_len(pos);
            if (tid == kLoader) {
                if (tma_pending && !mbar_wait_bounded(bar_tma, ph_tma, kTimeoutNs))
                    sMisc[1] = 1;
                if (tma_pending)
                    ph_tma ^= 1;
                issue_tma(tok);
            }
            if (stop == 2)
                continue;   // the new run waits for the copy
            // every thread runs the exact segment
            if (!wait_tma())
                break;
            if (!exact_segment(tok, Lx, 0, 0, pos + Lx))
                break;
            pos += Lx;
            tok += Lx;
            if (tid == kLoader && pos < end)
                issue_tma(tok);
        }
    }

    if (!aborted) {
        if (worker) {
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
        }
    } else {
        // let this CTA's own copies and MMAs drain (bounded) before its memory goes away
        if (tid == kLoader) {
            report(p.d_err, HS_DEVERR_TIMEOUT);
            if (n_tma > 0)
                mbar_wait_bounded(bar_tma, (n_tma - 1) & 1, kTimeoutNs);
            tc_commit(bar_ld);   // the D_A products this thread issued
            mbar_wait_bounded(bar_ld, 0, kTimeoutNs);
        }
        if (tid == kIssuer) {
            tc_commit(bar_s);
            mbar_wait_bounded(bar_s, ph_s, kTimeoutNs);
        }
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

bool gla_chunked_tc_supported(int d)
{
    return d == D;
}

cudaError_t launch_gla_chunked_tc(const GlaParams &p, int d, cudaStream_t s)
{
    if (!gla_chunked_tc_supported(d))
        return cudaErrorNotSupported;
    TmaMaps maps;
    const uint64_t inner = (uint64_t)p.n_heads * D;
    // rows up to the last token any problem has: copies never read beyond the tokens the
    // caller passed (boxes reaching further are zero-filled), so q/k/v/log_g may be
    // offset views whose last rows run past the end of the allocation
    uint64_t rows = 0;
    for (int32_t b = 0; b < p.batch; ++b) {
        const uint64_t r = (uint64_t)p.row0[b] + (uint64_t)p.n_tokens[b];
        rows = r > rows ? r : rows;
    }
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
