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
constexpr int NW = 256;   // worker threads (warps 0..7): operands and epilogues
constexpr int NT = NW + 32;  // + one warp whose lane 0 issues every MMA and TMA copy
constexpr int kIssuer = NW;
constexpr int kShort = 8; // segments of at most this many tokens run token by token
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kFastMinLog2 = -64.0f;      // factorised form if every 2^{Lam_last} >= 2^-64
constexpr uint64_t kTimeoutNs = 1000000000ull;
constexpr int kPrefetch = 3;                // segments requested into L2 ahead of the staged one

// shared memory map (offsets from a 1024-byte aligned base).  Every tf32
// shared-memory operand is K-major (kind::tf32 takes no transposed
// shared-memory operand); V^T is the A operand of both token-contracting
// products and lives in tensor memory.
constexpr uint32_t OFF_QT = 0;          // Q~   [64 tok i][128 d]  tf32, swizzled   32 KiB
constexpr uint32_t OFF_KT = 32768;      // K~   [64 tok j][128 d]                   32 KiB
constexpr uint32_t OFF_B2 = 65536;      // [A ; K~^T] [64 i + 128 d][64 tok j]  (K^^T on the exact path)  48 KiB
constexpr uint32_t OFF_SQ = 114688;     // staged q  bf16 [64][128]                16 KiB
constexpr uint32_t OFF_SK = 131072;     // staged k                                 16 KiB
constexpr uint32_t OFF_SV = 147456;     // staged v                                 16 KiB
constexpr uint32_t OFF_SG = 163840;     // staged log-gates f32 [64][128]           32 KiB
constexpr uint32_t OFF_GAM = 196608;    // 2^{Lam_last} per key dim, one buffer per chunk parity   1 KiB
constexpr uint32_t OFF_TOT = 197632;    // per-half log2-decay totals [2][128]      1 KiB
constexpr uint32_t OFF_BAR = 198656;    // 4 mbarriers
constexpr uint32_t OFF_MISC = 198688;   // TMEM base address, abort flag, exact-path flags (per parity)
constexpr uint32_t SMEM_BYTES = 198720 + 1024;
constexpr uint32_t STAGE_BYTES = 3 * 16384 + 32768;
constexpr uint32_t SLAB = 64 * 128;     // one 32-column slab of a 64-row operand
constexpr uint32_t SLAB_B2 = 192 * 128; // one 32-column slab of the 192-row operand [A ; K~^T]

// tensor memory: the output accumulator D_O alternates between two buffers by chunk
// parity, placed on either side of S^T so that [D_O0 | S^T] and [S^T | D_O1] are each one
// N=192 accumulator; V^T alternates likewise.  Even chunks order the 192-row operand as
// [A ; K~^T], odd chunks as [K~^T ; A].
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t TM_O0 = 0;           // D_O of even chunks (lane e, col i), 64 cols
constexpr uint32_t TM_S = 64;           // S^T  128 lanes x 128 cols
constexpr uint32_t TM_O1 = 192;         // D_O of odd chunks
constexpr uint32_t TM_A = 256;          // D_A  128 lanes x 64 cols (lanes 0..63 used)
constexpr uint32_t TM_V = 320;          // V^T  2 x 64 cols (lane e, col j)

constexpr uint32_t IDESC_N64 = idesc_tf32(128, 64, 0, 0);    // M=128, N=64, K-major x K-major
constexpr uint32_t IDESC_N128 = idesc_tf32(128, 128, 0, 0);  // M=128, N=128
constexpr uint32_t IDESC_N192 = idesc_tf32(128, 192, 0, 0);  // M=128, N=192

struct TmaMaps {
    CUtensorMap q, k, v, g;
};


// byte offset of element (i, j) of A, stored from row rowA of the 192-row operand
__device__ __forceinline__ uint32_t a_off(int rowA, int i, int j)
{
    return (uint32_t)((j >> 5) * SLAB_B2 + (rowA + i) * 128 + ((((j & 31) >> 2) ^ (i & 7)) << 4) +
                      ((j & 3) << 2));
}

// 16-byte chunk col4 (tokens 4*col4 .. 4*col4+3) of row d of K~^T, stored from row rowK
__device__ __forceinline__ uint32_t ktt_chunk(int rowK, int d, int col4)
{
    return (uint32_t)((col4 >> 3) * SLAB_B2 + (rowK + d) * 128 + (((col4 & 7) ^ (d & 7)) << 4));
}

__device__ __forceinline__ float warp_min(float v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        v = fminf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float bf16f(uint16_t x)
{
    return __uint_as_float(((uint32_t)x) << 16);
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
    float *sTot = reinterpret_cast<float *>(smem + OFF_TOT);
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
    const int C = p.ckpt_interval;

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
    const bool worker = warp < 8;
    const uint32_t lrow = (uint32_t)((warp & 3) * 32) << 16;   // this warp's TMEM lane quarter
    const int colhalf = warp >> 2;
    const int e_own = (warp & 3) * 32 + lane;                  // TMEM lane = value dim e
    // operand-building map: worker owns key dim d = e_own for tokens [32*th, 32*th+32)
    const int d = e_own;
    const int th = colhalf;
    uint32_t nat[8];       // byte offset of (row 32*th + r, col d) in a 64-row operand
    {
        const uint32_t base = (uint32_t)((warp & 3) * SLAB + (32 * th) * 128 + ((lane & 3) << 2));
        const int cd = lane >> 2;
#pragma unroll
        for (int r = 0; r < 8; ++r)
            nat[r] = base + r * 128 + ((uint32_t)(cd ^ r) << 4);
    }

    // issuer bookkeeping (lane 0 of warp 8) of work in flight, for the abort path
    bool tma_inflight = false;
    uint32_t ph_tma = 0, ph_a = 0, ph_o = 0, ph_s = 0;
    bool aborted = false;

    // L2 prefetch of the 64 tokens from local position t (if any are this problem's)
    auto prefetch = [&](int64_t t) {
        if (t >= n)
            return;
        const int32_t y = (int32_t)((int64_t)b * p.max_tokens + t);
        const int32_t x = h * D;
        tma_prefetch_2d(&maps.q, x, y);
        tma_prefetch_2d(&maps.k, x, y);
        tma_prefetch_2d(&maps.v, x, y);
        tma_prefetch_2d(&maps.g, x, y);
    };
    // staged inputs of the segment at local position tok_local; segments after the
    // first start on the 64-token grid, so the segment kPrefetch ahead starts at
    // tok_local + 64 * kPrefetch and is requested into L2 now
    auto issue_tma = [&](int64_t tok_local) {
        const int32_t y = (int32_t)((int64_t)b * p.max_tokens + tok_local);
        const int32_t x = h * D;
        mbar_arrive_expect_tx(bar_tma, STAGE_BYTES);
        tma_load_2d(sb + OFF_SQ, &maps.q, x, y, bar_tma);
        tma_load_2d(sb + OFF_SK, &maps.k, x, y, bar_tma);
        tma_load_2d(sb + OFF_SV, &maps.v, x, y, bar_tma);
        tma_load_2d(sb + OFF_SG, &maps.g, x, y, bar_tma);
        tma_inflight = true;
        if (tok_local > 0)
            prefetch(tok_local + (int64_t)CH * kPrefetch);
    };
    // the issuer waits on an mbarrier, then everyone meets; false if a wait ran out
    auto wait_all = [&](uint32_t bar, uint32_t &ph) -> bool {
        if (tid == kIssuer && !mbar_wait_bounded(bar, ph, kTimeoutNs))
            sMisc[1] = 1;
        __syncthreads();
        tc_fence_after();
        ph ^= 1;
        if (sMisc[1]) {
            aborted = true;
            return false;
        }
        return true;
    };
    auto wait_tma = [&]() -> bool {
        const bool ok = wait_all(bar_tma, ph_tma);
        if (tid == kIssuer)
            tma_inflight = false;
        return ok;
    };
    auto seg_len = [&](int64_t at) -> int { return (int)(min(end, (at / CH + 1) * CH) - at); };
    auto ckpt_slot = [&](int64_t seg_end) -> float * {
        if (!(C > 0 && seg_end % C == 0 && p.ckpt_slots != nullptr))
            return nullptr;
        float *slot = p.ckpt_slots[p.ck_base[b] + (seg_end / C - pos0 / C - 1)];
        if (slot == nullptr || (reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
            if (tid == 0)
                report(p.d_err, slot == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
            return nullptr;
        }
        return slot + (int64_t)h * D * D;
    };

    if (tid == kIssuer) {
        issue_tma(0);
        // the first kPrefetch segments after the first one
        const int64_t t1 = min(end, (pos0 / CH + 1) * CH) - pos0;
        for (int j = 0; j < kPrefetch; ++j)
            prefetch(t1 + (int64_t)CH * j);
    }

    // incoming state -> TMEM, transposed: S^T[e][d] = state[d][e]
    float *st_g = p.state + ((int64_t)b * p.n_heads + h) * D * D;
    if (worker) {
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

    // ---- a short segment (<= kShort tokens, staged inputs already waited for): the
    // per-token recurrence with the recurrent kernel's exact operation order (fma chains
    // over groups of 16 key rows, group partials summed left to right)
    auto short_segment = [&](int64_t tok_s, int L, int64_t seg_end) {
        for (int idx = tid; idx < L * D; idx += NT)
            sG[idx] = expf(sG[idx]);
        __syncthreads();
        float *part = reinterpret_cast<float *>(smem + OFF_QT);   // [kShort][8 groups][128]
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
            if (slot != nullptr) {
#pragma unroll
                for (int r = 0; r < 64; ++r)
                    slot[(int64_t)(colhalf * 64 + r) * D + e_own] = S[r];
            }
            tmem_wait_st();
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == kIssuer && seg_end < end)
            issue_tma(tok_s + L);
        float *ob = p.o + (((int64_t)b * p.max_tokens + tok_s) * p.n_heads + h) * D;
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

    // ---- prep of a long segment (staged inputs already waited for): zero the staged rows
    // past the segment, cumulative log2-gates (per-thread scan of 32 tokens, halves joined
    // through shared memory, path vote by a warp-shuffle min), Q~ into shared memory and
    // V^T into tensor memory buffer `par`.  Leaves lam[] in registers.
    float lam[32];
    float last = 0.f;
    auto prep = [&](int L, int par) {
        if (L < CH) {
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
        float run = 0.f;
        if (worker) {
#pragma unroll
            for (int x = 0; x < 32; ++x) {
                run = fmaf(sG[(32 * th + x) * D + d], kLog2e, run);
                lam[x] = run;
            }
            sTot[th * D + d] = run;
        }
        if (tid == 0)
            sMisc[2 + par] = 0;   // exact-path flag of this segment
        __syncthreads();
        if (worker) {
            const float tot0 = sTot[d];
            last = tot0 + sTot[D + d];   // Lam_last of key dim d
            if (th) {
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    lam[x] = tot0 + lam[x];
            } else {
                reinterpret_cast<float *>(smem + OFF_GAM)[par * D + d] = ex2(last);
            }
            const float wmin = warp_min(last);
            if (lane == 0 && wmin < kFastMinLog2)
                sMisc[2 + par] = 1;
            float vtr[32];
#pragma unroll
            for (int x = 0; x < 32; ++x) {
                const int i = 32 * th + x;
                const float qv = bf16f(sQ[i * D + d]);
                vtr[x] = bf16f(sV[i * D + d]);
                *reinterpret_cast<float *>(smem + OFF_QT + nat[x & 7] + (x >> 3) * 1024) =
                    rna_tf32(qv * ex2(lam[x]));
            }
            tmem_st32(tmem + lrow + TM_V + 64 * par + 32 * th, vtr);
            tmem_wait_st();
        }
        fence_proxy_async_smem();
    };

    // ---- output epilogue of a processed segment: D_O buffer `par` -> o (lane e, 32 rows)
    auto out_epilogue = [&](int64_t tok_s, int L, int par) {
        if (!worker)
            return;
        float r[32];
        const int ib = colhalf * 32;
        tmem_ld32(tmem + lrow + (par ? TM_O1 : TM_O0) + ib, r);
        tmem_wait_ld();
        float *op = p.o + (((int64_t)b * p.max_tokens + tok_s + ib) * p.n_heads + h) * D + e_own;
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
    };

    // ---- state decay by 2^{Lam_last} (buffer `par`), checkpoint from the same registers
    auto decay_state = [&](int par, float *slot) {
        if (!worker)
            return;
        const float *gam = reinterpret_cast<const float *>(smem + OFF_GAM) + par * D;
#pragma unroll
        for (int c0 = 0; c0 < 64; c0 += 32) {
            const int d0 = colhalf * 64 + c0;
            float r[32];
            tmem_ld32(tmem + lrow + TM_S + d0, r);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                const float4 g4 = *reinterpret_cast<const float4 *>(gam + d0 + 4 * c);
                r[4 * c] *= g4.x;
                r[4 * c + 1] *= g4.y;
                r[4 * c + 2] *= g4.z;
                r[4 * c + 3] *= g4.w;
            }
            tmem_st32(tmem + lrow + TM_S + d0, r);
            if (slot != nullptr) {
#pragma unroll
                for (int x = 0; x < 32; ++x)
                    slot[(int64_t)(d0 + x) * D + e_own] = r[x];
            }
        }
        tmem_wait_st();
    };

    int64_t pos = pos0, tok = 0;
    // leading short segment
    if (seg_len(pos) <= kShort) {
        if (!wait_tma())
            goto finish;
        short_segment(tok, seg_len(pos), pos + seg_len(pos));
        tok += seg_len(pos);
        pos += seg_len(pos);
    }

    // ---- pipelined long segments
    if (pos < end && seg_len(pos) > kShort) {
        if (!wait_tma())
            goto finish;
        prep(seg_len(pos), 0);
        int par = 0;
        bool prev_valid = false;
        int64_t tok_prev = 0;
        int L_prev = 0;
        while (true) {
            const int L = seg_len(pos);
            const int64_t seg_end = pos + L;
            const bool has_next = seg_end < end;
            const int L_next = has_next ? seg_len(seg_end) : 0;
            const bool next_long = has_next && L_next > kShort;
            const uint32_t rowA = par ? 128u : 0u, rowK = par ? 0u : 64u;
            const uint32_t tm_o = par ? TM_O1 : TM_O0;

            // Q~ / V^T of this segment and the previous decay are complete
            tc_fence_before();
            __syncthreads();
            const bool slow = sMisc[2 + par] != 0;
            if (tid == kIssuer) {
                // S^T Q~^T into D_O[par] (A operand read from tensor memory)
                tc_fence_after();
#pragma unroll
                for (int kk = 0; kk < D / 8; ++kk) {
                    const uint32_t koff = (kk >> 2) * SLAB + (kk & 3) * 32;
                    mma_tf32_ts(tmem + tm_o, tmem + TM_S + kk * 8,
                                sdesc_sw128(sb + OFF_QT + koff, 16, 1024), IDESC_N64, kk > 0);
                }
            }
            if (worker) {
                if (!slow) {
                    // K~ token-major (operand of Q~ K~^T) and transposed (state update)
#pragma unroll
                    for (int g = 0; g < 8; ++g) {
                        float4 kt4;
                        float *kv4 = &kt4.x;
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const int x = 4 * g + u;
                            const int i = 32 * th + x;
                            kv4[u] = rna_tf32(bf16f(sK[i * D + d]) * ex2(-lam[x]));
                            *reinterpret_cast<float *>(smem + OFF_KT + nat[x & 7] + (x >> 3) * 1024) = kv4[u];
                        }
                        *reinterpret_cast<float4 *>(smem + OFF_B2 + ktt_chunk(rowK, d, 8 * th + g)) = kt4;
                    }
                } else {
                    // exact path: K^ = k 2^{Lam_last - Lam} (transposed), cumulative log2-gates
                    // token-major in the (unused) K~ buffer
#pragma unroll
                    for (int g = 0; g < 8; ++g) {
                        float4 w;
                        float *wv = &w.x;
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const int x = 4 * g + u;
                            const int i = 32 * th + x;
                            wv[u] = rna_tf32(bf16f(sK[i * D + d]) * ex2(last - lam[x]));
                            reinterpret_cast<float *>(smem + OFF_KT)[i * D + d] = lam[x];
                        }
                        *reinterpret_cast<float4 *>(smem + OFF_B2 + ktt_chunk(rowK, d, 8 * th + g)) = w;
                    }
                }
            }
            fence_proxy_async_smem();
            __syncthreads();
            if (slow) {
                // A_ij = sum_d q_id k_jd 2^{Lam_id - Lam_jd}, j <= i < L, elementwise
                const float *lg = reinterpret_cast<const float *>(smem + OFF_KT);
                for (int idx = tid; idx < CH * CH; idx += NT) {
                    const int i = idx >> 6, j = idx & 63;
                    float acc = 0.f;
                    if (j <= i && i < L) {
                        for (int dd = 0; dd < D; ++dd)
                            acc = fmaf(bf16f(sQ[i * D + dd]) * bf16f(sK[j * D + dd]),
                                       ex2(lg[i * D + dd] - lg[j * D + dd]), acc);
                    }
                    *reinterpret_cast<float *>(smem + OFF_B2 + a_off(rowA, i, j)) = rna_tf32(acc);
                }
                fence_proxy_async_smem();
                __syncthreads();
            }
            if (tid == kIssuer) {
                tc_fence_after();
                if (!slow) {
                    // Q~ K~^T into D_A
#pragma unroll
                    for (int kk = 0; kk < D / 8; ++kk) {
                        const uint32_t koff = (kk >> 2) * SLAB + (kk & 3) * 32;
                        mma_tf32_ss(tmem + TM_A, sdesc_sw128(sb + OFF_QT + koff, 16, 1024),
                                    sdesc_sw128(sb + OFF_KT + koff, 16, 1024), IDESC_N64, kk > 0);
                    }
                }
                tc_commit(bar_a);     // covers S^T Q~^T too: Q~ is free once it arrives
                if (has_next)
                    issue_tma(tok + L);   // the staged inputs have been consumed
            }
            // output of the previous segment while the tensor core works
            if (prev_valid)
                out_epilogue(tok_prev, L_prev, par ^ 1);
            if (!wait_all(bar_a, ph_a))
                break;
            if (!slow && worker && (warp & 3) < 2) {
                // the causally masked intra-chunk matrix A -> rows rowA.. of [A ; K~^T]
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
                    const uint32_t o = (jb >> 5) * SLAB_B2 + (rowA + i) * 128 + ((uint32_t)(c ^ (i & 7)) << 4);
                    *reinterpret_cast<float4 *>(smem + OFF_B2 + o) = w;
                }
            }
            fence_proxy_async_smem();
            tc_fence_before();
            __syncthreads();
            if (tid == kIssuer) {
                // [D_O | S^T] += V^T [A ; K~^T]^T as one N=192 product (V^T from tensor
                // memory); on the exact path only D_O += V^T A^T here
                tc_fence_after();
                const uint32_t vt = tmem + TM_V + 64 * par;
#pragma unroll
                for (int kk = 0; kk < CH / 8; ++kk) {
                    const uint32_t koff = (kk >> 2) * SLAB_B2 + (kk & 3) * 32;
                    if (!slow)
                        mma_tf32_ts(tmem + (par ? TM_S : TM_O0), vt + kk * 8,
                                    sdesc_sw128(sb + OFF_B2 + koff, 16, 1024), IDESC_N192, 1);
                    else
                        mma_tf32_ts(tmem + tm_o, vt + kk * 8,
                                    sdesc_sw128(sb + OFF_B2 + koff + rowA * 128, 16, 1024), IDESC_N64, 1);
                }
                tc_commit(bar_o);
            }
            // next segment's inputs while the tensor core runs the second product
            if (next_long) {
                if (!wait_tma())
                    break;
                prep(L_next, par ^ 1);
            }
            if (!wait_all(bar_o, ph_o))
                break;
            float *slot = ckpt_slot(seg_end);
            decay_state(par, slow ? nullptr : slot);
            if (slow) {
                tc_fence_before();
                __syncthreads();
                if (tid == kIssuer) {
                    tc_fence_after();
                    const uint32_t vt = tmem + TM_V + 64 * par;
#pragma unroll
                    for (int kk = 0; kk < CH / 8; ++kk) {
                        const uint32_t koff = (kk >> 2) * SLAB_B2 + (kk & 3) * 32 + rowK * 128;
                        mma_tf32_ts(tmem + TM_S, vt + kk * 8, sdesc_sw128(sb + OFF_B2 + koff, 16, 1024),
                                    IDESC_N128, 1);
                    }
                    tc_commit(bar_s);
                }
                if (!wait_all(bar_s, ph_s))
                    break;
                if (worker && slot != nullptr) {
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
            prev_valid = true;
            tok_prev = tok;
            L_prev = L;
            pos = seg_end;
            tok += L;
            par ^= 1;
            if (!next_long)
                break;
        }
        if (aborted)
            goto finish;
        // output of the last pipelined segment
        out_epilogue(tok_prev, L_prev, par ^ 1);
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
    }

    // trailing short segment (its inputs were requested by the previous segment)
    if (pos < end) {
        if (!wait_tma())
            goto finish;
        short_segment(tok, seg_len(pos), pos + seg_len(pos));
        pos += seg_len(pos);
    }

finish:
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
    } else if (tid == kIssuer) {
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
    // rows up to the last problem's last token: copies never read beyond the tokens the
    // caller passed (boxes reaching further are zero-filled), so q/k/v/log_g may be
    // offset views whose batch stride runs past the end of the allocation
    const uint64_t rows = (uint64_t)(p.batch - 1) * (uint64_t)p.max_tokens +
                          (uint64_t)p.n_tokens[p.batch - 1];
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
