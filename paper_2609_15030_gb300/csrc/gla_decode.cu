// Gated linear attention, one token per problem (a decode step):
//     S' = diag(g) S + k v^T,   o = q S',   g = exp(a).
//
// One CTA per (problem, head), d^2/32 threads.  Thread (rg, cg) holds rows
// [16*rg, 16*rg+16) and columns [2*cg, 2*cg+2) of the d x d float32 state in
// registers; the lanes of a warp are column groups, so every state load and
// store of a warp is 256 contiguous bytes of one row.  Two columns per thread
// measured 2.90 us per bench decode step, against 3.05 us for four columns over
// half as many threads and 3.16 us for one column over twice as many.  The
// token's inputs are read straight from global memory (each row group's q/k/a
// are one broadcast per warp) before the state (issued in this order the step
// was 3.0 us instead of 3.2 us with four columns per thread), the state goes
// back to memory as soon as it is updated, and the row groups' partial outputs
// meet once in shared memory: one block-wide barrier per step.
//
// The arithmetic is exactly that of the per-token recurrent kernel and of the
// short segments of the chunked tensor-core kernel: g = expf(a); every element
// becomes fmaf(g_d, S[d][e], k_d * v_e); each group of 16 rows gives a partial
// dot product by one fma chain in increasing row order; o_e is the left-to-right
// sum of the group partials.  So the three kernels agree bit for bit.
#include "hs_internal.cuh"

namespace hs {
namespace {

__device__ __forceinline__ void prefetch_l2(const void *p)
{
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ float bf16_lo(uint32_t w)
{
    return __uint_as_float(w << 16);
}

__device__ __forceinline__ float bf16_hi(uint32_t w)
{
    return __uint_as_float(w & 0xFFFF0000u);
}

template <int D>
__global__ void __launch_bounds__((D / 2) * (D / 16)) gla_decode_kernel(const __grid_constant__ GlaParams p)
{
    constexpr int NCG = D / 2;        // column groups of 2 (lanes)
    constexpr int NRG = D / 16;       // row groups of 16
    __shared__ __align__(16) float spart[NRG][D];
    const int b = blockIdx.x / p.n_heads;
    const int h = blockIdx.x - b * p.n_heads;
    if (p.n_tokens[b] <= 0)
        return;
    const int64_t pos0 = p.pos0[b];
    const int tid = threadIdx.x;
    const int cg = tid % NCG;
    const int rg = tid / NCG;
    {
        const int64_t prow = ((int64_t)p.row0[b]) * p.n_heads + h;
        constexpr int LB = D / 64;     // 128-byte lines of one bf16 row (a float row is 2 LB)
        if (tid < LB)
            prefetch_l2(reinterpret_cast<const char *>(p.q + prow * D) + 128 * tid);
        else if (tid < 2 * LB)
            prefetch_l2(reinterpret_cast<const char *>(p.k + prow * D) + 128 * (tid - LB));
        else if (tid < 3 * LB)
            prefetch_l2(reinterpret_cast<const char *>(p.v + prow * D) + 128 * (tid - 2 * LB));
        else if (tid < 5 * LB)
            prefetch_l2(reinterpret_cast<const char *>(p.log_g + prow * D) + 128 * (tid - 3 * LB));
    }
    pdl_wait_and_release();

    // the token's inputs first (their lines were requested into L2 above), then the state
    const int64_t row = ((int64_t)p.row0[b]) * p.n_heads + h;   // the call's one token
    const uint4 *q8 = reinterpret_cast<const uint4 *>(p.q + row * D + 16 * rg);
    const uint4 *k8 = reinterpret_cast<const uint4 *>(p.k + row * D + 16 * rg);
    const uint32_t v2 = *reinterpret_cast<const uint32_t *>(p.v + row * D + 2 * cg);
    uint32_t qw[8], kw[8];
    *reinterpret_cast<uint4 *>(&qw[0]) = q8[0];
    *reinterpret_cast<uint4 *>(&qw[4]) = q8[1];
    *reinterpret_cast<uint4 *>(&kw[0]) = k8[0];
    *reinterpret_cast<uint4 *>(&kw[4]) = k8[1];
    // the row group's 16 gates: lane l computes g of row 16 rg + (l mod 16) once, and every
    // lane reads the value it needs from the lane of its half-warp that holds it (the same
    // expf, so bit-identical).  A row group spans d/64 warps, so both halves of a warp compute
    // the same 16 values.
    const int lane = tid & 31;
    const float g_own = expf(p.log_g[row * D + 16 * rg + (lane & 15)]);

    float *st = p.state + ((int64_t)b * p.n_heads + h) * D * D;
    float2 S[16];
#pragma unroll
    for (int r = 0; r < 16; ++r)
        S[r] = *reinterpret_cast<const float2 *>(st + (int64_t)(16 * rg + r) * D + 2 * cg);
    const float2 vv = make_float2(bf16_lo(v2), bf16_hi(v2));

    float2 acc = make_float2(0.f, 0.f);
#pragma unroll
    for (int r = 0; r < 16; ++r) {
        const float g = __shfl_sync(0xffffffffu, g_own, (lane & 16) | r);
        const float kk = (r & 1) ? bf16_hi(kw[r >> 1]) : bf16_lo(kw[r >> 1]);
        const float qq = (r & 1) ? bf16_hi(qw[r >> 1]) : bf16_lo(qw[r >> 1]);
        S[r].x = fmaf(g, S[r].x, kk * vv.x);
        S[r].y = fmaf(g, S[r].y, kk * vv.y);
        acc.x = fmaf(qq, S[r].x, acc.x);
        acc.y = fmaf(qq, S[r].y, acc.y);
    }
#pragma unroll
    for (int r = 0; r < 16; ++r)
        *reinterpret_cast<float2 *>(st + (int64_t)(16 * rg + r) * D + 2 * cg) = S[r];
    *reinterpret_cast<float2 *>(&spart[rg][2 * cg]) = acc;

    const int C = p.ckpt_interval;
    if (C > 0 && p.ckpt_slots != nullptr && (pos0 + 1) % C == 0) {
        float *slot = p.ckpt_slots[p.ck_base[b]];
        if (slot == nullptr) {
            if (tid == 0)
                report(p.d_err, HS_DEVERR_NULL);
        } else if ((reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
            if (tid == 0)
                report(p.d_err, HS_DEVERR_MISALIGNED);
        } else {
            slot += (int64_t)h * D * D;
#pragma unroll
            for (int r = 0; r < 16; ++r)
                *reinterpret_cast<float2 *>(slot + (int64_t)(16 * rg + r) * D + 2 * cg) = S[r];
        }
    }
    __syncthreads();
    // o_e = ((p_0 + p_1) + p_2) + ... over the row groups
    if (tid < D) {
        float sum = spart[0][tid];
#pragma unroll
        for (int g = 1; g < NRG; ++g)
            sum += spart[g][tid];
        p.o[row * D + tid] = sum;
    }
}

}  // namespace

cudaError_t launch_gla_decode(const GlaParams &p, int d, cudaStream_t s)
{
    const unsigned grid = (unsigned)p.batch * (unsigned)p.n_heads;
    if (d == 128)
        return launch_pdl(gla_decode_kernel<128>, dim3(grid), dim3(512), 0, s, p);
    return launch_pdl(gla_decode_kernel<64>, dim3(grid), dim3(128), 0, s, p);
}

}  // namespace hs
