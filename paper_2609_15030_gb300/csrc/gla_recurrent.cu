// Gated linear attention, one token at a time on CUDA cores:
//     S_t = diag(g_t) S_{t-1} + k_t v_t^T,   o_t = q_t S_t,   g_t = exp(a_t).
// (The paper runs its linear layers on FLA kernels and prints no recurrence;
// this is the form the library implements.)
//
// One CTA owns one (problem, head) and keeps its d x d float32 state in
// registers for the whole call, as 16 x 4 blocks (16 key rows, 4 value
// columns) per thread, read and written as 16-byte vectors.  Tokens are
// staged eight at a time in shared memory.
//
// Per token the arithmetic is fixed: g = expf(a); every element becomes
// fmaf(g_d, S[d][e], k_d * v_e); partial dot products over each group of 16
// consecutive key rows run as one sequential fma chain in increasing row
// order; o_e is the left-to-right sum of the d/16 group partials.  The chunked
// tensor-core kernel computes short segments with exactly these operations
// (d = 128), so the two kernels agree bit for bit on them.  The order depends
// only on each token's inputs and the incoming state, so resuming from any
// checkpoint reproduces a full recomputation bit for bit.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kTokBlock = 8;

__device__ __forceinline__ float bf16_to_f32(uint16_t x)
{
    return __uint_as_float(((uint32_t)x) << 16);
}

// CTA = (problem, head).  Thread (cg, rg) holds the 16 x 4 block of the state
// with rows [16*rg, 16*rg+16) and columns [4*cg, 4*cg+4): a warp covers 16-byte
// pieces of whole rows, so state loads and stores are fully coalesced vectors.
template <int D>
__global__ void __launch_bounds__((D / 4) * (D / 16)) gla_recurrent_kernel(const __grid_constant__ GlaParams p)
{
    constexpr int NCG = D / 4;        // column groups of 4
    constexpr int NRG = D / 16;       // row groups of 16
    constexpr int NTH = NCG * NRG;
    __shared__ __align__(16) float sq[kTokBlock][D], sk[kTokBlock][D], sg[kTokBlock][D], sv[kTokBlock][D];
    __shared__ __align__(16) float spart[kTokBlock][NRG][D];

    const int b = blockIdx.x / p.n_heads;
    const int h = blockIdx.x - b * p.n_heads;
    const int n = p.n_tokens[b];
    if (n <= 0)
        return;
    const int64_t pos0 = p.pos0[b];
    pdl_wait_and_release();
    const int tid = threadIdx.x;
    const int cg = tid % NCG;
    const int rg = tid / NCG;
    const int C = p.ckpt_interval;

    float *st = p.state + ((int64_t)b * p.n_heads + h) * D * D;
    float4 S[16];   // S[r] = state row 16*rg + r, columns 4*cg .. 4*cg+3
#pragma unroll
    for (int r = 0; r < 16; ++r)
        S[r] = *reinterpret_cast<const float4 *>(st + (int64_t)(16 * rg + r) * D + 4 * cg);

    for (int t0 = 0; t0 < n; t0 += kTokBlock) {
        const int tb = min(kTokBlock, n - t0);
        for (int idx = tid; idx < tb * D; idx += NTH) {
            const int tt = idx / D, d = idx - (idx / D) * D;
            const int64_t row = ((int64_t)p.row0[b] + t0 + tt) * p.n_heads + h;
            sq[tt][d] = bf16_to_f32(p.q[row * D + d]);
            sk[tt][d] = bf16_to_f32(p.k[row * D + d]);
            sv[tt][d] = bf16_to_f32(p.v[row * D + d]);
            sg[tt][d] = expf(p.log_g[row * D + d]);
        }
        __syncthreads();
        for (int tt = 0; tt < tb; ++tt) {
            const float4 v4 = *reinterpret_cast<const float4 *>(&sv[tt][4 * cg]);
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
            for (int r = 0; r < 16; ++r) {
                const int i = 16 * rg + r;
                const float g = sg[tt][i], kk = sk[tt][i], qq = sq[tt][i];
                S[r].x = fmaf(g, S[r].x, kk * v4.x);
                S[r].y = fmaf(g, S[r].y, kk * v4.y);
                S[r].z = fmaf(g, S[r].z, kk * v4.z);
                S[r].w = fmaf(g, S[r].w, kk * v4.w);
                acc.x = fmaf(qq, S[r].x, acc.x);
                acc.y = fmaf(qq, S[r].y, acc.y);
                acc.z = fmaf(qq, S[r].z, acc.z);
                acc.w = fmaf(qq, S[r].w, acc.w);
            }
            *reinterpret_cast<float4 *>(&spart[tt][rg][4 * cg]) = acc;
            if (C > 0 && p.ckpt_slots != nullptr) {
                const int64_t end = pos0 + t0 + tt + 1;
                if (end % C == 0) {
                    const int64_t slot_idx = p.ck_base[b] + (end / C - pos0 / C - 1);
                    float *slot = p.ckpt_slots[slot_idx];
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
                            *reinterpret_cast<float4 *>(slot + (int64_t)(16 * rg + r) * D + 4 * cg) = S[r];
                    }
                }
            }
        }
        if (t0 + tb >= n) {
            // final state out before the output reduction, so the store drains behind it
#pragma unroll
            for (int r = 0; r < 16; ++r)
                *reinterpret_cast<float4 *>(st + (int64_t)(16 * rg + r) * D + 4 * cg) = S[r];
        }
        __syncthreads();
        for (int idx = tid; idx < tb * D; idx += NTH) {
            const int tt = idx / D, e = idx - (idx / D) * D;
            float sum = spart[tt][0][e];
#pragma unroll
            for (int g = 1; g < NRG; ++g)
                sum += spart[tt][g][e];
            const int64_t row = ((int64_t)p.row0[b] + t0 + tt) * p.n_heads + h;
            p.o[row * D + e] = sum;
        }
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_gla_recurrent(const GlaParams &p, int d, cudaStream_t s)
{
    const unsigned grid = (unsigned)p.batch * (unsigned)p.n_heads;
    if (d == 128)
        return launch_pdl(gla_recurrent_kernel<128>, dim3(grid), dim3(256), 0, s, p);
    return launch_pdl(gla_recurrent_kernel<64>, dim3(grid), dim3(64), 0, s, p);
}

}  // namespace hs
