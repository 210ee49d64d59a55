// Gated linear attention, one token at a time on CUDA cores:
//     S_t = diag(g_t) S_{t-1} + k_t v_t^T,   o_t = q_t S_t,   g_t = exp(a_t).
// (The paper runs its linear layers on FLA kernels and prints no recurrence;
// this is the form the library implements.)
//
// One CTA owns one (problem, head) and keeps its d x d float32 state in
// registers for the whole call: thread (row group rg, column j) holds rows
// [rg*R, rg*R+R) of column j.  Tokens are staged eight at a time in shared
// memory; o_t is the fixed-order sum of the row groups' partial dot products.
// Per token and element: g = expf(a), S = fmaf(g, S, k*v), partial =
// fmaf(q, S, partial) in increasing row order; o = partial_0 + partial_1 + ...
// The chunked tensor-core kernel runs short segments with exactly these
// operations (d = 128), so the two kernels agree bit for bit on them.
// The operation order per token depends only on the token's inputs and the
// incoming state, so resuming from any checkpoint reproduces a full
// recomputation bit for bit.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kThreads = 256;
constexpr int kTokBlock = 8;

__device__ __forceinline__ float bf16_to_f32(uint16_t x)
{
    return __uint_as_float(((uint32_t)x) << 16);
}

template <int D>
__global__ void __launch_bounds__(kThreads) gla_recurrent_kernel(const __grid_constant__ GlaParams p)
{
    constexpr int NG = kThreads / D;  // row groups
    constexpr int R = D / NG;         // rows per thread
    __shared__ float sq[kTokBlock][D], sk[kTokBlock][D], sg[kTokBlock][D], sv[kTokBlock][D];
    __shared__ float spart[kTokBlock][NG][D];

    const int b = blockIdx.x / p.n_heads;
    const int h = blockIdx.x - b * p.n_heads;
    const int n = p.n_tokens[b];
    if (n <= 0)
        return;
    const int64_t pos0 = p.pos0[b];
    const int tid = threadIdx.x;
    const int j = tid % D;
    const int rg = tid / D;
    const int C = p.ckpt_interval;

    float *st = p.state + ((int64_t)b * p.n_heads + h) * D * D;
    float S[R];
#pragma unroll
    for (int r = 0; r < R; ++r)
        S[r] = st[(int64_t)(rg * R + r) * D + j];

    for (int t0 = 0; t0 < n; t0 += kTokBlock) {
        const int tb = min(kTokBlock, n - t0);
        for (int idx = tid; idx < tb * D; idx += kThreads) {
            const int tt = idx / D, d = idx - (idx / D) * D;
            const int64_t row = ((int64_t)b * p.max_tokens + t0 + tt) * p.n_heads + h;
            sq[tt][d] = bf16_to_f32(p.q[row * D + d]);
            sk[tt][d] = bf16_to_f32(p.k[row * D + d]);
            sv[tt][d] = bf16_to_f32(p.v[row * D + d]);
            sg[tt][d] = expf(p.log_g[row * D + d]);
        }
        __syncthreads();
        for (int tt = 0; tt < tb; ++tt) {
            const float vj = sv[tt][j];
            float acc = 0.f;
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int i = rg * R + r;
                S[r] = fmaf(sg[tt][i], S[r], sk[tt][i] * vj);
                acc = fmaf(sq[tt][i], S[r], acc);
            }
            spart[tt][rg][j] = acc;
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
                        for (int r = 0; r < R; ++r)
                            slot[(int64_t)(rg * R + r) * D + j] = S[r];
                    }
                }
            }
        }
        __syncthreads();
        for (int idx = tid; idx < tb * D; idx += kThreads) {
            const int tt = idx / D, e = idx - (idx / D) * D;
            float s = spart[tt][0][e];
#pragma unroll
            for (int g = 1; g < NG; ++g)
                s += spart[tt][g][e];
            const int64_t row = ((int64_t)b * p.max_tokens + t0 + tt) * p.n_heads + h;
            p.o[row * D + e] = s;
        }
        __syncthreads();
    }
#pragma unroll
    for (int r = 0; r < R; ++r)
        st[(int64_t)(rg * R + r) * D + j] = S[r];
}

}  // namespace

cudaError_t launch_gla_recurrent(const GlaParams &p, int d, cudaStream_t s)
{
    const unsigned grid = (unsigned)p.batch * (unsigned)p.n_heads;
    if (d == 128)
        gla_recurrent_kernel<128><<<grid, kThreads, 0, s>>>(p);
    else
        gla_recurrent_kernel<64><<<grid, kThreads, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace hs
