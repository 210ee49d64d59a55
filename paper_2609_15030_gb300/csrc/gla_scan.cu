// The state scan of the segment-parallel prefill (hs_linattn_prefill_scan).
//
// Over a problem's tail [pos0, pos0 + n), split into segments at the multiples of 64 of the
// absolute position grid, the recurrence S_t = diag(g_t) S_{t-1} + k_t v_t^T is linear in
// the state: for a segment of tokens [s, e),
//     S_e = diag(G) S_s + dS,   G = prod_{s<=t<e} g_t = exp(sum_t a_t),
// where dS is the segment's state when it starts from the zero state.  The first pass of the
// prefill computes every segment's dS at once (each segment its own problem for the
// tensor-core kernel); this kernel chains them: per (problem, head) and state element,
// S_{n+1} = G_n S_n + dS_n over the segments in order, recording each segment's start state
// S_n (the last pass computes the outputs from it), the checkpoint at every multiple of C
// and the final state.  Every step is an elementwise fma, so a run resumed at a checkpoint
// on the grid repeats the same operations from there: resumed and full computations agree
// bit for bit.
//
// One CTA per (problem, head, block of 512 state elements); thread i owns four consecutive
// elements of one key row d (a float4).  The D/4 lanes that share a row (a warp at D = 128,
// a half-warp at D = 64) sum the row's log-gates over the segment (256/D tokens per lane, then
// a butterfly, the same order in every lane).  The dS and log-gates of the next kPF segments
// are loaded while the current one is applied.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kThreads = 128;        // float4 per thread: 512 state elements per CTA
constexpr int kChunk = 64;           // segments on the 64-token absolute grid
constexpr int kPF = 4;               // segments loaded ahead

// sum over the W lanes of an aligned group (a butterfly: the same order in every lane)
template <int W>
__device__ __forceinline__ float group_sum(float v)
{
#pragma unroll
    for (int o = W / 2; o > 0; o >>= 1)
        v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <int D>
__global__ void __launch_bounds__(kThreads)
gla_scan_kernel(const __grid_constant__ ScanParams p)
{
    constexpr int BLOCKS = D * D / (4 * kThreads);   // CTAs per (problem, head)
    const int bh = blockIdx.x / BLOCKS;
    const int blk = blockIdx.x - bh * BLOCKS;
    const int b = bh / p.n_heads;
    const int h = bh - b * p.n_heads;
    const int lane = threadIdx.x & 31;
    const int f = (blk * kThreads + threadIdx.x) * 4;  // first of this thread's 4 elements
    const int d = f / D;                               // its key row (one row per warp at D = 128)
    const int64_t pos0 = p.pos0[b];
    const int64_t end = pos0 + p.n_tokens[b];
    const int64_t hs_ = (int64_t)h * D * D + f;        // offset inside one [n_heads][D][D] state
    const int64_t sstride = (int64_t)p.n_heads * D * D;
    const int C = p.ckpt_interval;
    pdl_wait_and_release();

    float4 *st = reinterpret_cast<float4 *>(p.state + (int64_t)b * sstride + hs_);
    float4 S = *st;
    // the sum of the log-gates of key row d over the tokens [s, e) of this problem
    constexpr int W = D / 4;            // lanes per key row
    constexpr int TPL = kChunk / W;     // tokens per lane
    const int r = lane % W;
    auto gate_sum = [&](int64_t s, int64_t e) -> float {
        float v = 0.f;
#pragma unroll
        for (int j = 0; j < TPL; ++j) {
            const int64_t t = s + r + W * j;
            if (t < e) {
                const int64_t row = (int64_t)p.row0[b] + (t - pos0);
                v += p.log_g[(row * p.n_heads + h) * D + d];
            }
        }
        return group_sum<W>(v);
    };
    // a ring of the next kPF segments' dS and log-gate sums, refilled as each is applied, so
    // that the loads of later segments overlap the chain of fmas
    auto seg_end_of = [&](int64_t at) -> int64_t { return min(end, (at / kChunk + 1) * kChunk); };
    float4 dq[kPF];
    float aq[kPF];
    int64_t ld_at = pos0;             // start of the next segment to load
    int32_t ld_seg = p.seg_base[b];
#pragma unroll
    for (int j = 0; j < kPF; ++j) {
        dq[j] = make_float4(0.f, 0.f, 0.f, 0.f);
        aq[j] = 0.f;
        if (ld_at < end) {
            const int64_t e = seg_end_of(ld_at);
            dq[j] = *reinterpret_cast<const float4 *>(p.dS + (int64_t)ld_seg * sstride + hs_);
            aq[j] = gate_sum(ld_at, e);
            ld_at = e;
            ++ld_seg;
        }
    }
    int64_t at = pos0;
    int32_t seg = p.seg_base[b];
    while (at < end) {
#pragma unroll
        for (int j = 0; j < kPF; ++j) {
            if (at < end) {
                const int64_t e = seg_end_of(at);
                *reinterpret_cast<float4 *>(p.Sn + (int64_t)seg * sstride + hs_) = S;
                const float G = expf(aq[j]);
                S.x = fmaf(G, S.x, dq[j].x);
                S.y = fmaf(G, S.y, dq[j].y);
                S.z = fmaf(G, S.z, dq[j].z);
                S.w = fmaf(G, S.w, dq[j].w);
                if (C > 0 && p.ckpt_slots != nullptr && e % C == 0) {
                    float *slot = p.ckpt_slots[p.ck_base[b] + (e / C - pos0 / C - 1)];
                    if (slot == nullptr || (reinterpret_cast<uintptr_t>(slot) & 15u) != 0) {
                        if (threadIdx.x == 0 && blk == 0 && h == 0)
                            report(p.d_err, slot == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
                    } else {
                        *reinterpret_cast<float4 *>(slot + hs_) = S;
                    }
                }
                if (ld_at < end) {
                    const int64_t e2 = seg_end_of(ld_at);
                    dq[j] = *reinterpret_cast<const float4 *>(p.dS + (int64_t)ld_seg * sstride + hs_);
                    aq[j] = gate_sum(ld_at, e2);
                    ld_at = e2;
                    ++ld_seg;
                }
                at = e;
                ++seg;
            }
        }
    }
    *st = S;
}

}  // namespace

cudaError_t launch_gla_scan(const ScanParams &p, int d, cudaStream_t s)
{
    const unsigned bh = (unsigned)p.batch * (unsigned)p.n_heads;
    if (bh == 0)
        return cudaSuccess;
    if (d == 128)
        return launch_pdl(gla_scan_kernel<128>, dim3(bh * (128 * 128 / (4 * kThreads))),
                          dim3(kThreads), 0, s, p);
    if (d == 64)
        return launch_pdl(gla_scan_kernel<64>, dim3(bh * (64 * 64 / (4 * kThreads))),
                          dim3(kThreads), 0, s, p);
    return cudaErrorNotSupported;
}

}  // namespace hs
