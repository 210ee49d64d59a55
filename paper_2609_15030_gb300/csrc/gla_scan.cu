// The state scan of the segment-parallel prefill (hs_linattn_prefill_scan).
//
// Over a problem's tail [pos0, pos0 + n), split into segments at the multiples of 64 of the
// absolute position grid, the recurrence S_t = diag(g_t) S_{t-1} + k_t v_t^T is linear in
// the state: for a segment of tokens [s, e),
//     S_e = diag(G) S_s + dS,   G = prod_{s<=t<e} g_t = 2^{sum_t a_t log2 e},
// where dS is the segment's state when it starts from the zero state.  The first pass of the
// prefill (gla_dstate.cu) computes every segment's dS and G at once; this kernel chains them:
// per (problem, head) and state element, S_{n+1} = G_n S_n + dS_n over the segments in order,
// recording each segment's start state S_n (the last pass computes the outputs from it), the
// checkpoint at every multiple of C and the final state.  Every step is an elementwise fma,
// so a run resumed at a checkpoint on the grid repeats the same operations from there:
// resumed and full computations agree bit for bit.
//
// One CTA per (problem, head, block of 512 state elements); thread i owns four consecutive
// elements (d, e..e+3) of one key row d (a float4), and the D/4 lanes of a row (a warp at
// D = 128, a half-warp at D = 64) are consecutive.  The first pass leaves G_n of row d at
// element (d, 0) of segment n's start-state block: the row's first lane, which owns that
// element, reads it there, passes it to the row's other lanes with a shuffle and then
// overwrites it with the start state.  The chain only streams: each thread copies its float4
// of dS_n (the first lane also G_n) for the next kStages segments into its own slots of
// shared-memory rings with cp.async (one commit group per segment, so that waiting for the
// oldest group never waits for a newer copy), applies the oldest and refills its slots.
#include "hs_internal.cuh"

namespace hs {
namespace {

constexpr int kThreads = 128;        // float4 per thread: 512 state elements per CTA
constexpr int kChunk = 64;           // segments on the 64-token absolute grid
constexpr int kStages = 16;          // segments whose dS and G are in flight

__device__ __forceinline__ void cp_async16(void *smem_dst, const void *gmem_src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                     (uint32_t)__cvta_generic_to_shared(smem_dst)),
                 "l"(gmem_src)
                 : "memory");
}

__device__ __forceinline__ void cp_async4(void *smem_dst, const void *gmem_src)
{
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                     (uint32_t)__cvta_generic_to_shared(smem_dst)),
                 "l"(gmem_src)
                 : "memory");
}

__device__ __forceinline__ void cp_async_commit()
{
    asm volatile("cp.async.commit_group;" ::: "memory");
}

// wait until at most kStages - 1 of this thread's commit groups are pending
__device__ __forceinline__ void cp_async_wait_oldest()
{
    asm volatile("cp.async.wait_group %0;" ::"n"(kStages - 1) : "memory");
}

template <int D>
__global__ void __launch_bounds__(kThreads)
gla_scan_kernel(const __grid_constant__ ScanParams p)
{
    constexpr int BLOCKS = D * D / (4 * kThreads);   // CTAs per (problem, head)
    __shared__ float4 sRing[kStages][kThreads];      // dS of the segments in flight
    __shared__ float sGate[kStages][kThreads];       // their G (in a row's first lane)
    constexpr int W = D / 4;                         // lanes per key row
    const int lane = threadIdx.x & 31;
    const bool row_lead = (lane & (W - 1)) == 0;
    const int bh = blockIdx.x / BLOCKS;
    const int blk = blockIdx.x - bh * BLOCKS;
    const int b = bh / p.n_heads;
    const int h = bh - b * p.n_heads;
    const int f = (blk * kThreads + threadIdx.x) * 4;  // first of this thread's 4 elements
    const int64_t pos0 = p.pos0[b];
    const int64_t end = pos0 + p.n_tokens[b];
    const int64_t hs_ = (int64_t)h * D * D + f;        // offset inside one [n_heads][D][D] state
    const int64_t sstride = (int64_t)p.n_heads * D * D;
    const int C = p.ckpt_interval;
    pdl_wait_and_release();

    float4 *st = reinterpret_cast<float4 *>(p.state + (int64_t)b * sstride + hs_);
    float4 S = *st;
    auto seg_end_of = [&](int64_t at) -> int64_t { return min(end, (at / kChunk + 1) * kChunk); };
    // the rings: one commit group per segment (empty past the last), kStages in flight
    int64_t ld_at = pos0;             // start of the next segment to copy
    int32_t ld_seg = p.seg_base[b];
    auto refill = [&](int slot) {
        if (ld_at < end) {
            const int64_t o = (int64_t)ld_seg * sstride + hs_;
            cp_async16(&sRing[slot][threadIdx.x], p.dS + o);
            if (row_lead)
                cp_async4(&sGate[slot][threadIdx.x], p.Sn + o);
            ld_at = seg_end_of(ld_at);
            ++ld_seg;
        }
        cp_async_commit();
    };
    for (int j = 0; j < kStages; ++j)
        refill(j);
    int64_t at = pos0;
    int32_t seg = p.seg_base[b];
    // the next checkpoint position on the grid and its slot pointer, read one checkpoint
    // ahead (only for positions within the call: the pointer array ends there)
    int64_t next_ck = (C > 0 && p.ckpt_slots != nullptr) ? (pos0 / C + 1) * C : INT64_MAX;
    int32_t ck = p.ck_base[b];
    float *cs_next = next_ck <= end ? p.ckpt_slots[ck] : nullptr;
    int slot = 0;
    while (at < end) {
        const int64_t e = seg_end_of(at);
        cp_async_wait_oldest();
        const float4 dq = sRing[slot][threadIdx.x];
        const float G = __shfl_sync(0xffffffffu, row_lead ? sGate[slot][threadIdx.x] : 0.f,
                                    lane & ~(W - 1));
        // the start state replaces the gate the first pass left in the row's first float4
        *reinterpret_cast<float4 *>(p.Sn + (int64_t)seg * sstride + hs_) = S;
        S.x = fmaf(G, S.x, dq.x);
        S.y = fmaf(G, S.y, dq.y);
        S.z = fmaf(G, S.z, dq.z);
        S.w = fmaf(G, S.w, dq.w);
        if (e == next_ck) {
            float *cs = cs_next;
            next_ck += C;
            if (next_ck <= end)
                cs_next = p.ckpt_slots[++ck];
            if (cs == nullptr || (reinterpret_cast<uintptr_t>(cs) & 15u) != 0) {
                if (threadIdx.x == 0 && blk == 0 && h == 0)
                    report(p.d_err, cs == nullptr ? HS_DEVERR_NULL : HS_DEVERR_MISALIGNED);
            } else {
                *reinterpret_cast<float4 *>(cs + hs_) = S;
            }
        }
        refill(slot);     // after the slot is consumed: its next copies cannot overtake the reads
        slot = slot + 1 == kStages ? 0 : slot + 1;
        at = e;
        ++seg;
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
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
