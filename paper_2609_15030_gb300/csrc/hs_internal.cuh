// Internal declarations shared by the library's translation units.
#pragma once

#include <atomic>
#include <cstdint>
#include <utility>
#include <cuda_runtime.h>

#include "hs.h"

namespace hs {

// Programmatic dependent launch: every kernel of the library is launched with
// programmatic stream serialization, so the next launch on the stream can be
// scheduled while this one runs.  Each kernel waits for its predecessors to
// complete (and their memory to be visible) before it touches global memory
// (L2 prefetches aside), then releases its own dependents; the tensor-core
// prefill only waits (see pdl_wait).
__device__ __forceinline__ void pdl_wait_and_release()
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// The wait alone, for a kernel whose CTAs hold most of an SM for a long time (the
// tensor-core prefill): it never triggers its dependents, so they launch only once its
// CTAs have exited.  Triggered while those CTAs are resident (even near their end), the
// next kernel's CTAs are placed onto the few SMs with room left, and a chain of short
// kernels that follows (decode steps) keeps that imbalance: measured on 64 decode steps
// after a prefill, 5.2 us per step instead of 2.85 us.
__device__ __forceinline__ void pdl_wait()
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t stream, Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// First detected device-side problem wins; kernels never clear the word.
// Launch a kernel that needs more than 48 KiB of dynamic shared memory.  Its limit is set
// with cudaFuncSetAttribute on the first launch on each device (bit `dev` of `done`) instead
// of on every call; if a launch still fails (the device's context was reset since), the
// error is cleared, the limit set again and the launch retried once.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl_big_smem(void (*kernel)(KArgs...), dim3 grid, dim3 block,
                                       size_t smem, cudaStream_t stream,
                                       std::atomic<uint64_t> &done, Args &&...args)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return e;
    const uint64_t bit = dev >= 0 && dev < 64 ? 1ull << dev : 0;
    if (bit == 0 || (done.load(std::memory_order_acquire) & bit) == 0) {
        e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess)
            return e;
        done.fetch_or(bit, std::memory_order_acq_rel);
        return launch_pdl(kernel, grid, block, smem, stream, std::forward<Args>(args)...);
    }
    e = launch_pdl(kernel, grid, block, smem, stream, args...);
    if (e == cudaSuccess)
        return e;
    (void)cudaGetLastError();
    done.fetch_and(~bit, std::memory_order_acq_rel);
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess)
        return e;
    done.fetch_or(bit, std::memory_order_acq_rel);
    return launch_pdl(kernel, grid, block, smem, stream, std::forward<Args>(args)...);
}

__device__ __forceinline__ void report(int32_t *d_err, int32_t code)
{
    if (d_err != nullptr)
        atomicCAS(d_err, 0, code);
}

// Per-call description of a linear-attention prefill, passed by value to the kernels.
struct GlaParams {
    const uint16_t *q;
    const uint16_t *k;
    const uint16_t *v;
    const float *log_g;
    float *o;
    float *state;
    float *const *ckpt_slots;  // device array or nullptr
    int32_t *d_err;
    int32_t batch;
    int32_t n_heads;
    int32_t ckpt_interval;     // 0: none
    int32_t stall_for_test;    // tensor-core kernel only: one wait that nothing completes (failure-detection tests)
    int32_t no_state_out;      // tensor-core kernel only: the final state is not written
    int64_t pos0[HS_MAX_BATCH];
    int32_t n_tokens[HS_MAX_BATCH];
    int32_t ck_base[HS_MAX_BATCH];  // index of the problem's first slot in ckpt_slots; in the
                                    // restart launch (no checkpoints), of its first segment's
                                    // start state in state
    int32_t row0[HS_MAX_BATCH];     // token row of the problem's first token in q/k/v/log_g/o
};

// launchers (return the launch's cudaError_t)
cudaError_t launch_kv_scatter(const void *const *staging, void *const *cache, int32_t n_layers,
                              const int32_t *bt, int32_t n_pages, int64_t page_bytes,
                              int64_t num_blocks, int32_t *d_err, int sm_count, cudaStream_t s);
cudaError_t launch_kv_gather(const void *const *cache, void *const *staging, int32_t n_layers,
                             const int32_t *bt, int32_t n_pages, int64_t page_bytes,
                             int64_t num_blocks, int32_t *d_err, int sm_count, cudaStream_t s);
cudaError_t launch_kv_slices(bool gather, const void *const *from, void *const *to, int32_t n_layers,
                             const int32_t *bt, int32_t n_pages, int64_t page_bytes, int32_t rows,
                             int64_t col_off, int64_t col_bytes, int64_t num_blocks, int32_t *d_err,
                             int sm_count, cudaStream_t s);
cudaError_t launch_restore_request(const void *const *staging, void *const *cache, int32_t n_layers,
                                   const int32_t *bt, int32_t n_pages, int64_t page_bytes,
                                   int64_t num_blocks, const float *const *src_slots,
                                   float *const *dst_slots, int32_t n_slots, int64_t floats_each,
                                   int32_t *d_err, int sm_count, cudaStream_t s);
cudaError_t launch_slot_copy(const float *const *src, float *const *dst, int32_t n,
                             int64_t floats_each, int32_t *d_err, int sm_count, cudaStream_t s);
// The elementwise state scan between the two tensor-core passes of hs_linattn_prefill_scan:
// per (problem, head), S_{n+1} = g_n * S_n + dS_n over the problem's segments (g_n the
// segment's decay factor per key dim, dS_n the segment's state from the zero state), recording
// each segment's start state, the checkpoints and the final state.
struct ScanParams {
    float *state;             // [batch][n_heads][d][d]: in the state at pos0, out at pos0 + n
    const float *dS;          // [segments][n_heads][d][d]: each segment from the zero state
    float *Sn;                // [segments][n_heads][d][d]: on entry each segment's decay G of
                              // key row d at element (d, 0); on return its start state
    float *const *ckpt_slots; // as GlaParams
    int32_t *d_err;
    int32_t batch;
    int32_t n_heads;
    int32_t ckpt_interval;
    int64_t pos0[HS_MAX_BATCH];
    int32_t n_tokens[HS_MAX_BATCH];
    int32_t row0[HS_MAX_BATCH];
    int32_t ck_base[HS_MAX_BATCH];
    int32_t seg_base[HS_MAX_BATCH];   // index of the problem's first segment in dS / Sn
};
cudaError_t launch_gla_scan(const ScanParams &p, int d, cudaStream_t s);
cudaError_t launch_gla_recurrent(const GlaParams &p, int d, cudaStream_t s);
cudaError_t launch_gla_decode(const GlaParams &p, int d, cudaStream_t s);
cudaError_t launch_gla_chunked_tc(const GlaParams &p, int d, cudaStream_t s);
// every segment from its own start state (see the kernel); ckpt_slots must be nullptr
cudaError_t launch_gla_chunked_tc_restart(const GlaParams &p, int d, cudaStream_t s);
bool gla_chunked_tc_supported(int d);

}  // namespace hs
