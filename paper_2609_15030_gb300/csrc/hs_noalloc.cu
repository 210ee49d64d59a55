// hs_linattn_prefill_scan_noalloc: the segment-parallel prefill with its workspace in a
// fixed array of this library, for callers that cannot allocate device memory when they
// run it.
//
// A serving engine typically reserves nearly all free HBM for its KV-cache block pool at
// start-up and gives out memory only from its own pools afterwards, and a request resumed
// inside its scheduler loop must not pay for cudaMalloc or cudaFree (which can synchronise
// the whole device and stall the other streams).  Such a caller has no place to take the
// segment-parallel prefill's workspace from.  This entry point takes it from the array
// below instead: HS_NOALLOC_SCRATCH_BYTES bytes, one array per device, loaded with this
// library's module for that device.
//
// Set-up: the first call on a device resolves the array's device address with
// cudaGetSymbolAddress (with that device current; with lazy module loading this is also when
// the array comes into existence) and caches it for later calls.  Make that first call before
// any stream capture.  Nothing else here calls the CUDA runtime; the prefill itself is
// hs_linattn_prefill_scan with the array as its workspace.
//
// Every call on a device shares the one array and finds the previous call's contents there.
// None of it has to start at zero: each call writes every word it reads before reading it.
// Calls whose work overlaps on the GPU (on two streams, or on two host threads without
// ordering) overwrite each other's workspace and give wrong results: order them on one
// stream or with events.
#include <atomic>
#include <mutex>

#include "hs_internal.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[HS_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::atomic<void *> g_scratch_addr[kMaxDevices];   // per device, nullptr until resolved
std::mutex g_setup_mutex;

// the array's address on the current device, resolved on the first call there
hs_status scratch_address(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return HS_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices)
        return HS_ERR_UNSUPPORTED;
    void *p = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (p == nullptr) {
        std::lock_guard<std::mutex> lock(g_setup_mutex);
        p = g_scratch_addr[dev].load(std::memory_order_relaxed);
        if (p == nullptr) {
            const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
            if (e != cudaSuccess || p == nullptr)
                return HS_ERR_CUDA;
            g_scratch_addr[dev].store(p, std::memory_order_release);
        }
    }
    *out = p;
    return HS_OK;
}

}  // namespace

hs_status hs_linattn_prefill_scan_noalloc(const hs_linattn_shape *shp, const uint16_t *q,
                                          const uint16_t *k, const uint16_t *v,
                                          const float *log_g, float *o, float *state,
                                          const int64_t *pos0, const int32_t *n_tokens,
                                          int32_t ckpt_interval, float *const *ckpt_slots,
                                          int32_t *d_err, cudaStream_t stream)
{
    // every host-side check first, so that a rejected call touches no CUDA state
    int64_t need = 0;
    hs_status st = hs_linattn_scan_workspace_bytes(shp, pos0, n_tokens, &need);
    if (st != HS_OK)
        return st;
    if (need > (int64_t)HS_NOALLOC_SCRATCH_BYTES)
        return HS_ERR_TOO_LARGE;
    if (ckpt_interval < 0)
        return HS_ERR_INVALID_ARG;
    if (ckpt_interval % HS_CHUNK != 0)
        return HS_ERR_UNSUPPORTED;
    if (need == 0)   // no tokens: hs_linattn_prefill_scan returns without using a workspace
        return hs_linattn_prefill_scan(shp, q, k, v, log_g, o, state, pos0, n_tokens,
                                       ckpt_interval, ckpt_slots, nullptr, 0, d_err, stream);
    const void *args[] = {q, k, v, log_g, o, state};
    for (const void *a : args)
        if (a == nullptr)
            return HS_ERR_INVALID_ARG;
    for (const void *a : args)
        if ((reinterpret_cast<uintptr_t>(a) & 15u) != 0)
            return HS_ERR_MISALIGNED;
    void *ws = nullptr;
    if ((st = scratch_address(&ws)) != HS_OK)
        return st;
    return hs_linattn_prefill_scan(shp, q, k, v, log_g, o, state, pos0, n_tokens, ckpt_interval,
                                   ckpt_slots, ws, (int64_t)HS_NOALLOC_SCRATCH_BYTES, d_err,
                                   stream);
}
