// Launch parameters of the segment-state kernel (gla_dstate.cu), the first pass of the
// segment-parallel prefill: every 64-token segment's state from the zero state.
#pragma once

#include "hs_internal.cuh"

namespace hs {

struct DStateParams {
    const uint16_t *k;        // [rows][n_heads][d] bf16
    const uint16_t *v;        // [rows][n_heads][d] bf16
    const float *log_g;       // [rows][n_heads][d]
    float *dS;                // [segments][n_heads][d][d]: written
    float *Sn;                // [segments][n_heads][d][d]: the segment's decay of key row d,
                              // 2^{sum of its log2-gates}, written at element (d, 0), where the
                              // scan reads it before writing the start state there
    int32_t *d_err;
    int32_t batch;
    int32_t n_heads;
    int32_t n_units;          // segments x n_heads
    int64_t pos0[HS_MAX_BATCH];
    int32_t n_tokens[HS_MAX_BATCH];
    int32_t row0[HS_MAX_BATCH];
    int32_t seg_base[HS_MAX_BATCH];   // index of the problem's first segment
};

// grid: CTAs (at most two per SM are resident; each walks units blockIdx.x, + grid, ...)
cudaError_t launch_gla_dstate(const DStateParams &p, int d, int grid, cudaStream_t s);

}  // namespace hs
