/*
 * hs_test.h -- a fault-injection entry point for the failure-detection tests.
 * It is not part of the restore-and-resume path and no product code calls it.
 *
 * hs_test_prefill_stalled takes the arguments of hs_linattn_prefill_from_state
 * (hs.h) and requires shp->kernel == HS_LINATTN_CHUNKED_TC (else
 * HS_ERR_UNSUPPORTED).  Every CTA of the tensor-core kernel first waits on an
 * mbarrier that nothing completes.  That wait is bounded like every wait of the
 * kernel (1 s of the GPU's global timer); when it runs out the CTA takes its
 * abort path: it stores HS_DEVERR_TIMEOUT into d_err (if d_err still holds 0),
 * waits (bounded) for its own copies in flight, frees its tensor memory and
 * returns without writing o, state or any checkpoint slot.  The context stays
 * usable, and later calls on the stream run normally.
 *
 * Argument checks, layouts, ownership and host-side errors are those of
 * hs_linattn_prefill_from_state.
 */
#ifndef HS_TEST_H
#define HS_TEST_H

#include "hs.h"

#ifdef __cplusplus
extern "C" {
#endif

hs_status hs_test_prefill_stalled(const hs_linattn_shape *shp, const uint16_t *q, const uint16_t *k,
                                  const uint16_t *v, const float *log_g, float *o, float *state,
                                  const int64_t *pos0, const int32_t *n_tokens,
                                  int32_t ckpt_interval, float *const *ckpt_slots, int32_t *d_err,
                                  cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif  // HS_TEST_H
