/*
 * stride_selftest.h -- a self-test hook for the bounded device-side waits of
 * libstride.so.  The paper has no counterpart: this exists so that the
 * library's failure path (a wait that runs out sets STRIDE_DEV_TIMEOUT and
 * the kernel returns, leaving the context usable) can be exercised on a GPU
 * without faulting or hanging it.
 */
#ifndef STRIDE_SELFTEST_H_
#define STRIDE_SELFTEST_H_

#include "stride.h"

#ifdef __cplusplus
extern "C" {
#endif

#define STRIDE_SELFTEST_LOOKBACK 0 /* the batch kernels' lookback wait on a predecessor flag */
#define STRIDE_SELFTEST_MBARRIER 1 /* the persistent kernel's bounded mbarrier wait */

/* Runs one of the library's real bounded waits on a flag (or an mbarrier)
 * that nothing ever sets, with the wait limit `timeout_ns` (the scoring
 * kernels use 2 s; pass e.g. 50 ms).  When the wait runs out the kernel ORs
 * STRIDE_DEV_TIMEOUT into *dev_status (device int32, required) and returns.
 * workspace: device, >= stride_score_batch_workspace_size(2) bytes,
 * 256-byte aligned (cleared by the call).  Asynchronous on stream; returns
 * STRIDE_OK after the launch, or an argument / CUDA error code. */
STRIDE_API int stride_selftest_bounded_wait(int32_t which, uint64_t timeout_ns, int32_t* dev_status,
                                            void* workspace, size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* STRIDE_SELFTEST_H_ */
