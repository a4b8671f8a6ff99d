/*
 * stride_selftest.h -- self-test and measurement hooks of libstride.so.  The
 * paper has no counterpart to either:
 * - the bounded-wait self-test exists so that the library's failure path (a
 *   wait that runs out sets STRIDE_DEV_TIMEOUT and the kernel returns,
 *   leaving the context usable) can be exercised on a GPU without faulting
 *   or hanging it;
 * - the read-only stream gives the floor the scoring kernels are measured
 *   against: how fast this GPU reads the same bytes, in the same 16-byte
 *   loads, with no arithmetic at all.
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

/* Reads bytes_each bytes of device buffer a, and of b when b is not NULL,
 * once, with the scoring kernels' 16-byte non-allocating loads: `grid` CTAs
 * of `threads` threads (a multiple of 32, at most 1,024), CTA c reading the
 * c-th contiguous 1/grid of each buffer.  Nothing is computed beyond an XOR
 * of the loaded words, written as one word per CTA to sink (device uint32
 * [grid]) so the loads cannot be dropped.  a and b must be 16-byte aligned
 * and bytes_each a multiple of 16.  Asynchronous on stream; returns STRIDE_OK
 * after the launch, or an argument / CUDA error code. */
STRIDE_API int stride_selftest_stream_read(const void* a, const void* b, uint64_t bytes_each, int32_t grid,
                                           int32_t threads, uint32_t* sink, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* STRIDE_SELFTEST_H_ */
