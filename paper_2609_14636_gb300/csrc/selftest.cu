// selftest.cu -- runs the library's real bounded waits on a flag (or an
// mbarrier) that nothing sets, so that the timeout path can be checked on a
// GPU: the wait runs out after timeout_ns, the kernel records
// STRIDE_DEV_TIMEOUT and returns.  No trap, no fault, no endless loop.
#include <cuda_runtime.h>

#include "mbarrier.cuh"
#include "row_scan.cuh"
#include "stride.h"
#include "stride_internal.h"
#include "stride_selftest.h"

namespace stride {

// One warp looks back from tile 1; tile 0's flag stays 0 (never published).
__global__ void selftest_lookback_kernel(const BatchParams p) {
  const int lane = threadIdx.x & 31;
  bool timed_out = false;
  (void)lookback(p, 1, lane, timed_out);
  if (lane == 0 && timed_out) set_status(p.dev_status, STRIDE_DEV_TIMEOUT);
}

// One warp waits on an mbarrier that expects one arrival and never gets it.
__global__ void selftest_mbarrier_kernel(int32_t* dev_status, uint64_t timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int32_t abort;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const bool ok = mbar_wait(&bar, 0u, timeout_ns, &abort);
  if (threadIdx.x == 0 && !ok) set_status(dev_status, STRIDE_DEV_TIMEOUT);
}

}  // namespace stride

extern "C" STRIDE_API int stride_selftest_bounded_wait(int32_t which, uint64_t timeout_ns,
                                                       int32_t* dev_status, void* workspace,
                                                       size_t workspace_bytes, void* stream) {
  if (!dev_status || timeout_ns == 0 || timeout_ns > 10000000000ull) return STRIDE_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  if (which == STRIDE_SELFTEST_LOOKBACK) {
    const stride::BatchWorkspaceLayout L = stride::batch_workspace_layout(2);
    if (!workspace || workspace_bytes < L.total || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
      return STRIDE_ERR_WORKSPACE;
    if (cudaMemsetAsync(workspace, 0, L.total, st) != cudaSuccess) return STRIDE_ERR_CUDA;
    char* ws = static_cast<char*>(workspace);
    stride::BatchParams p = {};
    p.n_rows = 2;
    p.dev_status = dev_status;
    p.ticket = reinterpret_cast<uint32_t*>(ws + L.ticket_off);
    p.flags = reinterpret_cast<uint32_t*>(ws + L.flags_off);
    p.agg = reinterpret_cast<stride::ScanSlot*>(ws + L.agg_off);
    p.incl = reinterpret_cast<stride::ScanSlot*>(ws + L.incl_off);
    p.timeout_ns = timeout_ns;
    stride::selftest_lookback_kernel<<<1, 32, 0, st>>>(p);
  } else if (which == STRIDE_SELFTEST_MBARRIER) {
    stride::selftest_mbarrier_kernel<<<1, 32, 0, st>>>(dev_status, timeout_ns);
  } else {
    return STRIDE_ERR_INVALID_ARG;
  }
  return cudaGetLastError() == cudaSuccess ? STRIDE_OK : STRIDE_ERR_CUDA;
}
