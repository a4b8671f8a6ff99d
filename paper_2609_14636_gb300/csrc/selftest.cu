// selftest.cu -- two hooks that are not part of the scoring path:
// * the library's real bounded waits run on a flag (or an mbarrier) that
//   nothing sets, so that the timeout path can be checked on a GPU: the wait
//   runs out after timeout_ns, the kernel records STRIDE_DEV_TIMEOUT and
//   returns.  No trap, no fault, no endless loop;
// * a read-only stream over one or two buffers, the floor the scoring
//   kernels are measured against.
#include <cuda_runtime.h>

#include "mbarrier.cuh"
#include "stride_device.cuh"
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

// Read-only streaming: CTA c reads its contiguous 1/grid of the 16-byte
// vectors of a (and of b), with the scoring kernels' non-allocating 16-byte
// loads, 8 in flight per thread per buffer, and folds them with XOR so the
// loads stay live; one word per CTA is written to sink.
__global__ void stream_read_kernel(const uint4* __restrict__ a, const uint4* __restrict__ b, uint64_t nv,
                                   uint32_t* __restrict__ sink) {
  const uint64_t g = gridDim.x;
  const uint64_t lo = nv * blockIdx.x / g, hi = nv * (blockIdx.x + 1) / g;
  constexpr int U = 8;
  uint32_t x = 0;
  uint64_t i = lo + threadIdx.x;
  const uint64_t step = blockDim.x;
  for (; i + (U - 1) * step < hi; i += U * step) {
    uint4 va[U], vb[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      va[u] = ld_stream(a + i + u * step);
      if (b) vb[u] = ld_stream(b + i + u * step);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      x ^= va[u].x ^ va[u].y ^ va[u].z ^ va[u].w;
      if (b) x ^= vb[u].x ^ vb[u].y ^ vb[u].z ^ vb[u].w;
    }
  }
  for (; i < hi; i += step) {
    const uint4 va = ld_stream(a + i);
    x ^= va.x ^ va.y ^ va.z ^ va.w;
    if (b) {
      const uint4 vb = ld_stream(b + i);
      x ^= vb.x ^ vb.y ^ vb.z ^ vb.w;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x ^= __shfl_xor_sync(0xffffffffu, x, o);
  __shared__ uint32_t s_x[32];
  if ((threadIdx.x & 31) == 0) s_x[threadIdx.x >> 5] = x;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t t = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t ^= s_x[w];
    sink[blockIdx.x] = t;
  }
}

}  // namespace stride

extern "C" STRIDE_API int stride_selftest_stream_read(const void* a, const void* b, uint64_t bytes_each,
                                                      int32_t grid, int32_t threads, uint32_t* sink,
                                                      void* stream) {
  if (!a || !sink || bytes_each == 0 || (bytes_each & 15u) != 0) return STRIDE_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(a) & 15u) != 0 || (reinterpret_cast<uintptr_t>(b) & 15u) != 0)
    return STRIDE_ERR_INVALID_ARG;
  if (grid < 1 || threads < 32 || threads > 1024 || (threads & 31) != 0) return STRIDE_ERR_INVALID_ARG;
  if (bytes_each / 16 > UINT64_MAX / (uint64_t)grid) return STRIDE_ERR_INVALID_ARG;  // slice bounds in 64 bits
  stride::stream_read_kernel<<<(unsigned)grid, (unsigned)threads, 0, (cudaStream_t)stream>>>(
      reinterpret_cast<const uint4*>(a), reinterpret_cast<const uint4*>(b), bytes_each / 16, sink);
  return cudaGetLastError() == cudaSuccess ? STRIDE_OK : STRIDE_ERR_CUDA;
}

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
