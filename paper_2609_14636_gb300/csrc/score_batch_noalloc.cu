// score_batch_noalloc.cu -- stride_score_batch without a caller workspace.
//
// Some callers cannot allocate device memory for the scan workspace that
// stride_score_batch needs: a process whose device memory is reserved up
// front by another allocator (a framework's caching allocator, a serving
// engine's cache pool) so that one more cudaMalloc fails or fragments it; a
// caller that cannot afford the implicit device synchronisation of
// cudaMalloc/cudaFree on its path; or a foreign-language caller that only has
// the inputs and outputs it was handed.  For them this file keeps the scratch
// in a file-scope __device__ array of fixed size, which the library holds on
// every device that loads it until the process exits, and launches the same
// scoring kernel with pointers into it.
//
// Limits and rules:
// - at most STRIDE_NOALLOC_MAX_ROWS rows per call (a larger window returns
//   STRIDE_ERR_TOO_LARGE before anything is launched);
// - every call, on every stream, shares the one array per device, and the
//   array keeps the previous call's contents: the call clears the part that
//   must start at zero (tickets and flags) before its scan reads it (with
//   cudaMemsetAsync, or from the small-window kernel).  Two calls that
//   overlap in time on the GPU race on the array and give wrong results:
//   order them on one stream (or with events);
// - the array's device address comes from cudaGetSymbolAddress (the first
//   call on a device may load the library's module onto it, so make that
//   first call before any stream capture).  It is looked up again on every
//   call made outside a stream capture, so a device reset between calls
//   (which may move the array) is followed; a call made while its stream is
//   capturing uses the address the last such call found.
// Nothing here calls cudaMalloc, cudaFree or any allocating routine.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <mutex>

#include "stride.h"
#include "stride_internal.h"

namespace {

constexpr size_t up256(size_t x) { return (x + 255) & ~size_t(255); }

// Same layout as stride_score_batch's workspace for STRIDE_NOALLOC_MAX_ROWS
// rows: 256-byte header, one uint32 flag per 128-byte line, two 32-byte scan
// slots and two float log-probs per row (13.11 MB for 65,536 rows).
constexpr size_t kNoAllocBytes =
    256 + up256(sizeof(uint32_t) * (size_t)stride::kFlagStride * (size_t)STRIDE_NOALLOC_MAX_ROWS) +
    2 * up256(sizeof(stride::ScanSlot) * (size_t)STRIDE_NOALLOC_MAX_ROWS) +
    2 * up256(sizeof(float) * (size_t)STRIDE_NOALLOC_MAX_ROWS);

// The scratch.  In host code `g_noalloc_scratch` is only a handle for the
// runtime: its device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

constexpr int kMaxDevices = 64;
void* g_scratch_addr[kMaxDevices] = {};
std::mutex g_setup_mutex;

// Device address of the scratch on the current device (with that device
// current): looked up afresh unless `stream` is capturing, in which case the
// address found by the last lookup on this device is used.
int scratch_for_current_device(cudaStream_t stream, void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return STRIDE_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return STRIDE_ERR_UNSUPPORTED_DEVICE;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(stream, &cap) != cudaSuccess) return STRIDE_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (cap == cudaStreamCaptureStatusNone || g_scratch_addr[dev] == nullptr) {
    if (cap != cudaStreamCaptureStatusNone) return STRIDE_ERR_CUDA;  // no address found before the capture
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || ptr == nullptr)
      return STRIDE_ERR_CUDA;
    g_scratch_addr[dev] = ptr;
  }
  *out = g_scratch_addr[dev];
  return STRIDE_OK;
}

}  // namespace

extern "C" STRIDE_API int stride_score_batch_noalloc(
    const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V, const int32_t* tokens,
    const int64_t* traj_row_off, const int64_t* turn_row_off, const int32_t* traj_turn_off,
    int32_t n_traj, int32_t n_turns, int64_t row_begin, int64_t row_end, int32_t stop_mode,
    const float* lambda, float lambda_all, stride_scan_state* state, const stride_row_outputs* out,
    stride_turn_stats* turn_stats, double* profile, int32_t* dev_status, void* stream) {
  if (row_begin < 0 || row_end < row_begin) return STRIDE_ERR_INVALID_ARG;
  if (row_end - row_begin > (int64_t)STRIDE_NOALLOC_MAX_ROWS) return STRIDE_ERR_TOO_LARGE;
  if (row_end == row_begin)  // the same argument checks as the workspace entry point, nothing launched
    return stride_score_batch(S, T, dtype, ld, V, tokens, traj_row_off, turn_row_off, traj_turn_off,
                              n_traj, n_turns, row_begin, row_end, stop_mode, lambda, lambda_all, state,
                              out, turn_stats, profile, dev_status, nullptr, 0, stream);
  static_assert(kNoAllocBytes % 256 == 0, "scratch size");
  if (stride::batch_workspace_layout(STRIDE_NOALLOC_MAX_ROWS).total > kNoAllocBytes)
    return STRIDE_ERR_CUDA;  // layout and array out of step: a build error, never expected
  void* scratch = nullptr;
  const int sc = scratch_for_current_device((cudaStream_t)stream, &scratch);
  if (sc != STRIDE_OK) return sc;
  // The scoring entry point clears the tickets and flags of the window and
  // launches the kernels with pointers into the scratch.
  return stride_score_batch(S, T, dtype, ld, V, tokens, traj_row_off, turn_row_off, traj_turn_off,
                            n_traj, n_turns, row_begin, row_end, stop_mode, lambda, lambda_all,
                            state, out, turn_stats, profile, dev_status, scratch, kNoAllocBytes,
                            stream);
}
