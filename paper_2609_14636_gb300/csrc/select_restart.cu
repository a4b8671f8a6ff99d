// select_restart.cu -- restart choice over stored trajectory records, and
// state initialisation (sm_103a).
//
// One warp per record (Sec. 4.2 steps 1-2, Eq. 6, Algorithm 1).  Lanes take
// 32 turns at a time: a ballot of "not correct" gives the length of the
// leading all-correct run (K_max grows by it, and stops growing at the first
// incorrect turn), and a shuffle reduction over (l_k, k) gives the lowest
// index of the minimum among the run's turns.  All compares are fp32, the
// precision of the stored record.
#include <math.h>

#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace stride {

constexpr int kSelectThreads = 256;

__global__ void __launch_bounds__(kSelectThreads) select_restart_kernel(const SelectParams p) {
  const int lane = threadIdx.x & 31;
  const int64_t w = ((int64_t)blockIdx.x * kSelectThreads + threadIdx.x) >> 5;
  if (w >= p.N) return;
  int nt = __ldg(p.n_turns + w);
  nt = nt < 0 ? 0 : (nt > p.T_max ? p.T_max : nt);
  const float* row = p.turn_mean + w * (int64_t)p.T_max;
  const uint8_t* mrow = p.correct ? p.correct + w * (int64_t)p.T_max : nullptr;
  int K = 0;
  float best_v = 0.f;
  int best_k = 0;
  bool have = false;
  for (int base = 0; base < nt; base += 32) {
    const int k = base + lane;
    const bool in = k < nt;
    const float v = in ? __ldg(row + k) : 0.f;
    const bool ok = in && (mrow == nullptr || __ldg(mrow + k) != 0) && (v > p.alpha);
    const unsigned bad = __ballot_sync(0xffffffffu, !ok);
    const int run = bad ? __ffs(bad) - 1 : 32;
    // argmin over lanes < run, lowest index on ties
    float cv = (lane < run) ? v : INFINITY;
    int ck = (lane < run) ? k : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, cv, o);
      const int ok2 = __shfl_xor_sync(0xffffffffu, ck, o);
      if (ov < cv || (ov == cv && ok2 < ck)) {
        cv = ov;
        ck = ok2;
      }
    }
    if (run > 0 && (!have || cv < best_v)) {
      best_v = cv;
      best_k = ck;
      have = true;
    }
    K += run;
    if (run < 32) break;
  }
  if (lane == 0) {
    p.k_max[w] = K;
    p.k_star[w] = K > 0 ? best_k : 0;
  }
}

// One warp per trajectory: keep the task's first k0 stored turns, append the
// trajectory's turn means, set the record length (Algorithm 1, record step).
__global__ void __launch_bounds__(kSelectThreads) buffer_record_kernel(
    float* buf_mean, int32_t* buf_n_turns, int32_t n_tasks, int32_t T_max, const int32_t* task,
    const int32_t* k0, const stride_turn_stats* ts, const int32_t* traj_turn_off, int32_t n_traj,
    int32_t* dev_status) {
  const int lane = threadIdx.x & 31;
  const int64_t i = ((int64_t)blockIdx.x * kSelectThreads + threadIdx.x) >> 5;
  if (i >= n_traj) return;
  const int32_t x = __ldg(task + i);
  if (x < 0 || x >= n_tasks) {
    if (lane == 0) set_status(dev_status, STRIDE_DEV_BAD_LAYOUT);
    return;
  }
  const int32_t stored = __ldg(buf_n_turns + x);
  int32_t keep = k0 ? __ldg(k0 + i) : 0;
  keep = keep < 0 ? 0 : (keep > stored ? stored : keep);
  const int32_t a = __ldg(traj_turn_off + i), b = __ldg(traj_turn_off + i + 1);
  const int32_t n_new = b > a ? b - a : 0;
  const int32_t len = keep + n_new < T_max ? keep + n_new : (keep < T_max ? T_max : keep);
  float* row = buf_mean + (int64_t)x * T_max;
  for (int32_t j = keep + lane; j < len; j += 32) row[j] = ts[a + (j - keep)].mean_t;
  if (lane == 0) buf_n_turns[x] = len;
}

__global__ void state_init_kernel(stride_scan_state* s, int32_t n) {
  // a programmatic dependent (the small-window and decode kernels) may be
  // scheduled now; each of those waits for this grid before its first read
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int32_t i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  stride_scan_state z;
  z.cum = 0.0;
  z.turn_sum_t = 0.0;
  z.turn_sum_d = 0.0;
  z.turn_sum_l = 0.0;
  z.loss = 0.0;
  z.rows_seen = 0;
  z.loss_tokens = 0;
  z.stop_row = -1;
  z.stop_turn = -1;
  z.turn_tokens = 0;
  z.turn_idx = 0;
  z.stopped = 0;
  s[i] = z;
}

cudaError_t launch_select_restart(const SelectParams& p, cudaStream_t stream) {
  const int64_t warps_per_block = kSelectThreads / 32;
  const unsigned grid = (unsigned)((p.N + warps_per_block - 1) / warps_per_block);
  select_restart_kernel<<<grid, kSelectThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_buffer_record(float* buf_mean, int32_t* buf_n_turns, int32_t n_tasks, int32_t T_max,
                                 const int32_t* task, const int32_t* k0, const stride_turn_stats* ts,
                                 const int32_t* traj_turn_off, int32_t n_traj, int32_t* dev_status,
                                 cudaStream_t stream) {
  const int64_t warps_per_block = kSelectThreads / 32;
  const unsigned grid = (unsigned)((n_traj + warps_per_block - 1) / warps_per_block);
  buffer_record_kernel<<<grid, kSelectThreads, 0, stream>>>(buf_mean, buf_n_turns, n_tasks, T_max, task, k0,
                                                            ts, traj_turn_off, n_traj, dev_status);
  return cudaGetLastError();
}

cudaError_t launch_state_init(stride_scan_state* state, int32_t n, cudaStream_t stream) {
  state_init_kernel<<<(n + 255) / 256, 256, 0, stream>>>(state, n);
  return cudaGetLastError();
}

}  // namespace stride
