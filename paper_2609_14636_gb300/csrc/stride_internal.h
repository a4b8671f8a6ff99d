// stride_internal.h -- launch interfaces between the C-ABI layer and the
// kernels.  Not installed; callers use include/stride.h.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "stride.h"

namespace stride {

// One published scan element of the batch kernel's lookback (32 bytes):
// running-sum terms, and the open turn's sums of log pi_T, d and logp_S * d.
struct alignas(32) ScanSlot {
  double c, st, sd, sl;
};

// Row r's scan flag is flags[r * kFlagStride]: one flag per 128-byte line.
// Every row of a window polls and reads its predecessors' flags; packed 32 to
// a line, a few lines took all of that traffic, and GB300 windows of 512-
// 1,024 rows scored 3-12 % faster with the flags spread out.
constexpr int kFlagStride = 32;

// Rows per tile (and threads per CTA) of the tiled scan on log-probs (build
// defines, for sweeps): on its own (stride_scan_logprobs, the sharded path)
// and as the programmatic dependent that completes a small window.  A sweep
// on GB300 (one size for both): the 148,909-row scan took 52.8 / 51.2 / 49.2
// / 49.6 us with tiles of 64 / 128 / 256 / 512 rows, the 512-row tiny step
// 36.6 / 36.7 / 37.4 / 39.0 us: many small tiles finish a small window's
// chain sooner, larger ones run a long scan with fewer lookbacks.  (The
// small window's tiles now run as one cluster, with no chain.)
#ifndef STRIDE_SCAN_TILE_ROWS
#define STRIDE_SCAN_TILE_ROWS 256
#endif
#ifndef STRIDE_SCAN_TILE_ROWS_DEPENDENT
#define STRIDE_SCAN_TILE_ROWS_DEPENDENT 128
#endif
constexpr int kScanTileRows = STRIDE_SCAN_TILE_ROWS;
constexpr int kScanTileRowsDependent = STRIDE_SCAN_TILE_ROWS_DEPENDENT;
static_assert(kScanTileRows % 32 == 0 && kScanTileRows >= 64 && kScanTileRows <= 1024,
              "whole warps, 2 to 32 of them");
static_assert(kScanTileRowsDependent % 32 == 0 && kScanTileRowsDependent >= 64 && kScanTileRowsDependent <= 1024,
              "whole warps, 2 to 32 of them");

struct BatchParams {
  const void* S;
  const void* T;
  const void* const* T_rows;  // per-window-row teacher row pointers (multi-teacher), or NULL
  int64_t ld;
  int32_t V;
  int32_t mode;
  const int32_t* tokens;
  const int64_t* traj_row_off;
  const int64_t* turn_row_off;
  const int32_t* traj_turn_off;
  int32_t n_traj;
  int32_t n_turns;
  int64_t row_begin;
  int64_t row_end;
  int64_t n_rows;
  const float* lambda;
  float lambda_all;
  stride_scan_state* state;
  stride_row_outputs out;
  stride_turn_stats* turn_stats;
  double* profile;  // [STRIDE_PROFILE_BINS * 3] or NULL, added to
  int32_t* dev_status;
  // workspace views
  uint32_t* ticket;
  uint32_t* flags;
  ScanSlot* agg;
  ScanSlot* incl;
  float* ws_logp_s;  // per window row, written by the small-window kernel for the tiled scan
  float* ws_logp_t;
  uint64_t timeout_ns;
};

struct StepParams {
  const void* S;
  const void* T;
  int64_t ld;
  int32_t V;
  int32_t mode;
  const int32_t* tokens;
  const uint8_t* turn_end;
  const int32_t* rollout_idx;  // compacted rows: row b is rollout rollout_idx[b]; NULL = row b is rollout b
  int32_t B;                   // rows of this step
  int32_t n_state;             // rollouts in state / lambda (compacted form: bound of rollout_idx)
  const float* lambda;
  float lambda_all;
  stride_scan_state* state;
  stride_row_outputs out;
  uint8_t* stopped_now;
  stride_turn_stats* turn_out;
  int32_t* dev_status;
};

struct SelectParams {
  const float* turn_mean;
  const int32_t* n_turns;
  const uint8_t* correct;
  float alpha;
  int32_t N;
  int32_t T_max;
  int32_t* k_star;
  int32_t* k_max;
};

// Workspace layout of stride_score_batch (all offsets 256-byte aligned).
struct BatchWorkspaceLayout {
  size_t ticket_off, flags_off, agg_off, incl_off, logp_s_off, logp_t_off, clear_bytes, total;
};
BatchWorkspaceLayout batch_workspace_layout(int64_t n_rows);

// Teacher row address of window row `tile`: the aligned T buffer, or the
// multi-teacher row table.
template <typename LT>
__device__ __forceinline__ const LT* teacher_row(const BatchParams& p, int64_t tile) {
  return p.T_rows ? reinterpret_cast<const LT*>(p.T_rows[tile])
                  : reinterpret_cast<const LT*>(p.T) + tile * p.ld;
}

constexpr int kMaxTeacherDomains = 8;
struct TeacherTable {
  const void* base[kMaxTeacherDomains];
  int64_t rows[kMaxTeacherDomains];
  int32_t n_domains;
  int64_t ld_bytes;
};
cudaError_t launch_teacher_rows(const BatchParams& p, const TeacherTable& tt, const uint8_t* traj_domain,
                                const int64_t* traj_T_row0, const void** rows_out, cudaStream_t stream);

// Multiprocessor count of the current device, looked up once per device
// (thread-safe); 0 with the CUDA error in *err if it cannot be queried.
int current_device_sms(int* dev_out, cudaError_t* err);

// Launchers return a cudaError_t from the launch.
// Clears what must start at zero in the workspace (clear_bytes from its
// start: the clearing kernel, or on the small-window path the split kernel
// itself) and launches the batch scoring kernels.
cudaError_t launch_score_batch(const BatchParams& p, int dtype, bool vec, size_t clear_bytes, cudaStream_t stream);
cudaError_t launch_score_batch_stream(const BatchParams& p, int dtype, cudaStream_t stream);
// Zeroes `bytes` (a multiple of 16) at ws as a programmatic dependent of the
// previous kernel on the stream (it waits for that kernel first).
cudaError_t launch_clear_workspace(void* ws, size_t bytes, int sms, cudaStream_t stream);
cudaError_t launch_score_step(const StepParams& p, int dtype, bool vec, cudaStream_t stream);
// Diagnostic overrides of the automatic kernel choices (process-wide; 0 on
// success, -1 for a value out of range).
int set_step_shape_override(int threads, int C);  // 0 = automatic; 128 or 512 threads, 1..16 CTAs per row
int set_batch_kernel_override(const char* name);  // NULL / "" / "auto" = automatic
cudaError_t launch_select_restart(const SelectParams& p, cudaStream_t stream);
cudaError_t launch_state_init(stride_scan_state* state, int32_t n, cudaStream_t stream);
cudaError_t launch_partial_lse(const void* S, const void* T, int dtype, bool vec, int64_t ld,
                               int32_t V_shard, int64_t col0, const int32_t* tokens, int64_t rows,
                               float* partials, int32_t* dev_status, cudaStream_t stream);
cudaError_t launch_combine_partials(const float* parts, int32_t n_shards, int64_t rows, float* logp_s,
                                    float* logp_t, float* lse_s, float* lse_t, int32_t* dev_status,
                                    cudaStream_t stream);
cudaError_t launch_scan_logprobs(const BatchParams& p, const float* logp_s, const float* logp_t,
                                 cudaStream_t stream, bool dependent = false);
cudaError_t launch_buffer_record(float* buf_mean, int32_t* buf_n_turns, int32_t n_tasks, int32_t T_max,
                                 const int32_t* task, const int32_t* k0, const stride_turn_stats* ts,
                                 const int32_t* traj_turn_off, int32_t n_traj, int32_t* dev_status,
                                 cudaStream_t stream);

}  // namespace stride
