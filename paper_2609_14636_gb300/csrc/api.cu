// api.cu -- the C ABI of include/stride.h: host-side argument checks, the
// device check, workspace carving and kernel launches.  No allocation, no
// synchronisation, no CPU fallback.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include <atomic>

#include "stride.h"
#include "stride_internal.h"

namespace {

constexpr int kMaxDevices = 64;
std::atomic<int> g_device_ok[kMaxDevices];  // 0 unknown, 1 sm_103, 2 other

int check_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return STRIDE_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return STRIDE_ERR_UNSUPPORTED_DEVICE;
  int s = g_device_ok[dev].load(std::memory_order_relaxed);
  if (s == 0) {
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
      return STRIDE_ERR_CUDA;
    s = (major == 10 && minor == 3) ? 1 : 2;
    g_device_ok[dev].store(s, std::memory_order_relaxed);
  }
  return s == 1 ? STRIDE_OK : STRIDE_ERR_UNSUPPORTED_DEVICE;
}

size_t dtype_bytes(int32_t dtype) {
  return dtype == STRIDE_DTYPE_BF16 ? 2 : (dtype == STRIDE_DTYPE_F32 ? 4 : 0);
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Checks shared by the two scoring calls.
int check_logits(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V) {
  if (dtype_bytes(dtype) == 0) return STRIDE_ERR_UNSUPPORTED_DTYPE;
  if (!S || !T) return STRIDE_ERR_INVALID_ARG;
  if (V < 1 || V > STRIDE_MAX_VOCAB || ld < V) return STRIDE_ERR_INVALID_ARG;
  return STRIDE_OK;
}

bool vector_ok(const void* S, const void* T, int32_t dtype, int64_t ld) {
  return aligned16(S) && aligned16(T) && ((ld * (int64_t)dtype_bytes(dtype)) % 16) == 0;
}

stride_row_outputs row_outputs(const stride_row_outputs* out) {
  stride_row_outputs o = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
  if (out) o = *out;
  return o;
}

}  // namespace

extern "C" {

const char* stride_status_string(int code) {
  switch (code) {
    case STRIDE_OK: return "STRIDE_OK";
    case STRIDE_ERR_INVALID_ARG: return "STRIDE_ERR_INVALID_ARG: invalid pointer, size, mode or layout";
    case STRIDE_ERR_UNSUPPORTED_DTYPE: return "STRIDE_ERR_UNSUPPORTED_DTYPE: dtype must be BF16 or F32";
    case STRIDE_ERR_WORKSPACE: return "STRIDE_ERR_WORKSPACE: workspace missing, too small or not 256-byte aligned";
    case STRIDE_ERR_CUDA: return "STRIDE_ERR_CUDA: a CUDA runtime call or kernel launch failed";
    case STRIDE_ERR_UNSUPPORTED_DEVICE: return "STRIDE_ERR_UNSUPPORTED_DEVICE: the current device is not sm_103 (GB300)";
    case STRIDE_ERR_TOO_LARGE: return "STRIDE_ERR_TOO_LARGE: window exceeds STRIDE_NOALLOC_MAX_ROWS rows of the built-in scratch";
    default: return "unknown stride status";
  }
}

int stride_abi_version(void) { return STRIDE_ABI_VERSION; }

int stride_state_init(stride_scan_state* state, int32_t n, void* stream) {
  if (n < 0 || (n > 0 && !state)) return STRIDE_ERR_INVALID_ARG;
  if (n == 0) return STRIDE_OK;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  return stride::launch_state_init(state, n, (cudaStream_t)stream) == cudaSuccess ? STRIDE_OK
                                                                                 : STRIDE_ERR_CUDA;
}

size_t stride_score_batch_workspace_size(int64_t window_rows) {
  if (window_rows <= 0) return 0;
  return stride::batch_workspace_layout(window_rows).total;
}

}  // extern "C"

namespace {

// Checks and fills the parameters shared by the batch entry points; T may
// be NULL when a teacher row table replaces it.
int prepare_batch(stride::BatchParams& p, stride::BatchWorkspaceLayout& L, const void* S,
                  const void* T, int32_t dtype, int64_t ld, int64_t V, const int32_t* tokens,
                  const int64_t* traj_row_off, const int64_t* turn_row_off,
                  const int32_t* traj_turn_off, int32_t n_traj, int32_t n_turns, int64_t row_begin,
                  int64_t row_end, int32_t stop_mode, const float* lambda, float lambda_all,
                  stride_scan_state* state, const stride_row_outputs* out,
                  stride_turn_stats* turn_stats, double* profile, int32_t* dev_status,
                  void* workspace, size_t workspace_bytes, size_t extra_ws_bytes) {
  const int lc = check_logits(S, T ? T : S, dtype, ld, V);
  if (lc != STRIDE_OK) return lc;
  if (row_begin < 0 || row_end < row_begin || row_end - row_begin > INT32_MAX)
    return STRIDE_ERR_INVALID_ARG;
  if (stop_mode != STRIDE_STOP_TURN_MEAN && stop_mode != STRIDE_STOP_TOKEN_SUM)
    return STRIDE_ERR_INVALID_ARG;
  if (n_traj < 1 || n_turns < 0 || !traj_row_off || !turn_row_off || !traj_turn_off || !state)
    return STRIDE_ERR_INVALID_ARG;
  if (!lambda && isnan(lambda_all)) return STRIDE_ERR_INVALID_ARG;
  const int64_t n_rows = row_end - row_begin;
  if (n_rows == 0) return STRIDE_OK;
  if (!tokens) return STRIDE_ERR_INVALID_ARG;
  L = stride::batch_workspace_layout(n_rows);
  if (!workspace || workspace_bytes < L.total + extra_ws_bytes ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return STRIDE_ERR_WORKSPACE;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  char* ws = static_cast<char*>(workspace);
  p = stride::BatchParams{};
  p.S = S;
  p.T = T;
  p.T_rows = nullptr;
  p.ld = ld;
  p.V = (int32_t)V;
  p.mode = stop_mode;
  p.tokens = tokens;
  p.traj_row_off = traj_row_off;
  p.turn_row_off = turn_row_off;
  p.traj_turn_off = traj_turn_off;
  p.n_traj = n_traj;
  p.n_turns = n_turns;
  p.row_begin = row_begin;
  p.row_end = row_end;
  p.n_rows = n_rows;
  p.lambda = lambda;
  p.lambda_all = lambda_all;
  p.state = state;
  p.out = row_outputs(out);
  p.turn_stats = turn_stats;
  p.profile = profile;
  p.dev_status = dev_status;
  p.ticket = reinterpret_cast<uint32_t*>(ws + L.ticket_off);
  p.flags = reinterpret_cast<uint32_t*>(ws + L.flags_off);
  p.agg = reinterpret_cast<stride::ScanSlot*>(ws + L.agg_off);
  p.incl = reinterpret_cast<stride::ScanSlot*>(ws + L.incl_off);
  p.ws_logp_s = reinterpret_cast<float*>(ws + L.logp_s_off);
  p.ws_logp_t = reinterpret_cast<float*>(ws + L.logp_t_off);
  p.timeout_ns = 2000000000ull;  // 2 s bound on any single device-side wait
  return STRIDE_OK;
}

}  // namespace

extern "C" {

int stride_score_batch(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V,
                       const int32_t* tokens, const int64_t* traj_row_off,
                       const int64_t* turn_row_off, const int32_t* traj_turn_off, int32_t n_traj,
                       int32_t n_turns, int64_t row_begin, int64_t row_end, int32_t stop_mode,
                       const float* lambda, float lambda_all, stride_scan_state* state,
                       const stride_row_outputs* out, stride_turn_stats* turn_stats,
                       double* profile, int32_t* dev_status, void* workspace,
                       size_t workspace_bytes, void* stream) {
  if (!T) return STRIDE_ERR_INVALID_ARG;
  stride::BatchParams p;
  stride::BatchWorkspaceLayout L;
  const int rc = prepare_batch(p, L, S, T, dtype, ld, V, tokens, traj_row_off, turn_row_off,
                               traj_turn_off, n_traj, n_turns, row_begin, row_end, stop_mode, lambda,
                               lambda_all, state, out, turn_stats, profile, dev_status, workspace,
                               workspace_bytes, 0);
  if (rc != STRIDE_OK || row_end == row_begin) return rc;
  cudaStream_t st = (cudaStream_t)stream;
  const bool vec = vector_ok(S, T, dtype, ld);
  return stride::launch_score_batch(p, dtype, vec, L.clear_bytes, st) == cudaSuccess ? STRIDE_OK
                                                                                     : STRIDE_ERR_CUDA;
}

int stride_score_batch_multi_teacher(const void* S, const void* const* T_domains,
                                     const int64_t* T_domain_rows, int32_t n_domains, int64_t ld_T,
                                     const uint8_t* traj_domain, const int64_t* traj_T_row0,
                                     int32_t dtype, int64_t ld, int64_t V, const int32_t* tokens,
                                     const int64_t* traj_row_off, const int64_t* turn_row_off,
                                     const int32_t* traj_turn_off, int32_t n_traj, int32_t n_turns,
                                     int64_t row_begin, int64_t row_end, int32_t stop_mode,
                                     const float* lambda, float lambda_all, stride_scan_state* state,
                                     const stride_row_outputs* out, stride_turn_stats* turn_stats,
                                     double* profile, int32_t* dev_status, void* workspace,
                                     size_t workspace_bytes, void* stream) {
  if (!T_domains || !T_domain_rows || n_domains < 1 || n_domains > stride::kMaxTeacherDomains ||
      !traj_domain || !traj_T_row0 || ld_T < V)
    return STRIDE_ERR_INVALID_ARG;
  stride::TeacherTable tt = {};
  bool aligned = true;
  for (int i = 0; i < n_domains; ++i) {
    if (!T_domains[i] || T_domain_rows[i] < 0) return STRIDE_ERR_INVALID_ARG;
    tt.base[i] = T_domains[i];
    tt.rows[i] = T_domain_rows[i];
    aligned = aligned && aligned16(T_domains[i]);
  }
  tt.n_domains = n_domains;
  tt.ld_bytes = ld_T * (int64_t)dtype_bytes(dtype);
  const int64_t n_rows = row_end > row_begin ? row_end - row_begin : 0;
  const size_t table_bytes = ((size_t)n_rows * sizeof(void*) + 255) & ~size_t(255);
  stride::BatchParams p;
  stride::BatchWorkspaceLayout L;
  const int rc = prepare_batch(p, L, S, nullptr, dtype, ld, V, tokens, traj_row_off, turn_row_off,
                               traj_turn_off, n_traj, n_turns, row_begin, row_end, stop_mode, lambda,
                               lambda_all, state, out, turn_stats, profile, dev_status, workspace,
                               workspace_bytes, table_bytes);
  if (rc != STRIDE_OK || n_rows == 0) return rc;
  const void** rows = reinterpret_cast<const void**>(static_cast<char*>(workspace) + L.total);
  cudaStream_t st = (cudaStream_t)stream;
  if (stride::launch_teacher_rows(p, tt, traj_domain, traj_T_row0, rows, st) != cudaSuccess)
    return STRIDE_ERR_CUDA;
  p.T_rows = rows;
  const bool vec = aligned && aligned16(S) && ((ld * (int64_t)dtype_bytes(dtype)) % 16) == 0 &&
                   (tt.ld_bytes % 16) == 0;
  return stride::launch_score_batch(p, dtype, vec, L.clear_bytes, st) == cudaSuccess ? STRIDE_OK
                                                                                     : STRIDE_ERR_CUDA;
}

}  // extern "C"

namespace {

// Checks and launch shared by the two decode-step entry points.
int score_step_common(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V,
                      const int32_t* tokens, const uint8_t* turn_end, const int32_t* rollout_idx,
                      int32_t rows, int32_t n_state, int32_t stop_mode, const float* lambda,
                      float lambda_all, stride_scan_state* state, const stride_row_outputs* out,
                      uint8_t* stopped_now, stride_turn_stats* turn_out, int32_t* dev_status,
                      void* stream) {
  const int lc = check_logits(S, T, dtype, ld, V);
  if (lc != STRIDE_OK) return lc;
  if (rows < 0 || rows > (INT32_MAX / 16) || n_state < 0) return STRIDE_ERR_INVALID_ARG;
  if (stop_mode != STRIDE_STOP_TURN_MEAN && stop_mode != STRIDE_STOP_TOKEN_SUM)
    return STRIDE_ERR_INVALID_ARG;
  if (!lambda && isnan(lambda_all)) return STRIDE_ERR_INVALID_ARG;
  if (rows == 0) return STRIDE_OK;
  if (!tokens || !turn_end || !state || n_state < 1) return STRIDE_ERR_INVALID_ARG;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  stride::StepParams p;
  p.S = S;
  p.T = T;
  p.ld = ld;
  p.V = (int32_t)V;
  p.mode = stop_mode;
  p.tokens = tokens;
  p.turn_end = turn_end;
  p.rollout_idx = rollout_idx;
  p.B = rows;
  p.n_state = n_state;
  p.lambda = lambda;
  p.lambda_all = lambda_all;
  p.state = state;
  p.out = row_outputs(out);
  p.stopped_now = stopped_now;
  p.turn_out = turn_out;
  p.dev_status = dev_status;
  const bool vec = vector_ok(S, T, dtype, ld);
  return stride::launch_score_step(p, dtype, vec, (cudaStream_t)stream) == cudaSuccess
             ? STRIDE_OK
             : STRIDE_ERR_CUDA;
}

}  // namespace

extern "C" {

int stride_score_step(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V,
                      const int32_t* tokens, const uint8_t* turn_end, int32_t B,
                      int32_t stop_mode, const float* lambda, float lambda_all,
                      stride_scan_state* state, const stride_row_outputs* out,
                      uint8_t* stopped_now, stride_turn_stats* turn_out, int32_t* dev_status,
                      void* stream) {
  return score_step_common(S, T, dtype, ld, V, tokens, turn_end, nullptr, B, B, stop_mode, lambda,
                           lambda_all, state, out, stopped_now, turn_out, dev_status, stream);
}

int stride_score_step_compact(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V,
                              const int32_t* tokens, const uint8_t* turn_end,
                              const int32_t* rollout_idx, int32_t n_rows, int32_t n_rollouts,
                              int32_t stop_mode, const float* lambda, float lambda_all,
                              stride_scan_state* state, const stride_row_outputs* out,
                              uint8_t* stopped_now, stride_turn_stats* turn_out,
                              int32_t* dev_status, void* stream) {
  if (n_rows > 0 && !rollout_idx) return STRIDE_ERR_INVALID_ARG;
  return score_step_common(S, T, dtype, ld, V, tokens, turn_end, rollout_idx, n_rows, n_rollouts,
                           stop_mode, lambda, lambda_all, state, out, stopped_now, turn_out,
                           dev_status, stream);
}

int stride_force_batch_kernel(const char* name) {
  return stride::set_batch_kernel_override(name) == 0 ? STRIDE_OK : STRIDE_ERR_INVALID_ARG;
}

int stride_force_step_shape(int32_t cta_threads, int32_t cluster_size) {
  return stride::set_step_shape_override(cta_threads, cluster_size) == 0 ? STRIDE_OK : STRIDE_ERR_INVALID_ARG;
}

int stride_select_restart(const float* turn_mean, const int32_t* n_turns, const uint8_t* correct,
                          float alpha, int32_t N, int32_t T_max, int32_t* k_star,
                          int32_t* k_max, void* stream) {
  if (N < 0 || T_max < 0 || isnan(alpha)) return STRIDE_ERR_INVALID_ARG;
  if (N == 0) return STRIDE_OK;
  if (!n_turns || !k_star || !k_max || (T_max > 0 && !turn_mean)) return STRIDE_ERR_INVALID_ARG;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  stride::SelectParams p;
  p.turn_mean = turn_mean;
  p.n_turns = n_turns;
  p.correct = correct;
  p.alpha = alpha;
  p.N = N;
  p.T_max = T_max;
  p.k_star = k_star;
  p.k_max = k_max;
  return stride::launch_select_restart(p, (cudaStream_t)stream) == cudaSuccess ? STRIDE_OK
                                                                              : STRIDE_ERR_CUDA;
}

int stride_partial_lse(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V_shard,
                       int64_t col0, const int32_t* tokens, int64_t rows, float* partials,
                       int32_t* dev_status, void* stream) {
  const int lc = check_logits(S, T, dtype, ld, V_shard);
  if (lc != STRIDE_OK) return lc;
  if (rows < 0 || rows > INT32_MAX || col0 < 0) return STRIDE_ERR_INVALID_ARG;
  if (rows == 0) return STRIDE_OK;
  if (!tokens || !partials) return STRIDE_ERR_INVALID_ARG;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  return stride::launch_partial_lse(S, T, dtype, vector_ok(S, T, dtype, ld), ld, (int32_t)V_shard, col0,
                                    tokens, rows, partials, dev_status, (cudaStream_t)stream) == cudaSuccess
             ? STRIDE_OK
             : STRIDE_ERR_CUDA;
}

int stride_combine_partials(const float* partials, int32_t n_shards, int64_t rows, float* logp_s,
                            float* logp_t, float* lse_s, float* lse_t, int32_t* dev_status,
                            void* stream) {
  if (n_shards < 1 || rows < 0) return STRIDE_ERR_INVALID_ARG;
  if (rows == 0) return STRIDE_OK;
  if (!partials) return STRIDE_ERR_INVALID_ARG;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  return stride::launch_combine_partials(partials, n_shards, rows, logp_s, logp_t, lse_s, lse_t, dev_status,
                                         (cudaStream_t)stream) == cudaSuccess
             ? STRIDE_OK
             : STRIDE_ERR_CUDA;
}

int stride_scan_logprobs(const float* logp_s, const float* logp_t, const int64_t* traj_row_off,
                         const int64_t* turn_row_off, const int32_t* traj_turn_off, int32_t n_traj,
                         int32_t n_turns, int64_t row_begin, int64_t row_end, int32_t stop_mode,
                         const float* lambda, float lambda_all, stride_scan_state* state, float* opd,
                         stride_turn_stats* turn_stats, double* profile, int32_t* dev_status,
                         void* workspace, size_t workspace_bytes, void* stream) {
  if (row_begin < 0 || row_end < row_begin || row_end - row_begin > INT32_MAX)
    return STRIDE_ERR_INVALID_ARG;
  if (stop_mode != STRIDE_STOP_TURN_MEAN && stop_mode != STRIDE_STOP_TOKEN_SUM)
    return STRIDE_ERR_INVALID_ARG;
  if (n_traj < 1 || n_turns < 0 || !traj_row_off || !turn_row_off || !traj_turn_off || !state)
    return STRIDE_ERR_INVALID_ARG;
  if (!lambda && isnan(lambda_all)) return STRIDE_ERR_INVALID_ARG;
  const int64_t n_rows = row_end - row_begin;
  if (n_rows == 0) return STRIDE_OK;
  if (!logp_s || !logp_t) return STRIDE_ERR_INVALID_ARG;
  const stride::BatchWorkspaceLayout L = stride::batch_workspace_layout(n_rows);
  if (!workspace || workspace_bytes < L.total || (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return STRIDE_ERR_WORKSPACE;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  char* ws = static_cast<char*>(workspace);
  stride::BatchParams p = {};
  p.V = 1;
  p.mode = stop_mode;
  p.traj_row_off = traj_row_off;
  p.turn_row_off = turn_row_off;
  p.traj_turn_off = traj_turn_off;
  p.n_traj = n_traj;
  p.n_turns = n_turns;
  p.row_begin = row_begin;
  p.row_end = row_end;
  p.n_rows = n_rows;
  p.lambda = lambda;
  p.lambda_all = lambda_all;
  p.state = state;
  p.out = stride_row_outputs{nullptr, nullptr, opd, nullptr, nullptr, nullptr, nullptr};
  p.turn_stats = turn_stats;
  p.profile = profile;
  p.dev_status = dev_status;
  p.ticket = reinterpret_cast<uint32_t*>(ws + L.ticket_off);
  p.flags = reinterpret_cast<uint32_t*>(ws + L.flags_off);
  p.agg = reinterpret_cast<stride::ScanSlot*>(ws + L.agg_off);
  p.incl = reinterpret_cast<stride::ScanSlot*>(ws + L.incl_off);
  p.timeout_ns = 2000000000ull;
  cudaStream_t st = (cudaStream_t)stream;
  int sm_dev = 0;
  cudaError_t sm_err = cudaSuccess;
  const int sms = stride::current_device_sms(&sm_dev, &sm_err);
  if (sms <= 0) return STRIDE_ERR_CUDA;
  if (stride::launch_clear_workspace(workspace, L.clear_bytes, sms, st) != cudaSuccess) return STRIDE_ERR_CUDA;
  return stride::launch_scan_logprobs(p, logp_s, logp_t, st) == cudaSuccess ? STRIDE_OK : STRIDE_ERR_CUDA;
}

int stride_buffer_record(float* buf_mean, int32_t* buf_n_turns, int32_t n_tasks, int32_t T_max,
                         const int32_t* task_of_traj, const int32_t* k0_of_traj,
                         const stride_turn_stats* turn_stats, const int32_t* traj_turn_off,
                         int32_t n_traj, int32_t* dev_status, void* stream) {
  if (n_traj < 0 || n_tasks < 0 || T_max < 0) return STRIDE_ERR_INVALID_ARG;
  if (n_traj == 0) return STRIDE_OK;
  if (!buf_mean || !buf_n_turns || !task_of_traj || !turn_stats || !traj_turn_off)
    return STRIDE_ERR_INVALID_ARG;
  const int dc = check_device();
  if (dc != STRIDE_OK) return dc;
  return stride::launch_buffer_record(buf_mean, buf_n_turns, n_tasks, T_max, task_of_traj, k0_of_traj,
                                      turn_stats, traj_turn_off, n_traj, dev_status,
                                      (cudaStream_t)stream) == cudaSuccess
             ? STRIDE_OK
             : STRIDE_ERR_CUDA;
}

}  // extern "C"
