/*
 * stride.h -- C ABI of the STRIDE scoring path (arXiv 2609.14636) on one
 * NVIDIA GB300 (sm_103a).
 *
 * The library computes the per-token teacher/student scoring that STRIDE's
 * adaptive early stopping and prefix buffer act on:
 *
 *   log pi_S(y_t), log pi_T(y_t)   log-softmax over the vocabulary, gathered
 *                                  at the sampled token (Eq. 1, Eq. 4);
 *   d_t = log pi_S - log pi_T      the per-token OPD signal, = -r_t of Eq. 1
 *                                  (the per-token KL estimate of Sec. 3.2);
 *   l_k                            per-turn mean teacher log-prob (Eq. 4);
 *   first crossing                 the first turn K* whose running sum of
 *                                  turn means, over the newly generated turns
 *                                  only, falls below lambda (Eq. 5 with the
 *                                  prefix-buffer offset of Sec. 4.1), or the
 *                                  first token whose running teacher log-prob
 *                                  falls below lambda (Sec. 5.5);
 *   k*, K_max                      the weakest correct turn of Eq. 6 behind
 *                                  the quality gate of Sec. 4.2;
 *   OPD loss                       the token-level loss of Eq. 2 on the
 *                                  retained tokens (Algorithm 1: the tokens
 *                                  kept, including the triggering turn);
 *   within-turn profile            d and log pi_T by relative position within
 *                                  a turn, in deciles (Observation 1).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All array pointers are DEVICE pointers owned by the caller (allocate them
 *   with cudaMalloc, torch, ...).  Struct pointers passed as "host struct" are
 *   read on the host during the call only.  The library allocates no memory;
 *   scratch space is a caller-provided workspace whose size a *_workspace_size
 *   query returns.
 * - Every compute call is asynchronous on the caller's `stream` (a
 *   cudaStream_t passed as void*; NULL = the legacy default stream) and
 *   returns a stride_status after host-side argument checks and the launch.
 *   A non-zero return means nothing was launched (or the launch failed:
 *   STRIDE_ERR_CUDA).
 * - Errors found on the device are OR-ed into the caller's int32 `dev_status`
 *   word (STRIDE_DEV_* bits; nullable), readable after the stream has
 *   synchronised.  Kernels never trap: a bad row gets NaN outputs.
 * - Logit rows are row-major with a row stride `ld` (elements, ld >= V), and
 *   1 <= V <= STRIDE_MAX_VOCAB (for a vocabulary shard, its V_shard).
 *   Rows whose address and stride are 16-byte aligned take the vectorised
 *   path; others take a scalar path with the same results.
 * - Turn and row indices reported per trajectory are 0-based and local to the
 *   trajectory.  The paper's turns are 1-based, so the returned k* equals its
 *   K0 = k* - 1 (Algorithm 1): the number of turns reused as context.
 * - Every compute call is a plain kernel launch or a short chain of them
 *   (the batch paths clear their workspace with a kernel of the chain), so
 *   a sequence of calls can be captured in a CUDA graph.
 * - The library is built for sm_103a only; on another device the calls return
 *   STRIDE_ERR_UNSUPPORTED_DEVICE.  There is no CPU fallback.
 * - The batch calls choose among three kernels with the same results: for
 *   windows of at most 8 rows per SM, a kernel that splits each row over a
 *   thread-block cluster of 1, 2, 4 or 8 CTAs (the window is one wave); a
 *   persistent bulk-copy kernel for 16-byte-aligned rows; and one CTA per
 *   row otherwise.  The decode-step calls split each row over a cluster of
 *   1 to 16 CTAs of 128 or 512 threads, chosen from the step's row count so
 *   that all rows run in one wave.  stride_force_batch_kernel and
 *   stride_force_step_shape (below) fix these choices for tests and
 *   diagnosis.
 */
#ifndef STRIDE_H_
#define STRIDE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define STRIDE_ABI_VERSION 3

#if defined(__GNUC__)
#define STRIDE_API __attribute__((visibility("default")))
#else
#define STRIDE_API
#endif

/* ---- return codes ------------------------------------------------------ */
typedef enum stride_status {
  STRIDE_OK = 0,
  STRIDE_ERR_INVALID_ARG = 1,        /* a pointer, size, mode or layout is invalid */
  STRIDE_ERR_UNSUPPORTED_DTYPE = 2,  /* dtype is not BF16 or F32 */
  STRIDE_ERR_WORKSPACE = 3,          /* workspace missing, too small or misaligned */
  STRIDE_ERR_CUDA = 4,               /* a CUDA runtime call or launch failed */
  STRIDE_ERR_UNSUPPORTED_DEVICE = 5, /* current device is not compute capability 10.3 */
  STRIDE_ERR_TOO_LARGE = 6           /* window larger than STRIDE_NOALLOC_MAX_ROWS (no-allocation entry point) */
} stride_status;

/* ---- device status bits (OR-ed into *dev_status) ----------------------- */
#define STRIDE_DEV_TOKEN_RANGE 0x1 /* a token is outside [0, V): that row is NaN */
#define STRIDE_DEV_BAD_LAYOUT 0x2  /* offsets not monotone, an empty turn, or a row outside its turn */
#define STRIDE_DEV_TIMEOUT 0x4     /* a bounded device-side wait gave up (results of that call are invalid) */

/* ---- enums ---------------------------------------------------------------- */
#define STRIDE_DTYPE_BF16 0 /* logits are bfloat16 */
#define STRIDE_DTYPE_F32 1  /* logits are float32 */

/* The largest vocabulary (logits per row, or per shard row) the scoring
 * calls accept.  The kernels index a row's columns with 32-bit integers;
 * 2^30 keeps every column index plus a CTA's stride below 2^31.  A larger
 * V (or V_shard) returns STRIDE_ERR_INVALID_ARG before any launch. */
#define STRIDE_MAX_VOCAB (1 << 30)

#define STRIDE_STOP_TURN_MEAN 0 /* Eq. 5: running sum of per-turn means l_k, tested at turn ends */
#define STRIDE_STOP_TOKEN_SUM 1 /* Sec. 5.5: running sum of token log-probs, tested at every token */

/* ---- per-trajectory / per-rollout carried state (80 bytes) ---------------
 * Initialise with stride_state_init.  It is both the carry between calls
 * (chunked batch scoring, decode steps) and the per-trajectory result.
 * A trajectory's running sum starts from `cum` at its first row (0 after
 * init), which is how the prefix-buffer offset is expressed: pass only the
 * newly generated turns of a restarted rollout (Sec. 4.1; Algorithm 1).
 * `loss` accumulates the OPD-loss terms logp_S * d (= -log pi_S * r_t, Eq. 2)
 * of the retained tokens: in turn mode every token of the turns up to and
 * including the triggering turn, in token mode every token up to and
 * including the triggering token, all tokens while the rule has not fired. */
typedef struct stride_scan_state {
  double cum;          /* running sum through the last scored token (Eq. 5 LHS or token sum) */
  double turn_sum_t;   /* open turn: sum of log pi_T so far */
  double turn_sum_d;   /* open turn: sum of d so far */
  double turn_sum_l;   /* open turn: sum of logp_S * d so far */
  double loss;         /* OPD loss (Eq. 2) over the retained tokens scored so far */
  int64_t rows_seen;   /* tokens of this trajectory scored so far */
  int64_t loss_tokens; /* retained tokens scored so far */
  int64_t stop_row;    /* token position (trajectory-local) of the first crossing; -1 = none */
  int32_t stop_turn;   /* turn (trajectory-local, 0-based) of the first crossing; -1 = none */
  int32_t turn_tokens; /* tokens in the open turn */
  int32_t turn_idx;    /* index of the open turn (trajectory-local) */
  int32_t stopped;     /* non-zero once the stop rule has fired */
} stride_scan_state;

/* ---- per-turn statistics (40 bytes) --------------------------------------- */
typedef struct stride_turn_stats {
  double sum_t;  /* sum of log pi_T over the turn's tokens */
  double sum_d;  /* sum of d over the turn's tokens (turn mean KL = sum_d / n, Sec. 3.2) */
  double sum_l;  /* sum of logp_S * d over the turn's tokens (the turn's OPD loss, Eq. 2) */
  double cum;    /* running sum after this turn (Eq. 5 LHS; token sum at the turn's end in TOKEN_SUM) */
  float mean_t;  /* l_k = sum_t / n (Eq. 4), rounded to fp32 */
  int32_t n;     /* tokens in the turn (n_k) */
} stride_turn_stats;

/* ---- within-turn position profile ------------------------------------------
 * double [STRIDE_PROFILE_BINS][3]: for each decile j of relative position in
 * a turn (token i of a turn of n tokens is in decile floor(10 i / n)), the sum
 * of d, the sum of log pi_T and the token count (Observation 1).  The
 * scoring call ADDS to it; zero it before the first call. */
#define STRIDE_PROFILE_BINS 10

/* ---- optional per-row outputs (host struct of device pointers) ------------
 * Each pointer is nullable; a non-NULL pointer receives one float per row. */
typedef struct stride_row_outputs {
  float* logp_s; /* log pi_S(y_t) */
  float* logp_t; /* log pi_T(y_t) */
  float* opd;    /* d_t = log pi_S(y_t) - log pi_T(y_t) = -r_t (Eq. 1) */
  float* lse_s;  /* log sum_j exp(S_j) */
  float* lse_t;  /* log sum_j exp(T_j) */
  float* x_s;    /* S[y_t], the gathered student logit (exact) */
  float* x_t;    /* T[y_t], the gathered teacher logit (exact) */
} stride_row_outputs;

/* Initialise n states: zeros, stop_row = -1, stop_turn = -1.
 * state: device [n].  Asynchronous on stream. */
STRIDE_API int stride_state_init(stride_scan_state* state, int32_t n, void* stream);

/* Workspace bytes stride_score_batch needs for a window of `window_rows`
 * rows (0 for an empty window).  The workspace must be 256-byte aligned. */
STRIDE_API size_t stride_score_batch_workspace_size(int64_t window_rows);

/* Score a window of rows of ragged trajectories, with turn offsets.
 * (Eq. 1, Eq. 4, Eq. 5 with the prefix-buffer offset, Sec. 5.5.)
 *
 * Global layout (device arrays, int64 rows): trajectory i owns rows
 * [traj_row_off[i], traj_row_off[i+1]) and turns [traj_turn_off[i],
 * traj_turn_off[i+1]); turn k owns rows [turn_row_off[k], turn_row_off[k+1]).
 * Every turn must hold at least one row (Eq. 4 divides by n_k).
 * traj_row_off[0] <= row_begin <= row_end <= traj_row_off[n_traj].
 *
 * This call scores global rows [row_begin, row_end): S, T point at the logits
 * of row_begin ([row_end-row_begin, ld], dtype STRIDE_DTYPE_*), tokens at its
 * token (int32 [row_end-row_begin]).  Calling with consecutive windows on one
 * stream, with the same `state`, gives the same results as one call over all
 * rows: the state carries each trajectory's running sum and open-turn sums
 * across window edges.
 *
 * stop_mode: STRIDE_STOP_TURN_MEAN or STRIDE_STOP_TOKEN_SUM.  lambda: device
 * float [n_traj] per-trajectory thresholds, or NULL to use lambda_all for
 * every trajectory (the scale of lambda depends on the generation unit and is
 * chosen per domain, Sec. 4.1).  The test is strict: sum < lambda (a NaN
 * entry of the array never fires: nothing stops and every token is
 * retained; a NaN lambda_all is rejected).  The token or turn that triggers
 * is retained (Sec. 4.1), and so is a trajectory's first turn or token
 * whatever its starting sum.  Later turns are still scored; the stop fields
 * keep the first crossing.
 *
 * state: device [n_traj], in/out (see stride_scan_state).
 * out: host struct of optional per-row outputs indexed by (row - row_begin); NULL for none.
 * turn_stats: device [n_turns] or NULL; turn k is written by the call that
 * scores its last row.
 * profile: device double [STRIDE_PROFILE_BINS * 3] or NULL; added to.
 * dev_status: device int32 or NULL.
 * workspace: device, >= stride_score_batch_workspace_size(row_end-row_begin)
 * bytes, 256-byte aligned; it is cleared by the call, holds nothing between
 * calls, and one workspace must not be shared by calls that overlap in time.
 * Returns STRIDE_OK or an error code; launches nothing when row_begin == row_end. */
STRIDE_API int stride_score_batch(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V,
                       const int32_t* tokens, const int64_t* traj_row_off,
                       const int64_t* turn_row_off, const int32_t* traj_turn_off, int32_t n_traj,
                       int32_t n_turns, int64_t row_begin, int64_t row_end, int32_t stop_mode,
                       const float* lambda, float lambda_all, stride_scan_state* state,
                       const stride_row_outputs* out, stride_turn_stats* turn_stats,
                       double* profile, int32_t* dev_status, void* workspace,
                       size_t workspace_bytes, void* stream);

/* stride_score_batch with one teacher per domain, without gathering the
 * teacher rows (Sec. 5.3: in cross-domain multi-teacher OPD each trajectory
 * is scored by the expert teacher of its own domain).
 *
 * The student logits S are as in stride_score_batch (one row per window
 * row).  The teacher logits of domain j live in their own buffer
 * T_domains[j] ([T_domain_rows[j], ld_T] row-major, device; T_domains and
 * T_domain_rows are HOST arrays of n_domains <= 8 entries).  Trajectory i is
 * scored against domain traj_domain[i] (device uint8 [n_traj]); its rows are
 * rows traj_T_row0[i], traj_T_row0[i]+1, ... of that buffer (device int64
 * [n_traj]).  A domain or teacher row out of range sets
 * STRIDE_DEV_BAD_LAYOUT (that row's results are meaningless; nothing faults).
 * The workspace must hold stride_score_batch_workspace_size(rows) plus 8
 * bytes per row (rounded up to 256).  All other arguments and results are
 * those of stride_score_batch. */
STRIDE_API int stride_score_batch_multi_teacher(
    const void* S, const void* const* T_domains, const int64_t* T_domain_rows, int32_t n_domains,
    int64_t ld_T, const uint8_t* traj_domain, const int64_t* traj_T_row0, int32_t dtype, int64_t ld,
    int64_t V, const int32_t* tokens, const int64_t* traj_row_off, const int64_t* turn_row_off,
    const int32_t* traj_turn_off, int32_t n_traj, int32_t n_turns, int64_t row_begin,
    int64_t row_end, int32_t stop_mode, const float* lambda, float lambda_all,
    stride_scan_state* state, const stride_row_outputs* out, stride_turn_stats* turn_stats,
    double* profile, int32_t* dev_status, void* workspace, size_t workspace_bytes, void* stream);

/* ---- vocabulary-sharded logits and given log-probs -------------------------
 * With tensor parallelism a model's logits are split by vocabulary columns
 * across ranks.  Each rank reduces its shard (stride_partial_lse), the ranks
 * exchange the 24-byte partials (all-gather; not done by this library), and
 * stride_combine_partials forms the log-probs; stride_scan_logprobs then
 * runs the rest of the path on them.  The result equals stride_score_batch
 * on the full rows (Eq. 1, Eq. 4 log-softmax; the scan as in
 * stride_score_batch). */

/* Partial log-sum-exp of one vocabulary shard.  S, T: [rows, ld], this
 * shard's V_shard columns (global columns col0 .. col0+V_shard-1); tokens:
 * int32 [rows], global token ids.  partials: float [rows][6] =
 * (m_S, s_S, m_T, s_T, S[y], T[y]) with LSE = m + ln(s) over the shard's
 * columns, and the gathered logits NaN when y is not in this shard. */
STRIDE_API int stride_partial_lse(const void* S, const void* T, int32_t dtype, int64_t ld,
                                  int64_t V_shard, int64_t col0, const int32_t* tokens,
                                  int64_t rows, float* partials, int32_t* dev_status, void* stream);

/* Merges n_shards partials ([n_shards][rows][6], shard-major) into
 * log-probs: LSE over all shards, the token's logit from the one shard that
 * holds it (none or several: STRIDE_DEV_TOKEN_RANGE and NaN).  Outputs
 * float [rows] each, nullable. */
STRIDE_API int stride_combine_partials(const float* partials, int32_t n_shards, int64_t rows,
                                       float* logp_s, float* logp_t, float* lse_s, float* lse_t,
                                       int32_t* dev_status, void* stream);

/* The scan part of stride_score_batch on given per-token log-probs
 * (logp_s, logp_t: float, indexed by row - row_begin): d (opd, nullable),
 * turn statistics, the stop rule, the OPD loss on retained tokens, the
 * profile and the carried state, with the same layout, window, state and
 * workspace rules (workspace: stride_score_batch_workspace_size(rows)). */
STRIDE_API int stride_scan_logprobs(const float* logp_s, const float* logp_t,
                                    const int64_t* traj_row_off, const int64_t* turn_row_off,
                                    const int32_t* traj_turn_off, int32_t n_traj, int32_t n_turns,
                                    int64_t row_begin, int64_t row_end, int32_t stop_mode,
                                    const float* lambda, float lambda_all, stride_scan_state* state,
                                    float* opd, stride_turn_stats* turn_stats, double* profile,
                                    int32_t* dev_status, void* workspace, size_t workspace_bytes,
                                    void* stream);

/* One decode step over B rollouts (Algorithm 1, inner turn loop, one
 * generated token per rollout).
 *
 * S, T: [B, ld] logits of this step's token of each rollout; tokens: int32
 * [B]; turn_end: uint8 [B], non-zero when this token closes the rollout's
 * current turn.  state: device [B], in/out.  A rollout whose state.stopped is
 * set is masked: its logits are not read, its state is not changed, its
 * per-row outputs are NaN.  For an active rollout the token is scored, the
 * open turn accumulates, and:
 *   TOKEN_SUM: cum += log pi_T; stop if cum < lambda;
 *   TURN_MEAN: at a turn end, l = turn_sum_t / turn_tokens (Eq. 4),
 *              cum += l, stop if cum < lambda (Eq. 5).
 * Every scored token is retained, so its logp_S * d is added to state.loss.
 * stopped_now: uint8 [B] or NULL, 1 where the rule fired at this step.
 * turn_out: device [B] or NULL: the stats of the turn closed at this step
 * (n = 0 where none closed).  lambda / lambda_all as for stride_score_batch.
 * The call needs no workspace. */
STRIDE_API int stride_score_step(const void* S, const void* T, int32_t dtype, int64_t ld, int64_t V,
                      const int32_t* tokens, const uint8_t* turn_end, int32_t B,
                      int32_t stop_mode, const float* lambda, float lambda_all,
                      stride_scan_state* state, const stride_row_outputs* out,
                      uint8_t* stopped_now, stride_turn_stats* turn_out, int32_t* dev_status,
                      void* stream);

/* stride_score_step with the live rollouts' rows packed (Algorithm 1, inner
 * turn loop: only rollouts that have not stopped generate a token, so a
 * rollout engine that batches only live sequences hands over one row per
 * live rollout).
 *
 * Row b (0 <= b < n_rows) of S, T ([n_rows, ld]), tokens (int32 [n_rows]),
 * turn_end (uint8 [n_rows]) and of every per-row output (out, stopped_now,
 * turn_out: [n_rows] each, nullable) belongs to rollout rollout_idx[b]
 * (device int32 [n_rows], distinct values in [0, n_rollouts)), whose carried
 * state is state[rollout_idx[b]] (device [n_rollouts], in/out) and whose
 * threshold is lambda[rollout_idx[b]] (device float [n_rollouts]) or
 * lambda_all.  The step rule is that of stride_score_step.  Unlike the
 * masked form, a row's logits are read before its state: a row whose
 * rollout has already stopped is read, not scored (NaN outputs, state
 * unchanged).  An index outside [0, n_rollouts) sets STRIDE_DEV_BAD_LAYOUT
 * and NaN outputs for that row; repeated indices race.  The cluster size
 * grows as n_rows shrinks, so a step of a few live rollouts still spreads
 * its rows over the GPU.  No workspace; n_rows = 0 launches nothing. */
STRIDE_API int stride_score_step_compact(const void* S, const void* T, int32_t dtype, int64_t ld,
                                         int64_t V, const int32_t* tokens, const uint8_t* turn_end,
                                         const int32_t* rollout_idx, int32_t n_rows,
                                         int32_t n_rollouts, int32_t stop_mode, const float* lambda,
                                         float lambda_all, stride_scan_state* state,
                                         const stride_row_outputs* out, uint8_t* stopped_now,
                                         stride_turn_stats* turn_out, int32_t* dev_status,
                                         void* stream);

/* Restart choice over N stored trajectory records (Sec. 4.2 steps 1-2,
 * Eq. 6, Algorithm 1).
 *
 * turn_mean: float [N, T_max] row-major (entry i's per-turn l_k); n_turns:
 * int32 [N] (0 <= n_turns[i] <= T_max); correct: uint8 [N, T_max] or NULL
 * (an external correctness mask ANDed with the gate).
 *   correct_k = (correct == NULL || correct[i,k]) && (turn_mean[i,k] > alpha)
 *   K_max     = length of the longest all-correct run starting at turn 0
 *   k*        = argmin_{0 <= k < K_max} turn_mean[i,k], lowest index on ties
 *   K_max = 0 gives k* = 0 (no reusable prefix).
 * alpha = -INFINITY disables the gate (the paper's math setting; App. A uses
 * alpha = -0.8 for agentic runs).  NaN means are never correct.
 * k_star, k_max: int32 [N] outputs.  k_star is 0-based and equals K0. */
STRIDE_API int stride_select_restart(const float* turn_mean, const int32_t* n_turns, const uint8_t* correct,
                          float alpha, int32_t N, int32_t T_max, int32_t* k_star,
                          int32_t* k_max, void* stream);

/* stride_score_batch for callers that cannot allocate device memory.
 *
 * The paper has no counterpart: this is a deployment variant of
 * stride_score_batch.  Some callers cannot provide the scratch workspace,
 * because the device memory is reserved up front by another allocator (a
 * framework's caching allocator, a serving engine's cache pool) so that one
 * more cudaMalloc fails or fragments it, because their path cannot take the
 * implicit device synchronisation of cudaMalloc/cudaFree, or because they
 * were handed only inputs and outputs.  This entry point takes the same
 * arguments minus the workspace and uses a fixed scratch array that the
 * library holds on every device that loads it (about 13.1 MB) until the
 * process exits.  It allocates nothing.
 *
 * - Windows of more than STRIDE_NOALLOC_MAX_ROWS rows return
 *   STRIDE_ERR_TOO_LARGE; nothing is launched.  Score longer inputs in
 *   windows (the carried state makes that exact).
 * - All calls on a device share the one scratch array, which keeps the last
 *   call's contents; each call clears what must start at zero.  Calls that
 *   overlap in time on the GPU race on it: order them on one stream.
 * - The array's device address is looked up (cudaGetSymbolAddress) on every
 *   call made outside a stream capture, so a device reset between calls is
 *   followed; the first call on a device may load the library's module, so
 *   make it before any stream capture.  A call on a capturing stream uses
 *   the address found by the last call outside a capture (none yet:
 *   STRIDE_ERR_CUDA).
 * - An empty window (row_begin == row_end) gets the argument checks of
 *   stride_score_batch and launches nothing. */
#define STRIDE_NOALLOC_MAX_ROWS 65536
STRIDE_API int stride_score_batch_noalloc(const void* S, const void* T, int32_t dtype, int64_t ld,
                                          int64_t V, const int32_t* tokens,
                                          const int64_t* traj_row_off, const int64_t* turn_row_off,
                                          const int32_t* traj_turn_off, int32_t n_traj,
                                          int32_t n_turns, int64_t row_begin, int64_t row_end,
                                          int32_t stop_mode, const float* lambda, float lambda_all,
                                          stride_scan_state* state, const stride_row_outputs* out,
                                          stride_turn_stats* turn_stats, double* profile,
                                          int32_t* dev_status, void* stream);

/* Record trajectories in a device-resident prefix buffer H(x) (Algorithm 1:
 * "record this trajectory's {l_k} to H(x)"; Sec. 4.2 step 3, prefix reuse).
 *
 * buf_mean: float [n_tasks, T_max] and buf_n_turns: int32 [n_tasks], the
 * buffer, updated in place (the same layout stride_select_restart reads, so
 * score -> record -> select runs on the device).  Trajectory i belongs to
 * task task_of_traj[i] (int32 [n_traj]) and reused the first k0_of_traj[i]
 * turns of that task's stored record as context (int32 [n_traj], the k* the
 * previous select returned; NULL = 0 for all); its record becomes those
 * stored turns followed by the l_k (turn_stats[k].mean_t) of its own turns
 * traj_turn_off[i] .. traj_turn_off[i+1]-1, truncated to T_max.  k0 is
 * clamped to the stored length.  Each task may appear at most once per call
 * (otherwise the records of the duplicates race).  A task id outside
 * [0, n_tasks) sets STRIDE_DEV_BAD_LAYOUT and that trajectory is skipped. */
STRIDE_API int stride_buffer_record(float* buf_mean, int32_t* buf_n_turns, int32_t n_tasks,
                                    int32_t T_max, const int32_t* task_of_traj,
                                    const int32_t* k0_of_traj, const stride_turn_stats* turn_stats,
                                    const int32_t* traj_turn_off, int32_t n_traj,
                                    int32_t* dev_status, void* stream);

/* ---- diagnostic overrides (no counterpart in the paper) ----------------------
 * Process-wide settings for tests and diagnosis; they change which kernel
 * runs, never the results beyond floating-point rounding.  Set them between
 * calls, not while other threads launch.
 *
 * stride_force_batch_kernel: NULL, "" or "auto" = automatic choice; "split"
 * (automatic cluster size), "split1", "split2", "split4", "split8" (the
 * small-window kernel with that cluster size), "stream" (the persistent
 * kernel; rows that are not 16-byte aligned still take the per-row kernel)
 * or "rows" (one CTA per row).  Its initial value is the environment variable
 * STRIDE_BATCH_KERNEL (same names), read once, at the first batch call.
 * stride_force_step_shape: the decode-step calls' CTA size (128 or 512
 * threads; 0 = 128 when a cluster size is given) and CTAs per row (1..16;
 * 0 = 1 when a CTA size is given); (0, 0) = automatic.  A shape the device
 * cannot place makes the step calls return STRIDE_ERR_CUDA.
 * Both return STRIDE_ERR_INVALID_ARG for an unknown name, size or shape. */
STRIDE_API int stride_force_batch_kernel(const char* name);
STRIDE_API int stride_force_step_shape(int32_t cta_threads, int32_t cluster_size);

/* Human-readable name of a stride_status code (static string). */
STRIDE_API const char* stride_status_string(int code);

/* STRIDE_ABI_VERSION of the loaded library. */
STRIDE_API int stride_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* STRIDE_H_ */
