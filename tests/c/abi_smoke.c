/* A C99 caller of libstride.so: only include/stride.h and the CUDA runtime.
 * (Also three decode steps on the same rows, and the vocabulary limit.)
 *
 * Scores 9 rows of uniform fp32 logits (student = teacher = 0 over V = 1000)
 * in two trajectories (turns of 3 + 2 rows, and 4 rows) under the token-sum
 * rule with lambda = -20, then makes one restart choice.  Every expected
 * value is closed form: log pi(y) = -ln V for uniform logits; the running
 * sum after t+1 tokens is -(t+1) ln V, first below -20 at the third token
 * (trajectory-local row 2, turn 0); d = 0, so the loss is 0 over the 3
 * retained tokens; the turn means are -ln V.  Prints "abi_smoke ok" and
 * exits 0 on success. */
#include <cuda_runtime.h>
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include "stride.h"

#define CHECK_CUDA(x)                                                             \
  do {                                                                            \
    cudaError_t e_ = (x);                                                         \
    if (e_ != cudaSuccess) {                                                      \
      fprintf(stderr, "%s: %s\n", #x, cudaGetErrorString(e_));                    \
      return 2;                                                                   \
    }                                                                             \
  } while (0)
#define EXPECT(c)                                                                 \
  do {                                                                            \
    if (!(c)) {                                                                   \
      fprintf(stderr, "line %d: expected %s\n", __LINE__, #c);                    \
      return 1;                                                                   \
    }                                                                             \
  } while (0)

int main(void) {
  enum { V = 1000, R = 9, NTRAJ = 2, NTURN = 3 };
  const int64_t traj_row_off[NTRAJ + 1] = {0, 5, 9};
  const int64_t turn_row_off[NTURN + 1] = {0, 3, 5, 9};
  const int32_t traj_turn_off[NTRAJ + 1] = {0, 2, 3};
  int32_t tokens[R];
  for (int r = 0; r < R; ++r) tokens[r] = (r * 97) % V;

  float *dS, *dT, *dlp_s, *dlp_t, *dopd;
  int32_t *dtok, *dturn_off32, *dstatus;
  int64_t *dtraj, *dturn;
  stride_scan_state* dstate;
  stride_turn_stats* dts;
  CHECK_CUDA(cudaMalloc((void**)&dS, sizeof(float) * R * V));
  CHECK_CUDA(cudaMalloc((void**)&dT, sizeof(float) * R * V));
  CHECK_CUDA(cudaMemset(dS, 0, sizeof(float) * R * V));
  CHECK_CUDA(cudaMemset(dT, 0, sizeof(float) * R * V));
  CHECK_CUDA(cudaMalloc((void**)&dtok, sizeof tokens));
  CHECK_CUDA(cudaMalloc((void**)&dtraj, sizeof traj_row_off));
  CHECK_CUDA(cudaMalloc((void**)&dturn, sizeof turn_row_off));
  CHECK_CUDA(cudaMalloc((void**)&dturn_off32, sizeof traj_turn_off));
  CHECK_CUDA(cudaMemcpy(dtok, tokens, sizeof tokens, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(dtraj, traj_row_off, sizeof traj_row_off, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(dturn, turn_row_off, sizeof turn_row_off, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(dturn_off32, traj_turn_off, sizeof traj_turn_off, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMalloc((void**)&dlp_s, sizeof(float) * R));
  CHECK_CUDA(cudaMalloc((void**)&dlp_t, sizeof(float) * R));
  CHECK_CUDA(cudaMalloc((void**)&dopd, sizeof(float) * R));
  CHECK_CUDA(cudaMalloc((void**)&dstate, sizeof(stride_scan_state) * NTRAJ));
  CHECK_CUDA(cudaMalloc((void**)&dts, sizeof(stride_turn_stats) * NTURN));
  CHECK_CUDA(cudaMalloc((void**)&dstatus, sizeof(int32_t)));
  CHECK_CUDA(cudaMemset(dstatus, 0, sizeof(int32_t)));
  const size_t ws_bytes = stride_score_batch_workspace_size(R);
  void* dws = NULL;
  CHECK_CUDA(cudaMalloc(&dws, ws_bytes));

  EXPECT(stride_abi_version() == STRIDE_ABI_VERSION);
  EXPECT(stride_state_init(dstate, NTRAJ, NULL) == STRIDE_OK);
  stride_row_outputs out;
  memset(&out, 0, sizeof out);
  out.logp_s = dlp_s;
  out.logp_t = dlp_t;
  out.opd = dopd;
  /* an argument error is refused synchronously and launches nothing */
  EXPECT(stride_score_batch(dS, dT, STRIDE_DTYPE_F32, V, 0, dtok, dtraj, dturn, dturn_off32, NTRAJ, NTURN, 0, R,
                            STRIDE_STOP_TOKEN_SUM, NULL, -20.f, dstate, &out, dts, NULL, dstatus, dws, ws_bytes,
                            NULL) == STRIDE_ERR_INVALID_ARG);
  EXPECT(stride_score_batch(dS, dT, STRIDE_DTYPE_F32, V, V, dtok, dtraj, dturn, dturn_off32, NTRAJ, NTURN, 0, R,
                            STRIDE_STOP_TOKEN_SUM, NULL, -20.f, dstate, &out, dts, NULL, dstatus, dws, ws_bytes,
                            NULL) == STRIDE_OK);
  CHECK_CUDA(cudaDeviceSynchronize());

  float lp_s[R], lp_t[R], opd[R];
  stride_scan_state st[NTRAJ];
  stride_turn_stats ts[NTURN];
  int32_t status = -1;
  CHECK_CUDA(cudaMemcpy(lp_s, dlp_s, sizeof lp_s, cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(lp_t, dlp_t, sizeof lp_t, cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(opd, dopd, sizeof opd, cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(st, dstate, sizeof st, cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(ts, dts, sizeof ts, cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(&status, dstatus, sizeof status, cudaMemcpyDeviceToHost));
  EXPECT(status == 0);
  const double lnv = log((double)V);
  for (int r = 0; r < R; ++r) {
    EXPECT(fabs(lp_s[r] + lnv) <= 2e-3 && fabs(lp_t[r] + lnv) <= 2e-3);
    EXPECT(fabs(opd[r]) <= 2e-3);
  }
  for (int i = 0; i < NTRAJ; ++i) {
    EXPECT(st[i].stopped && st[i].stop_row == 2 && st[i].stop_turn == 0);
    EXPECT(st[i].loss_tokens == 3 && fabs(st[i].loss) <= 1e-9);
    EXPECT(st[i].rows_seen == traj_row_off[i + 1] - traj_row_off[i]);
    EXPECT(fabs(st[i].cum + lnv * (double)st[i].rows_seen) <= 1e-5 * lnv * (double)st[i].rows_seen);
  }
  const int n_expect[NTURN] = {3, 2, 4};
  for (int k = 0; k < NTURN; ++k) {
    EXPECT(ts[k].n == n_expect[k]);
    EXPECT(fabs(ts[k].mean_t + lnv) <= 2e-3);
  }

  /* restart choice: l = (-1, -3, -0.5, -9), mask (1, 1, 0, 1), no gate:
   * the correct prefix is turns 0-1 (K_max = 2), the weakest of them turn 1 */
  const float means[4] = {-1.f, -3.f, -0.5f, -9.f};
  const unsigned char mask[4] = {1, 1, 0, 1};
  const int32_t nt = 4;
  float* dmeans;
  unsigned char* dmask;
  int32_t *dnt, *dks, *dkm;
  CHECK_CUDA(cudaMalloc((void**)&dmeans, sizeof means));
  CHECK_CUDA(cudaMalloc((void**)&dmask, sizeof mask));
  CHECK_CUDA(cudaMalloc((void**)&dnt, sizeof nt));
  CHECK_CUDA(cudaMalloc((void**)&dks, sizeof(int32_t)));
  CHECK_CUDA(cudaMalloc((void**)&dkm, sizeof(int32_t)));
  CHECK_CUDA(cudaMemcpy(dmeans, means, sizeof means, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(dmask, mask, sizeof mask, cudaMemcpyHostToDevice));
  CHECK_CUDA(cudaMemcpy(dnt, &nt, sizeof nt, cudaMemcpyHostToDevice));
  EXPECT(stride_select_restart(dmeans, dnt, dmask, -INFINITY, 1, 4, dks, dkm, NULL) == STRIDE_OK);
  int32_t ks = -1, km = -1;
  CHECK_CUDA(cudaMemcpy(&ks, dks, sizeof ks, cudaMemcpyDeviceToHost));
  CHECK_CUDA(cudaMemcpy(&km, dkm, sizeof km, cudaMemcpyDeviceToHost));
  EXPECT(ks == 1 && km == 2);

  /* three decode steps over rows 0-1 as two rollouts (token-sum rule,
   * lambda = -20): each step adds -ln V, so the third (-20.72) stops both,
   * and every scored token is retained */
  enum { B = 2 };
  stride_scan_state* dst2;
  unsigned char *dte, *dsn;
  CHECK_CUDA(cudaMalloc((void**)&dst2, sizeof(stride_scan_state) * B));
  CHECK_CUDA(cudaMalloc((void**)&dte, B));
  CHECK_CUDA(cudaMalloc((void**)&dsn, B));
  CHECK_CUDA(cudaMemset(dte, 0, B));
  EXPECT(stride_state_init(dst2, B, NULL) == STRIDE_OK);
  unsigned char sn[B];
  for (int s = 0; s < 3; ++s) {
    EXPECT(stride_score_step(dS, dT, STRIDE_DTYPE_F32, V, V, dtok, dte, B, STRIDE_STOP_TOKEN_SUM, NULL, -20.f,
                             dst2, &out, dsn, NULL, dstatus, NULL) == STRIDE_OK);
    CHECK_CUDA(cudaMemcpy(sn, dsn, sizeof sn, cudaMemcpyDeviceToHost));
    for (int b = 0; b < B; ++b) EXPECT(sn[b] == (s == 2));
  }
  stride_scan_state st2[B];
  CHECK_CUDA(cudaMemcpy(st2, dst2, sizeof st2, cudaMemcpyDeviceToHost));
  for (int b = 0; b < B; ++b) {
    EXPECT(st2[b].stopped && st2[b].stop_row == 2 && st2[b].rows_seen == 3 && st2[b].loss_tokens == 3);
    EXPECT(fabs(st2[b].cum + 3.0 * lnv) <= 1e-5 * 3.0 * lnv);
  }

  /* the vocabulary limit is checked on the host: one column more is refused */
  EXPECT(stride_score_batch(dS, dT, STRIDE_DTYPE_F32, (int64_t)STRIDE_MAX_VOCAB + 1, (int64_t)STRIDE_MAX_VOCAB + 1,
                            dtok, dtraj, dturn, dturn_off32, NTRAJ, NTURN, 0, R, STRIDE_STOP_TOKEN_SUM, NULL, -20.f,
                            dstate, &out, dts, NULL, dstatus, dws, ws_bytes, NULL) == STRIDE_ERR_INVALID_ARG);
  printf("abi_smoke ok\n");
  return 0;
}
