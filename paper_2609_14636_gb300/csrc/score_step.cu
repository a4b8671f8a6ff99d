// score_step.cu -- one decode step over B active rollouts (sm_103a).
//
// Algorithm 1's inner loop scores one generated token per rollout per step.
// A step holds only B rows (B = 256 in the decode workload), too few for one
// CTA per row to fill 152 SMs, so each row is split over the kStepCluster
// CTAs of one thread-block cluster: every CTA streams a slice of the
// vocabulary of both the student and the teacher row into online
// log-sum-exp pairs, the pairs meet in rank 0 through distributed shared
// memory, and rank 0 forms the token's log-probs and advances the rollout's
// carried state (open-turn sums, turn close with Eq. 4, stop test of Eq. 5 or
// Sec. 5.5).  Rollouts whose state says stopped exit before reading a byte.
// No workspace, no atomics, no spin-waits: the cluster barrier is hardware.
//
// Launch shape (chosen by a sweep of CTA size x cluster size x unroll on
// GB300, B = 256, V = 151,936): 128-thread CTAs, 4 per cluster, at most 64
// registers so 8 fit per SM, so a 256-rollout step is one wave of 1,024
// CTAs (27.5 us per step; 8-CTA clusters of 256 threads took 44.7 us, 128-
// thread CTAs in 8-CTA clusters 35.9 us).  Steps are launched with programmatic
// dependent launch: a step's CTAs may be scheduled while the previous
// kernel on the stream finishes, and each waits (griddepcontrol.wait) for
// that kernel's completion before its first global read, so the caller's
// inputs and the carried state are always complete when read.
#include <cooperative_groups.h>
#include <math.h>

#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace cg = cooperative_groups;

namespace stride {

#ifndef STRIDE_STEP_THREADS
#define STRIDE_STEP_THREADS 128
#endif
#ifndef STRIDE_STEP_CLUSTER
#define STRIDE_STEP_CLUSTER 4
#endif
#ifndef STRIDE_STEP_UNROLL
#define STRIDE_STEP_UNROLL 4
#endif
#ifndef STRIDE_STEP_MIN_BLOCKS
#define STRIDE_STEP_MIN_BLOCKS 8
#endif

constexpr int kStepThreads = STRIDE_STEP_THREADS;
constexpr int kStepWarps = kStepThreads / 32;
constexpr int kStepCluster = STRIDE_STEP_CLUSTER;
constexpr int kStepUnroll = STRIDE_STEP_UNROLL;

template <typename LT, bool VEC>
__global__ void __cluster_dims__(kStepCluster, 1, 1) __launch_bounds__(kStepThreads, STRIDE_STEP_MIN_BLOCKS)
    score_step_kernel(const StepParams p) {
  __shared__ float s_red[4][kStepWarps];
  __shared__ float s_part[4];
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int b = (int)(blockIdx.x / kStepCluster);
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  stride_scan_state* sp = p.state + b;
  const float nan = __int_as_float(0x7fc00000);
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  // Every CTA of the cluster reads the flag before the first cluster barrier
  // and rank 0 writes it only after that barrier, so all agree.
  if (__ldcg(&sp->stopped)) {
    if (rank == 0 && tid == 0) {
      const stride_row_outputs& o = p.out;
      if (o.logp_s) o.logp_s[b] = nan;
      if (o.logp_t) o.logp_t[b] = nan;
      if (o.opd) o.opd[b] = nan;
      if (o.lse_s) o.lse_s[b] = nan;
      if (o.lse_t) o.lse_t[b] = nan;
      if (o.x_s) o.x_s[b] = nan;
      if (o.x_t) o.x_t[b] = nan;
      if (p.stopped_now) p.stopped_now[b] = 0;
      if (p.turn_out) p.turn_out[b] = stride_turn_stats{0.0, 0.0, 0.0, 0.0, 0.f, 0};
    }
    return;
  }

  const LT* srow = reinterpret_cast<const LT*>(p.S) + (int64_t)b * p.ld;
  const LT* trow = reinterpret_cast<const LT*>(p.T) + (int64_t)b * p.ld;

  // The token id is loaded now and its logits gathered after the stream: a
  // gather before it held rank 0 back by about 0.7 us on average (GB300
  // timeline), and the cluster waits for its slowest rank.
  int32_t y = 0;
  float xs = nan, xt = nan;
  if (rank == 0 && tid == 0) y = __ldg(p.tokens + b);

  // vocabulary slice of this rank (whole 16-byte vectors on the vector path;
  // the last rank also takes the ragged tail)
  int c0, c1;
  if (VEC) {
    constexpr int P = LogitTraits<LT>::kPerVec;
    const int nv = p.V / P;
    const int per = (nv + kStepCluster - 1) / kStepCluster;
    c0 = min(nv, rank * per) * P;
    c1 = (rank == kStepCluster - 1) ? p.V : min(nv, (rank + 1) * per) * P;
  } else {
    const int per = (p.V + kStepCluster - 1) / kStepCluster;
    c0 = min(p.V, rank * per);
    c1 = min(p.V, (rank + 1) * per);
  }
  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  stream_pair<LT, VEC, kStepUnroll>(srow, trow, c0, c1, tid, kStepThreads, mS, sS, mT, sT);
  if (rank == 0 && tid == 0 && y >= 0 && y < p.V) {
    xs = to_f32(srow[y]);
    xt = to_f32(trow[y]);
  }
  warp_merge2(mS, sS, mT, sT);
  if (lane == 0) {
    s_red[0][warp] = mS;
    s_red[1][warp] = sS;
    s_red[2][warp] = mT;
    s_red[3][warp] = sT;
  }
  __syncthreads();
  if (warp == 0) {
    mS = lane < kStepWarps ? s_red[0][lane] : kMaxStart;
    sS = lane < kStepWarps ? s_red[1][lane] : 0.f;
    mT = lane < kStepWarps ? s_red[2][lane] : kMaxStart;
    sT = lane < kStepWarps ? s_red[3][lane] : 0.f;
    warp_merge2(mS, sS, mT, sT);
    if (lane == 0) {
      s_part[0] = mS;
      s_part[1] = sS;
      s_part[2] = mT;
      s_part[3] = sT;
    }
  }
  cluster.sync();

  if (rank == 0 && warp == 0) {
    mS = kMaxStart;
    sS = 0.f;
    mT = kMaxStart;
    sT = 0.f;
    if (lane < kStepCluster) {
      const float* peer = cluster.map_shared_rank(s_part, lane);
      mS = peer[0];
      sS = peer[1];
      mT = peer[2];
      sT = peer[3];
    }
    warp_merge2(mS, sS, mT, sT);
    if (lane == 0) {
      const float lse_s = lse_finish(mS, sS);
      const float lse_t = lse_finish(mT, sT);
      const float lps = xs - lse_s;
      const float lpt = xt - lse_t;
      const float dd = lps - lpt;
      if (!(y >= 0 && y < p.V)) set_status(p.dev_status, STRIDE_DEV_TOKEN_RANGE);
      const stride_row_outputs& o = p.out;
      if (o.logp_s) o.logp_s[b] = lps;
      if (o.logp_t) o.logp_t[b] = lpt;
      if (o.opd) o.opd[b] = dd;
      if (o.lse_s) o.lse_s[b] = lse_s;
      if (o.lse_t) o.lse_t[b] = lse_t;
      if (o.x_s) o.x_s[b] = xs;
      if (o.x_t) o.x_t[b] = xt;

      // carried state (Algorithm 1 inner loop)
      stride_scan_state st = *sp;
      const float lam = p.lambda ? __ldg(p.lambda + b) : p.lambda_all;
      const double term = (double)lps * (double)dd;  // -log pi_S * r_t (Eq. 2); every scored token is retained
      st.turn_sum_t += (double)lpt;
      st.turn_sum_d += (double)dd;
      st.turn_sum_l += term;
      st.loss += term;
      st.loss_tokens += 1;
      st.turn_tokens += 1;
      const int64_t pos = st.rows_seen;
      st.rows_seen += 1;
      uint8_t fired = 0;
      if (p.mode == STRIDE_STOP_TOKEN_SUM) {
        st.cum += (double)lpt;
        if (st.cum < (double)lam) fired = 1;
      }
      stride_turn_stats ts{0.0, 0.0, 0.0, 0.0, 0.f, 0};
      if (__ldg(p.turn_end + b)) {
        const double mean = st.turn_sum_t / (double)st.turn_tokens;  // Eq. 4
        if (p.mode == STRIDE_STOP_TURN_MEAN) {
          st.cum += mean;  // Eq. 5
          if (st.cum < (double)lam) fired = 1;
        }
        ts.sum_t = st.turn_sum_t;
        ts.sum_d = st.turn_sum_d;
        ts.sum_l = st.turn_sum_l;
        ts.cum = st.cum;
        ts.mean_t = (float)mean;
        ts.n = st.turn_tokens;
        st.turn_idx += 1;
        st.turn_tokens = 0;
        st.turn_sum_t = 0.0;
        st.turn_sum_d = 0.0;
        st.turn_sum_l = 0.0;
      }
      if (fired) {
        st.stopped = 1;
        st.stop_row = pos;
        // the turn the firing token belongs to (closed or still open)
        st.stop_turn = (__ldg(p.turn_end + b)) ? st.turn_idx - 1 : st.turn_idx;
      }
      *sp = st;
      if (p.stopped_now) p.stopped_now[b] = fired;
      if (p.turn_out) p.turn_out[b] = ts;
    }
  }
  cluster.sync();  // peers keep their shared memory until rank 0 has read it
}

template <typename LT, bool VEC>
static cudaError_t launch_step_pdl(const StepParams& p, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.B * kStepCluster);
  cfg.blockDim = dim3(kStepThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, score_step_kernel<LT, VEC>, p);
}

cudaError_t launch_score_step(const StepParams& p, int dtype, bool vec, cudaStream_t stream) {
  cudaError_t e;
  if (dtype == STRIDE_DTYPE_BF16)
    e = vec ? launch_step_pdl<__nv_bfloat16, true>(p, stream) : launch_step_pdl<__nv_bfloat16, false>(p, stream);
  else
    e = vec ? launch_step_pdl<float, true>(p, stream) : launch_step_pdl<float, false>(p, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace stride
