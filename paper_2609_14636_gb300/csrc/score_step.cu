// score_step.cu -- one decode step over the live rollouts of a batch (sm_103a).
//
// Algorithm 1's inner loop scores one generated token per rollout per step.
// A step holds only a few hundred rows, too few for one CTA per row to fill
// 152 SMs, so each row is split over the C CTAs of one thread-block cluster:
// every CTA streams a slice of the vocabulary of both the student and the
// teacher row into online log-sum-exp pairs, the pairs meet in rank 0 through
// distributed shared memory, and rank 0 forms the token's log-probs and
// advances the rollout's carried state (open-turn sums, turn close with
// Eq. 4, stop test of Eq. 5 or Sec. 5.5).  No workspace, no atomics, no
// spin-waits: the cluster barrier is hardware.
//
// Two row layouts share the kernel:
//  * masked (stride_score_step): row b is rollout b of the batch; a rollout
//    whose state says stopped exits before reading a byte;
//  * compacted (stride_score_step_compact): the caller packs the live
//    rollouts' rows, row b is rollout rollout_idx[b], whose state and lambda
//    are read through that index.  As rollouts stop the step shrinks, and the
//    cluster size grows with it, so a small step still fills the GPU.
//
// Launch shape.  CTAs of 128 threads (8 per SM) or 512 threads (2 per SM),
// both at most 64 registers per thread; the cluster size C and the CTA size
// come from the step's row count (choose_shape below): a 256-row step keeps
// 4-CTA clusters of 128 threads (1,024 CTAs), a 64-row step takes 12, a
// step of 32 rows or fewer 8-CTA clusters of 512 threads.
//
// Steps are launched with programmatic dependent launch: a step's CTAs may be
// scheduled while the previous kernel on the stream finishes, and each waits
// (griddepcontrol.wait) for that kernel's completion before its first global
// read, so the caller's inputs and the carried state are always complete
// when read.
#include <cooperative_groups.h>
#include <math.h>

#include <atomic>

#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace cg = cooperative_groups;

namespace stride {

#ifndef STRIDE_STEP_UNROLL
#define STRIDE_STEP_UNROLL 4
#endif

constexpr int kStepUnroll = STRIDE_STEP_UNROLL;
constexpr int kStepMaxCluster = 16;
// Two CTA shapes, both at most 64 registers per thread: 128 threads, 8 CTAs
// per SM (the shape of steps with many rows), and 512 threads, 2 per SM (more
// threads per row when a step has too few rows to fill the GPU with
// 128-thread CTAs even in the largest clusters).
constexpr int kStepThreadsSmall = 128;
constexpr int kStepThreadsLarge = 512;
template <int THREADS>
struct StepShape {
  static constexpr int kWarps = THREADS / 32;
  static constexpr int kMinBlocks = 1024 / THREADS;  // 64 registers per thread
};

namespace {

__device__ __forceinline__ void write_row_nan(const StepParams& p, int b) {
  const float nan = __int_as_float(0x7fc00000);
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

}  // namespace

// The 80-byte state as ten 8-byte L2 loads (no L1: the previous step's
// cluster wrote it on another SM), issued together.
__device__ __forceinline__ stride_scan_state load_state(const stride_scan_state* sp) {
  static_assert(sizeof(stride_scan_state) == 80, "state layout");
  union {
    stride_scan_state s;
    unsigned long long w[10];
  } u;
  const unsigned long long* src = reinterpret_cast<const unsigned long long*>(sp);
#pragma unroll
  for (int i = 0; i < 10; ++i) u.w[i] = __ldcg(src + i);
  return u.s;
}

template <typename LT, bool VEC, bool COMPACT, int THREADS>
__global__ void __launch_bounds__(THREADS, StepShape<THREADS>::kMinBlocks) score_step_kernel(const StepParams p) {
  constexpr int kStepWarps = StepShape<THREADS>::kWarps;
  __shared__ float s_red[4][kStepWarps];
  __shared__ float4 s_part[kStepMaxCluster];  // rank 0: every rank's (mS, sS, mT, sT), written by the ranks
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int rank = (int)cluster.block_rank();
  const int b = (int)(blockIdx.x / (unsigned)C);  // row of this step
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  // first barrier phase: arriving here and waiting before the first remote
  // store guarantees every CTA of the cluster has started (its shared memory
  // exists); the wait comes after the stream, so it costs nothing
  cluster_arrive_relaxed();
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (!COMPACT) {
    // A stopped rollout's whole cluster leaves before reading a logit (every
    // CTA reads the flag, which only this step's rank 0 writes, after the
    // cluster's last remote store).
    if (__ldcg(&p.state[b].stopped)) {
      if (rank == 0 && tid == 0) write_row_nan(p, b);
      return;
    }
  }

  const LT* srow = reinterpret_cast<const LT*>(p.S) + (int64_t)b * p.ld;
  const LT* trow = reinterpret_cast<const LT*>(p.T) + (int64_t)b * p.ld;

  // The token id (and, compacted, the rollout id) is loaded now, the token's
  // logits and the rollout's state after the stream, so rank 0 streams as
  // early as the other ranks (a gather before the stream held rank 0 back by
  // about 0.7 us on average, GB300 timeline) and the state's latency hides
  // behind the merge and the cluster barrier.  A compacted row streams
  // without first reading its rollout's state: the caller passes live
  // rollouts, and a row whose state turns out stopped is discarded.
  int32_t y = 0, r = b;
  if (rank == 0 && tid == 0) {
    y = __ldg(p.tokens + b);
    if (COMPACT) r = __ldg(p.rollout_idx + b);
  }

  // vocabulary slice of this rank (whole 16-byte vectors on the vector path;
  // the last rank also takes the ragged tail)
  int c0, c1;
  if (VEC) {
    constexpr int P = LogitTraits<LT>::kPerVec;
    const int nv = p.V / P;
    const int per = (nv + C - 1) / C;
    c0 = min(nv, rank * per) * P;
    c1 = (rank == C - 1) ? p.V : min(nv, (rank + 1) * per) * P;
  } else {
    const int per = (p.V + C - 1) / C;
    c0 = min(p.V, rank * per);
    c1 = min(p.V, (rank + 1) * per);
  }
  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  stream_pair<LT, VEC, kStepUnroll>(srow, trow, c0, c1, tid, THREADS, mS, sS, mT, sT);

  float xs = __int_as_float(0x7fc00000), xt = xs, lam = 0.f;
  bool valid = false, closes = false;
  stride_scan_state st;
  if (rank == 0 && tid == 0) {
    if (y >= 0 && y < p.V) {
      xs = to_f32(srow[y]);
      xt = to_f32(trow[y]);
    }
    valid = !COMPACT || (r >= 0 && r < p.n_state);
    if (valid) {
      st = load_state(p.state + r);
      lam = p.lambda ? __ldg(p.lambda + r) : p.lambda_all;
      closes = __ldg(p.turn_end + b) != 0;
    }
  }
  warp_merge2(mS, sS, mT, sT);
  if (lane == 0) {
    s_red[0][warp] = mS;
    s_red[1][warp] = sS;
    s_red[2][warp] = mT;
    s_red[3][warp] = sT;
  }
  __syncthreads();
  cluster_wait_acquire();  // (first phase) every CTA of the cluster has started
  if (warp == 0) {
    mS = lane < kStepWarps ? s_red[0][lane] : kMaxStart;
    sS = lane < kStepWarps ? s_red[1][lane] : 0.f;
    mT = lane < kStepWarps ? s_red[2][lane] : kMaxStart;
    sT = lane < kStepWarps ? s_red[3][lane] : 0.f;
    warp_merge2(mS, sS, mT, sT);
    if (lane == 0) {
      float4* dst = cluster.map_shared_rank(s_part, 0);
      dst[rank] = make_float4(mS, sS, mT, sT);
    }
  }
  // second phase: the ranks' stores are released to rank 0, the other
  // ranks leave (nobody reads their shared memory)
  cluster_arrive_release();
  if (rank != 0) return;
  cluster_wait_acquire();

  if (warp == 0) {
    mS = kMaxStart;
    sS = 0.f;
    mT = kMaxStart;
    sT = 0.f;
    if (lane < C) {
      const float4 q = s_part[lane];
      mS = q.x;
      sS = q.y;
      mT = q.z;
      sT = q.w;
    }
    warp_merge2(mS, sS, mT, sT);
    if (lane == 0) {
      if (!valid) {
        set_status(p.dev_status, STRIDE_DEV_BAD_LAYOUT);
        write_row_nan(p, b);
      } else if (COMPACT && st.stopped) {
        write_row_nan(p, b);
      } else {
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
        if (closes) {
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
          st.stop_turn = closes ? st.turn_idx - 1 : st.turn_idx;
        }
        p.state[r] = st;
        if (p.stopped_now) p.stopped_now[b] = fired;
        if (p.turn_out) p.turn_out[b] = ts;
      }
    }
  }
}

namespace {

// Forced launch shape (0 = automatic), set by stride_force_step_shape.
std::atomic<int> g_force_threads{0};
std::atomic<int> g_force_cluster{0};

constexpr int kMaxDev = 64;

// Launch shape of a step with `rows` rows.  Sweeps on GB300 (B = 256
// rollouts, V = 151,936 bf16, row counts 8..256, CTAs of 128 threads in
// clusters of 4..16 and of 512 threads in clusters of 2..16, 64-step
// graphs, us per step) found the fastest step
//  * from 33 rows up: 128-thread CTAs, the step's rows x C filling about 0.85
//    of one wave (8 CTAs per SM), C at most 12 -- 4 CTAs per row at 256 rows
//    (26.4 us), 8 at 128 (15.7), 12 at 64 (10.6); filling the whole wave
//    (1,120-1,216 CTAs) or clusters of 16 cost 2-5 us a step;
//  * at 32 rows or fewer: 512-thread CTAs in clusters of 8 (8 rows: 5.1 us
//    against 6.0 for 128-thread CTAs in clusters of 16); larger clusters of
//    512-thread CTAs were slower (16 rows in clusters of 16: 8.9 us).
struct Shape {
  int threads, cluster;
};

Shape choose_shape(int64_t rows, int sms) {
  const int ft = g_force_threads.load(std::memory_order_relaxed);
  const int fc = g_force_cluster.load(std::memory_order_relaxed);
  if (ft > 0 || fc > 0) return Shape{ft > 0 ? ft : kStepThreadsSmall, fc > 0 ? fc : 1};
  if (rows <= 4) return Shape{kStepThreadsLarge, 16};
  if (rows <= 32) return Shape{kStepThreadsLarge, 8};
  const int64_t fill = (int64_t)sms * 8 * 85 / 100;  // 128-thread CTAs in 0.85 of a wave
  int64_t c = fill / rows;
  if (c > 12) c = 12;
  return Shape{kStepThreadsSmall, (int)(c < 1 ? 1 : c)};
}

// Cluster sizes above 8 need the non-portable attribute, set once per device
// for each kernel (one set of statics per template instance).
template <typename LT, bool VEC, bool COMPACT, int THREADS>
cudaError_t allow_large_clusters(int dev) {
  static std::atomic<int> done[kMaxDev];
  if (done[dev].load(std::memory_order_acquire)) return cudaSuccess;
  const cudaError_t e =
      cudaFuncSetAttribute(score_step_kernel<LT, VEC, COMPACT, THREADS>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  if (e == cudaSuccess) done[dev].store(1, std::memory_order_release);
  return e;
}

template <typename LT, bool VEC, bool COMPACT, int THREADS>
cudaError_t launch_step_pdl(const StepParams& p, int C, int dev, cudaStream_t stream) {
  if (C > 8) {
    const cudaError_t e = allow_large_clusters<LT, VEC, COMPACT, THREADS>(dev);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.B * (unsigned)C);
  cfg.blockDim = dim3(THREADS);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, score_step_kernel<LT, VEC, COMPACT, THREADS>, p);
}

template <bool COMPACT, int THREADS>
cudaError_t launch_step_form(const StepParams& p, int dtype, bool vec, int C, int dev, cudaStream_t stream) {
  if (dtype == STRIDE_DTYPE_BF16)
    return vec ? launch_step_pdl<__nv_bfloat16, true, COMPACT, THREADS>(p, C, dev, stream)
               : launch_step_pdl<__nv_bfloat16, false, COMPACT, THREADS>(p, C, dev, stream);
  return vec ? launch_step_pdl<float, true, COMPACT, THREADS>(p, C, dev, stream)
             : launch_step_pdl<float, false, COMPACT, THREADS>(p, C, dev, stream);
}

}  // namespace

int set_step_shape_override(int threads, int C) {
  if (C < 0 || C > kStepMaxCluster) return -1;
  if (threads != 0 && threads != kStepThreadsSmall && threads != kStepThreadsLarge) return -1;
  g_force_threads.store(threads, std::memory_order_relaxed);
  g_force_cluster.store(C, std::memory_order_relaxed);
  return 0;
}

cudaError_t launch_score_step(const StepParams& p, int dtype, bool vec, cudaStream_t stream) {
  int dev = 0;
  cudaError_t e = cudaSuccess;
  const int sms = current_device_sms(&dev, &e);
  if (sms <= 0) return e != cudaSuccess ? e : cudaErrorInvalidDevice;
  Shape sh = choose_shape(p.B, sms);
  // a few whole vectors per thread of a rank at least
  while (sh.cluster > 1 && (int64_t)p.V < (int64_t)sh.threads * sh.cluster) sh.cluster >>= 1;
  if (sh.threads == kStepThreadsLarge && (int64_t)p.V < (int64_t)kStepThreadsLarge * 2) sh.threads = kStepThreadsSmall;
  const bool compact = p.rollout_idx != nullptr;
  if (sh.threads == kStepThreadsLarge)
    e = compact ? launch_step_form<true, kStepThreadsLarge>(p, dtype, vec, sh.cluster, dev, stream)
                : launch_step_form<false, kStepThreadsLarge>(p, dtype, vec, sh.cluster, dev, stream);
  else
    e = compact ? launch_step_form<true, kStepThreadsSmall>(p, dtype, vec, sh.cluster, dev, stream)
                : launch_step_form<false, kStepThreadsSmall>(p, dtype, vec, sh.cluster, dev, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace stride
