// score_batch.cu -- fused batch scoring kernel for ragged trajectories
// (sm_103a).
//
// One CTA per row, rows taken in ticket order.  Each CTA
//   1. streams the student row and the teacher row once, interleaved, with
//      16-byte non-allocating loads, into single-pass online log-sum-exp
//      pairs (stride_device.cuh);
//   2. gathers S[y], T[y] and forms log pi_S(y), log pi_T(y) and
//      d = log pi_S - log pi_T (Eq. 1, Eq. 4);
//   3. takes part in a decoupled-lookback segmented scan over rows that
//      carries, per trajectory, the running stop sum and, per turn, the sums
//      of log pi_T and d;
//   4. at a turn's last row writes the turn's statistics (n_k, l_k = Eq. 4)
//      and, where the stop test applies, records the first crossing of
//      lambda with atomicMin (Eq. 5 / Sec. 5.5).
//
// The row tail (steps 2-4) and the scan protocol live in row_scan.cuh.
#include <cooperative_groups.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <mutex>

#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"
#include "row_scan.cuh"

namespace stride {

int current_device_sms(int* dev_out, cudaError_t* err) {
  constexpr int kMaxDev = 64;
  static std::atomic<int> cache[kMaxDev];  // 0 = not looked up yet
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (dev_out) *dev_out = dev;
  if (e != cudaSuccess || dev < 0 || dev >= kMaxDev) {
    if (err) *err = e != cudaSuccess ? e : cudaErrorInvalidDevice;
    return 0;
  }
  int sms = cache[dev].load(std::memory_order_relaxed);
  if (sms > 0) return sms;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess || sms <= 0) {
    if (err) *err = e != cudaSuccess ? e : cudaErrorInvalidDevice;
    return 0;
  }
  cache[dev].store(sms, std::memory_order_relaxed);
  return sms;
}

constexpr int kBatchThreads = 512;
constexpr int kBatchWarps = kBatchThreads / 32;
constexpr int kBatchUnroll = 4;

template <typename LT, bool VEC>
__global__ void __launch_bounds__(kBatchThreads, 2) score_batch_kernel(const BatchParams p) {
  __shared__ int64_t s_tile;
  __shared__ float s_red[4][kBatchWarps];
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  if (tid == 0) s_tile = (int64_t)atomicAdd(p.ticket, 1u);
  __syncthreads();
  const int64_t tile = s_tile;
  const int64_t r = p.row_begin + tile;
  const LT* srow = reinterpret_cast<const LT*>(p.S) + tile * p.ld;
  const LT* trow = teacher_row<LT>(p, tile);

  // Warp 0 starts the dependent lookups (token -> gathered logits, row ->
  // trajectory -> turn) before streaming, so their latency overlaps the
  // other warps' loads; warp 1 checks the layout arrays.
  int32_t y = 0;
  float xs = __int_as_float(0x7fc00000), xt = xs;
  RowMeta meta;
  if (warp == 0) {
    if (lane == 0) {
      y = __ldg(p.tokens + tile);
      if (y >= 0 && y < p.V) {
        xs = to_f32(srow[y]);
        xt = to_f32(trow[y]);
      }
    }
    meta = find_row_meta(p, r, lane);
  } else if (warp == 1 && lane == 0) {
    validate_layout(p, tile);
  }

  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  stream_pair<LT, VEC, kBatchUnroll>(srow, trow, 0, p.V, tid, kBatchThreads, mS, sS, mT, sT);
  warp_merge2(mS, sS, mT, sT);
  if (lane == 0) {
    s_red[0][warp] = mS;
    s_red[1][warp] = sS;
    s_red[2][warp] = mT;
    s_red[3][warp] = sT;
  }
  __syncthreads();
  if (warp != 0) return;

  mS = lane < kBatchWarps ? s_red[0][lane] : kMaxStart;
  sS = lane < kBatchWarps ? s_red[1][lane] : 0.f;
  mT = lane < kBatchWarps ? s_red[2][lane] : kMaxStart;
  sT = lane < kBatchWarps ? s_red[3][lane] : 0.f;
  warp_merge2(mS, sS, mT, sT);
  const float lse_s = lse_finish(mS, sS);
  const float lse_t = lse_finish(mT, sT);

  finish_row(p, tile, r, meta, y, xs, xt, lse_s, lse_t, lane);
}

// Small windows: a few rows per SM leave the persistent kernel latency-bound
// (each SM streams its rows one after another), so a window of at most 8
// rows per SM splits every row over the C CTAs of a thread-block cluster
// instead (C = 1: one CTA per row), C chosen at launch (split_cluster below)
// so that the window is one wave of 128-thread CTAs.  Cluster i scores
// window row i: every rank streams its share of the vocabulary of S and T,
// rank 0 merges the ranks' pairs through distributed shared memory, writes
// the row's outputs and leaves its two log-probs in the workspace.  The scan
// (turn statistics, stop rule, loss, profile, carried state) then runs as
// the tiled scan on those log-probs (vocab_parallel.cu), launched as a
// programmatic dependent of this kernel.  In a window whose rows all finish
// streaming together, a lookback per row cost a chain of prefixes after the
// last row (12 us on a 512-row segment); the tiled scan scans 128 rows per
// CTA, and a window of at most 16 such tiles runs as one cluster whose
// tiles exchange their aggregates through distributed shared memory (no
// chain at all).
namespace cg = cooperative_groups;
constexpr int kSplitMaxCluster = 8;
constexpr int kSplitThreads = 128;
constexpr int kSplitWarps = kSplitThreads / 32;
constexpr int kSplitBlocksPerSm = 8;  // 128 threads at <= 64 registers

template <typename LT, bool VEC>
__global__ void __launch_bounds__(kSplitThreads, kSplitBlocksPerSm)
    score_batch_split_kernel(const BatchParams p) {
  __shared__ float s_red[4][kSplitWarps];
  __shared__ float4 s_part[kSplitMaxCluster];  // rank 0: every rank's (mS, sS, mT, sT), written by the ranks
  // first cluster-barrier phase: waited on before the first remote store
  // (every CTA of the cluster has started by then)
  cluster_arrive_relaxed();
  // Launched as a programmatic dependent of the previous kernel on the
  // stream: the CTAs may be scheduled while it finishes, and each waits for
  // its completion before the first global access.  Only then may the
  // dependent scan be scheduled, so that whatever the previous kernels
  // wrote (the layout, the carried state) is complete when the scan reads
  // it before its own wait.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  if (blockIdx.x == 0) {
    // What the scan needs at zero: its tile ticket (the header's second
    // word) and one flag per tile of kScanTileRowsDependent rows.  The scan
    // reads them only after this grid has completed.
    const int64_t n_tiles = (p.n_rows + kScanTileRowsDependent - 1) / kScanTileRowsDependent;
    for (int64_t t = threadIdx.x; t < n_tiles; t += blockDim.x) p.flags[t * kFlagStride] = 0u;
    if (threadIdx.x == 0) p.ticket[1] = 0u;
  }
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int n_ranks = (int)cluster.num_blocks();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t tile = blockIdx.x / n_ranks;  // window row
  const LT* srow = reinterpret_cast<const LT*>(p.S) + tile * p.ld;
  const LT* trow = teacher_row<LT>(p, tile);

  // The token id is loaded now; its logits are gathered, and this row's
  // share of the layout checks made (the scan skips them), after the
  // stream, where they overlap the wait for the other ranks.
  int32_t y = 0;
  float xs = __int_as_float(0x7fc00000), xt = xs;
  if (rank == 0 && tid == 0) y = __ldg(p.tokens + tile);
  int c0, c1;
  if (VEC) {
    constexpr int P = LogitTraits<LT>::kPerVec;
    const int nv = p.V / P;
    const int per = (nv + n_ranks - 1) / n_ranks;
    c0 = min(nv, rank * per) * P;
    c1 = (rank == n_ranks - 1) ? p.V : min(nv, (rank + 1) * per) * P;
  } else {
    const int per = (p.V + n_ranks - 1) / n_ranks;
    c0 = min(p.V, rank * per);
    c1 = min(p.V, (rank + 1) * per);
  }
  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  stream_pair<LT, VEC, 4>(srow, trow, c0, c1, tid, kSplitThreads, mS, sS, mT, sT);
  if (rank == 0 && tid == 0 && y >= 0 && y < p.V) {
    xs = to_f32(srow[y]);
    xt = to_f32(trow[y]);
  } else if (rank == 0 && tid == 32) {
    validate_layout(p, tile);
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
    mS = lane < kSplitWarps ? s_red[0][lane] : kMaxStart;
    sS = lane < kSplitWarps ? s_red[1][lane] : 0.f;
    mT = lane < kSplitWarps ? s_red[2][lane] : kMaxStart;
    sT = lane < kSplitWarps ? s_red[3][lane] : 0.f;
    warp_merge2(mS, sS, mT, sT);
    if (lane == 0) cluster.map_shared_rank(s_part, 0)[rank] = make_float4(mS, sS, mT, sT);
  }
  // second phase: the ranks' pairs are released to rank 0; the other ranks
  // leave (nobody reads their shared memory)
  cluster_arrive_release();
  if (rank != 0) return;
  cluster_wait_acquire();
  if (warp == 0) {
    mS = kMaxStart;
    sS = 0.f;
    mT = kMaxStart;
    sT = 0.f;
    if (lane < n_ranks) {
      const float4 q = s_part[lane];
      mS = q.x;
      sS = q.y;
      mT = q.z;
      sT = q.w;
    }
    warp_merge2(mS, sS, mT, sT);
    if (lane == 0) {
      const float lse_s = lse_finish(mS, sS), lse_t = lse_finish(mT, sT);
      if (!(y >= 0 && y < p.V)) set_status(p.dev_status, STRIDE_DEV_TOKEN_RANGE);
      const float lps = xs - lse_s, lpt = xt - lse_t;
      const stride_row_outputs& o = p.out;
      if (o.logp_s) o.logp_s[tile] = lps;
      if (o.logp_t) o.logp_t[tile] = lpt;
      if (o.lse_s) o.lse_s[tile] = lse_s;
      if (o.lse_t) o.lse_t[tile] = lse_t;
      if (o.x_s) o.x_s[tile] = xs;
      if (o.x_t) o.x_t[tile] = xt;
      p.ws_logp_s[tile] = lps;
      p.ws_logp_t[tile] = lpt;
    }
  }
}

// Multi-teacher pre-pass: the teacher row of each window row, from its
// trajectory's domain buffer.  A row whose domain or domain row is out of
// range gets its domain-0 row 0 (always valid memory) and sets
// STRIDE_DEV_BAD_LAYOUT: its results are meaningless, never a fault.
__global__ void teacher_rows_kernel(const BatchParams p, const TeacherTable tt,
                                    const uint8_t* __restrict__ traj_domain,
                                    const int64_t* __restrict__ traj_T_row0, const void** rows_out) {
  // A programmatic dependent of the previous kernel, which may be the
  // previous window's scoring kernel still reading this workspace's table:
  // wait for it before the first store; the clearing and scoring kernels
  // that follow may be scheduled at once (they wait for this grid in turn).
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= p.n_rows) return;
  const int64_t r = p.row_begin + t;
  int64_t lo = 0, hi = p.n_traj - 1;  // largest i with traj_row_off[i] <= r
  while (lo < hi) {
    const int64_t mid = (lo + hi + 1) >> 1;
    if (__ldg(p.traj_row_off + mid) <= r) lo = mid; else hi = mid - 1;
  }
  const int dom = __ldg(traj_domain + lo);
  const int64_t tr = __ldg(traj_T_row0 + lo) + (r - __ldg(p.traj_row_off + lo));
  const unsigned char* row = static_cast<const unsigned char*>(tt.base[0]);
  if (dom < tt.n_domains && tr >= 0 && tr < tt.rows[dom] && r >= __ldg(p.traj_row_off)) {
    row = static_cast<const unsigned char*>(tt.base[dom]) + tr * tt.ld_bytes;
  } else {
    set_status(p.dev_status, STRIDE_DEV_BAD_LAYOUT);
  }
  rows_out[t] = row;
}

cudaError_t launch_teacher_rows(const BatchParams& p, const TeacherTable& tt, const uint8_t* traj_domain,
                                const int64_t* traj_T_row0, const void** rows_out, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((p.n_rows + 255) / 256));
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, teacher_rows_kernel, p, tt, traj_domain, traj_T_row0, rows_out);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

BatchWorkspaceLayout batch_workspace_layout(int64_t n_rows) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  BatchWorkspaceLayout L;
  const size_t n = n_rows > 0 ? (size_t)n_rows : 0;
  L.ticket_off = 0;
  L.flags_off = 256;
  L.agg_off = L.flags_off + up(n * sizeof(uint32_t) * kFlagStride);
  L.incl_off = L.agg_off + up(n * sizeof(ScanSlot));
  L.logp_s_off = L.incl_off + up(n * sizeof(ScanSlot));
  L.logp_t_off = L.logp_s_off + up(n * sizeof(float));
  L.total = L.logp_t_off + up(n * sizeof(float));
  L.clear_bytes = L.agg_off;  // ticket + flags
  if (n == 0) L.total = 0;
  return L;
}

// Cluster size of the small-window kernel: the largest C in {8, 4, 2, 1}
// whose n_rows * C CTAs fit in one wave (kSplitBlocksPerSm per SM), 0 when
// even C = 1 does not (the window then takes the persistent kernel).  A
// sweep on GB300 over windows of 64..2,432 rows (bf16 V = 151,936 and fp32
// V = 32,000) found this choice within a few percent of the best cluster size
// at every window, and up to 1,216 rows faster than the persistent kernel,
// which streams each SM's few rows one after another; from 1,600 rows on the
// persistent kernel is faster.
// STRIDE_SPLIT_FORCE_CLUSTER (a build define) fixes C for launch-shape sweeps.
#ifndef STRIDE_SPLIT_FORCE_CLUSTER
#define STRIDE_SPLIT_FORCE_CLUSTER 0
#endif
static int split_cluster(int64_t n_rows, int sms) {
  if (STRIDE_SPLIT_FORCE_CLUSTER > 0) return STRIDE_SPLIT_FORCE_CLUSTER;
  const int64_t slots = (int64_t)kSplitBlocksPerSm * sms;
  for (int c = kSplitMaxCluster; c >= 1; c >>= 1)
    if (n_rows * c <= slots) return c;
  return 0;
}

// Forced batch kernel (tests and diagnosis): 0 automatic, kForceStream,
// kForceRows, or kForceSplit + C (C = 0: the split kernel with its automatic
// cluster size).  Its first value comes from the environment variable
// STRIDE_BATCH_KERNEL, read once per process at the first batch call;
// stride_force_batch_kernel changes it.
constexpr int kForceStream = 1, kForceRows = 2, kForceSplit = 16;
static std::atomic<int> g_batch_force{-1};  // -1: environment not read yet

static int parse_batch_kernel(const char* name) {
  if (!name || !*name || !strcmp(name, "auto")) return 0;
  if (!strcmp(name, "stream")) return kForceStream;
  if (!strcmp(name, "rows")) return kForceRows;
  if (!strcmp(name, "split")) return kForceSplit;
  if (!strcmp(name, "split1")) return kForceSplit + 1;
  if (!strcmp(name, "split2")) return kForceSplit + 2;
  if (!strcmp(name, "split4")) return kForceSplit + 4;
  if (!strcmp(name, "split8")) return kForceSplit + 8;
  return -1;
}

static int batch_kernel_override() {
  int f = g_batch_force.load(std::memory_order_relaxed);
  if (f >= 0) return f;
  static std::once_flag once;
  std::call_once(once, [] {
    const int v = parse_batch_kernel(getenv("STRIDE_BATCH_KERNEL"));
    int expect = -1;
    g_batch_force.compare_exchange_strong(expect, v < 0 ? 0 : v);
  });
  return g_batch_force.load(std::memory_order_relaxed);
}

int set_batch_kernel_override(const char* name) {
  const int v = parse_batch_kernel(name);
  if (v < 0) return -1;
  (void)batch_kernel_override();  // the environment's value, if any, is superseded from here on
  g_batch_force.store(v, std::memory_order_relaxed);
  return 0;
}

template <typename LT, bool VEC>
static cudaError_t launch_split(const BatchParams& p, int C, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(p.n_rows * C));
  cfg.blockDim = dim3(kSplitThreads);
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
  return cudaLaunchKernelEx(&cfg, score_batch_split_kernel<LT, VEC>, p);
}

// Clears what a batch call needs at zero in its workspace (the ticket and
// the scan flags), launched as a programmatic dependent of the previous
// kernel on the stream: its CTAs wait for that kernel (which may be the
// previous window's scoring kernel, still using the same workspace) before
// the first store.  It lets its own dependent, the scoring kernel, be
// scheduled at once: that kernel's CTAs set up their shared memory and
// barriers while the previous window drains, then wait for this grid to
// complete.  (It replaces a memset node, which ended the programmatic chain:
// 7.5 us between one 16,384-row window's last CTA and the next one's first
// on GB300.)
__global__ void clear_workspace_kernel(uint4* __restrict__ p, int64_t n16) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const uint4 z = make_uint4(0u, 0u, 0u, 0u);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += (int64_t)gridDim.x * blockDim.x)
    p[i] = z;
}

cudaError_t launch_clear_workspace(void* ws, size_t bytes, int sms, cudaStream_t stream) {
  const int64_t n16 = (int64_t)(bytes / 16);  // workspace offsets are 256-byte multiples
  if (n16 <= 0) return cudaSuccess;
  int64_t blocks = (n16 + 255) / 256;
  if (blocks > 2 * (int64_t)sms) blocks = 2 * (int64_t)sms;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, clear_workspace_kernel, reinterpret_cast<uint4*>(ws), n16);
}

cudaError_t launch_score_batch(const BatchParams& p, int dtype, bool vec, size_t clear_bytes, cudaStream_t stream) {
  // Small windows split each row over a cluster (split_cluster); 16-byte-
  // aligned rows with at least one whole vector otherwise take the
  // persistent bulk-copy kernel (score_batch_stream.cu); the rest take one
  // CTA per row.
  int dev = 0;
  cudaError_t qe = cudaSuccess;
  const int sms = current_device_sms(&dev, &qe);
  if (sms <= 0) return qe != cudaSuccess ? qe : cudaErrorInvalidDevice;
  const int force = batch_kernel_override();
  const bool f_split = force >= kForceSplit;
  const bool f_stream = force == kForceStream;
  const bool f_rows = force == kForceRows;
  int C = (f_stream || f_rows) ? 0 : split_cluster(p.n_rows, sms);
  if (f_split) {
    const int want = force - kForceSplit;
    if (want > 0) C = want;
    else if (C == 0) C = 2;
  }
  if (C > 0 && p.V < 32 * (int64_t)C) C = f_split ? 1 : 0;  // a few logits per rank at least
  if (C > 0) {
    // no memset: the split kernel clears the scan's ticket and tile flags
    cudaError_t e;
    if (dtype == STRIDE_DTYPE_BF16)
      e = vec ? launch_split<__nv_bfloat16, true>(p, C, stream) : launch_split<__nv_bfloat16, false>(p, C, stream);
    else
      e = vec ? launch_split<float, true>(p, C, stream) : launch_split<float, false>(p, C, stream);
    if (e != cudaSuccess) return e;
    // the scan on the rows' log-probs; its tile tickets use the header's
    // second word (cleared with the first)
    BatchParams q = p;
    q.ticket = p.ticket + 1;
    return launch_scan_logprobs(q, p.ws_logp_s, p.ws_logp_t, stream, true);
  }
  {
    const cudaError_t e = launch_clear_workspace(p.ticket, clear_bytes, sms, stream);
    if (e != cudaSuccess) return e;
  }
  const int per_vec = dtype == STRIDE_DTYPE_BF16 ? 8 : 4;
  // (the persistent kernel counts a row's bytes in 32 bits: rows of up to
  // 2 GB, far beyond any vocabulary, take it)
  const int64_t row_bytes = (int64_t)p.V * (dtype == STRIDE_DTYPE_BF16 ? 2 : 4);
  if (vec && p.V >= per_vec && row_bytes <= ((int64_t)1 << 31) && !f_rows)
    return launch_score_batch_stream(p, dtype, stream);
  const dim3 grid((unsigned)p.n_rows), block(kBatchThreads);
  if (dtype == STRIDE_DTYPE_BF16) {
    if (vec)
      score_batch_kernel<__nv_bfloat16, true><<<grid, block, 0, stream>>>(p);
    else
      score_batch_kernel<__nv_bfloat16, false><<<grid, block, 0, stream>>>(p);
  } else {
    if (vec)
      score_batch_kernel<float, true><<<grid, block, 0, stream>>>(p);
    else
      score_batch_kernel<float, false><<<grid, block, 0, stream>>>(p);
  }
  return cudaGetLastError();
}

}  // namespace stride
