// vocab_parallel.cu -- the scoring path for vocabulary-sharded logits and for
// given log-probs (sm_103a).
//
// When a teacher (or student) runs with tensor parallelism its logits are
// split by vocabulary columns across ranks.  Each rank reduces its shard of
// a row to a log-sum-exp pair (m, s) and, if the sampled token falls in its
// columns, the token's logit: 24 bytes per row for S and T together
// (partial_lse_kernel).  After the ranks exchange those, the pairs merge
// into the row's log-sum-exp (combine_kernel), which gives the same
// log-probs as the full row.  The rest of the path (turn statistics, stop
// rule, OPD loss, profile, carried state) then runs on the log-probs
// (scan_logprobs_tile_kernel): a segmented scan per tile of 256 rows, and
// the fused kernels' decoupled lookback (row_scan.cuh) between tiles -- or,
// for a small window after the small-window kernel, tiles of 128 rows in
// one thread-block cluster that exchange their aggregates through
// distributed shared memory.
#include <cooperative_groups.h>
#include <math.h>

#include <atomic>

#include "row_scan.cuh"
#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace stride {

// Shard-pass launch shape (build defines, for sweeps): threads per CTA,
// 16-byte loads in flight per thread and tensor, and CTAs per SM promised
// to the register allocator.  A sweep on GB300 (4 shards of the batch-
// scoring rows, 37,984 bf16 logits per shard row; ms for the 4 passes):
// 128 threads x 4 loads at 8 CTAs per SM (58 registers) 12.25; 256 x 3 at
// 8 per SM 12.26; 128 x 4 unbounded (7 per SM) 12.30; 256 x 4 at 4 per SM
// 12.48; 256 x 2 12.82; 256 x 4 unbounded (66 registers, 3 per SM) 13.03.
#ifndef STRIDE_PARTIAL_THREADS
#define STRIDE_PARTIAL_THREADS 128
#endif
#ifndef STRIDE_PARTIAL_UNROLL
#define STRIDE_PARTIAL_UNROLL 4
#endif
#ifndef STRIDE_PARTIAL_MIN_BLOCKS
#define STRIDE_PARTIAL_MIN_BLOCKS 8
#endif
constexpr int kPartialThreads = STRIDE_PARTIAL_THREADS;
constexpr int kPartialWarps = kPartialThreads / 32;
static_assert(kPartialThreads % 32 == 0 && kPartialWarps <= 32, "whole warps, at most 32");

struct PartialParams {
  const void* S;
  const void* T;
  int64_t ld;
  int32_t V_shard;
  int64_t col0;
  int32_t V_total;
  const int32_t* tokens;
  int64_t rows;
  float* partials;  // [rows][6]
  int32_t* dev_status;
};

// One CTA per row: (m, s) of S and T over this shard's columns, and the
// gathered logits when the token is one of them (NaN otherwise).
template <typename LT, bool VEC>
__global__ void __launch_bounds__(kPartialThreads, STRIDE_PARTIAL_MIN_BLOCKS) partial_lse_kernel(const PartialParams p) {
  __shared__ float s_red[4][kPartialWarps];
  const int64_t r = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const LT* srow = reinterpret_cast<const LT*>(p.S) + r * p.ld;
  const LT* trow = reinterpret_cast<const LT*>(p.T) + r * p.ld;
  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  stream_pair<LT, VEC, STRIDE_PARTIAL_UNROLL>(srow, trow, 0, p.V_shard, tid, kPartialThreads, mS, sS, mT, sT);
  warp_merge2(mS, sS, mT, sT);
  if (lane == 0) {
    s_red[0][warp] = mS;
    s_red[1][warp] = sS;
    s_red[2][warp] = mT;
    s_red[3][warp] = sT;
  }
  __syncthreads();
  if (warp != 0) return;
  mS = lane < kPartialWarps ? s_red[0][lane] : kMaxStart;
  sS = lane < kPartialWarps ? s_red[1][lane] : 0.f;
  mT = lane < kPartialWarps ? s_red[2][lane] : kMaxStart;
  sT = lane < kPartialWarps ? s_red[3][lane] : 0.f;
  warp_merge2(mS, sS, mT, sT);
  if (lane == 0) {
    const float nan = __int_as_float(0x7fc00000);
    const int32_t y = __ldg(p.tokens + r);
    const int64_t c = (int64_t)y - p.col0;
    float xs = nan, xt = nan;
    if (c >= 0 && c < p.V_shard) {
      xs = to_f32(srow[c]);
      xt = to_f32(trow[c]);
    }
    float* o = p.partials + r * 6;
    o[0] = mS;
    o[1] = sS;
    o[2] = mT;
    o[3] = sT;
    o[4] = xs;
    o[5] = xt;
  }
}

// One thread per row: merge the shards' pairs, take the logit from the shard
// that owns the token (exactly one must), form the log-probs.
__global__ void combine_kernel(const float* __restrict__ parts, int32_t n_shards, int64_t rows,
                               float* logp_s, float* logp_t, float* lse_s, float* lse_t,
                               int32_t* dev_status) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= rows) return;
  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  float xs = 0.f, xt = 0.f;
  int owners = 0;
  for (int k = 0; k < n_shards; ++k) {
    const float* q = parts + ((int64_t)k * rows + r) * 6;
    lse_merge(mS, sS, q[0], q[1]);
    lse_merge(mT, sT, q[2], q[3]);
    if (!isnan(q[4]) || !isnan(q[5])) {
      xs = q[4];
      xt = q[5];
      ++owners;
    }
  }
  const float ls = lse_finish(mS, sS), lt = lse_finish(mT, sT);
  const float nan = __int_as_float(0x7fc00000);
  if (owners != 1) {
    set_status(dev_status, STRIDE_DEV_TOKEN_RANGE);
    xs = nan;
    xt = nan;
  }
  if (logp_s) logp_s[r] = xs - ls;
  if (logp_t) logp_t[r] = xt - lt;
  if (lse_s) lse_s[r] = ls;
  if (lse_t) lse_t[r] = lt;
}

// The scan on given log-probs, one tile of TILE consecutive rows per CTA (one
// row per thread; kScanTileRows on its own, kScanTileRowsDependent after the
// small-window kernel), tiles taken in ticket order (by block index in a
// small dependent grid, below).  Without a logit pass to hide it, a lookback
// per row is what the time goes to (each row waits on its predecessors'
// prefixes), so the rows of a tile are scanned together in the CTA and only
// the tile takes part in the decoupled lookback:
//   1. warps 0 and 1 find the tile's first turn and trajectory; the CTA
//      stages the offsets of the next kScanTileRows + 1 turns and
//      trajectories in shared memory and every thread finds its row's turn
//      and trajectory there;
//   2. each row's element: the stop-sum term, log pi_T, d, logp_S * d, and
//      two restart marks -- the open-turn sums restart at a turn's first row,
//      the running sum at a seeded row (a trajectory's first row, or the
//      window's), whose element already holds the carried state;
//   3. a segmented inclusive scan of the tile's elements (warp shuffles, then
//      the warps' totals);
//   4. the tile's aggregate is published (as an INCLUSIVE prefix at once if
//      the tile holds a seeded row, since nothing before it matters then;
//      tile 0 always does), warp 0 folds its predecessors' (row_scan.cuh
//      lookback) and publishes the tile's inclusive prefix (the cluster
//      form, below: the aggregates go to the later tiles' shared memory,
//      and warp 0 folds its predecessors' there);
//   5. every row completes with its inclusive and exclusive prefixes: turn
//      statistics and carried state (row_tail), the within-turn profile into
//      the CTA's shared bins;
//   6. a second segmented scan (restarting at trajectory starts) gives each
//      trajectory's retained loss and first crossing in the tile, so the
//      trajectory's record takes one update per tile instead of one per row
//      (the rows of a token-sum segment below lambda all contended for it).
constexpr int kRestartTurn = 1;  // st, sd, sl restart at this row
constexpr int kRestartSum = 2;   // c restarts (a seeded row)

// A row's element inside a tile.  The running stop sum c is fp64 (the stop
// rule compares it with lambda); the open-turn sums of log pi_T, d and the
// loss term are fp32 inside the tile (at most kScanTileRows terms each,
// summed in a tree: relative error a few 1e-7 of the summed magnitudes), in
// the cluster form's fold of at most 16 tile aggregates, and where the
// tile's prefix meets a row; the lookback's prefix over tiles and every
// stored sum are fp64.  GB300 runs FP64 at 1/64 of the FP32 rate, and the
// tile scans' fp64 adds were what a small window's scan waited on (a
// 512-row window in one CTA: 6.6 us for the block scan).
struct TileElem {
  double c;
  float st, sd, sl;
  int flags;
};

// A prefix over tiles as the lookback folds it: fp64 throughout.  (A row's
// inclusive and exclusive values, and the cluster form's fold, use TileElem:
// the stop sum fp64, the open-turn sums fp32.)
struct PreElem {
  double c, st, sd, sl;
};

__device__ __forceinline__ TileElem tile_combine(const TileElem& a, const TileElem& b) {
  TileElem r;
  r.c = (b.flags & kRestartSum) ? b.c : a.c + b.c;
  r.st = (b.flags & kRestartTurn) ? b.st : a.st + b.st;
  r.sd = (b.flags & kRestartTurn) ? b.sd : a.sd + b.sd;
  r.sl = (b.flags & kRestartTurn) ? b.sl : a.sl + b.sl;
  r.flags = a.flags | b.flags;
  return r;
}

// A tile's prefix followed by an in-tile prefix.
__device__ __forceinline__ PreElem pre_combine(const PreElem& a, const TileElem& b) {
  PreElem r;
  r.c = (b.flags & kRestartSum) ? b.c : a.c + b.c;
  r.st = (b.flags & kRestartTurn) ? (double)b.st : a.st + (double)b.st;
  r.sd = (b.flags & kRestartTurn) ? (double)b.sd : a.sd + (double)b.sd;
  r.sl = (b.flags & kRestartTurn) ? (double)b.sl : a.sl + (double)b.sl;
  return r;
}

__device__ __forceinline__ TileElem tile_shfl_up(const TileElem& v, int d) {
  TileElem o;
  o.c = __shfl_up_sync(0xffffffffu, v.c, d);
  o.st = __shfl_up_sync(0xffffffffu, v.st, d);
  o.sd = __shfl_up_sync(0xffffffffu, v.sd, d);
  o.sl = __shfl_up_sync(0xffffffffu, v.sl, d);
  o.flags = __shfl_up_sync(0xffffffffu, v.flags, d);
  return o;
}

// Per-trajectory sums of the tile's rows for the trajectory's record: the
// retained rows' loss terms and count, and whether a row crossed lambda.
// Restarts at a trajectory's first row.
struct TrajElem {
  float loss;  // a tile's rows only; added to the fp64 record
  int count;
  int crossed;
  int restart;
};

__device__ __forceinline__ TrajElem traj_combine(const TrajElem& a, const TrajElem& b) {
  if (b.restart) return b;
  return TrajElem{a.loss + b.loss, a.count + b.count, a.crossed | b.crossed, a.restart};
}

__device__ __forceinline__ TrajElem traj_shfl_up(const TrajElem& v, int d) {
  TrajElem o;
  o.loss = __shfl_up_sync(0xffffffffu, v.loss, d);
  o.count = __shfl_up_sync(0xffffffffu, v.count, d);
  o.crossed = __shfl_up_sync(0xffffffffu, v.crossed, d);
  o.restart = __shfl_up_sync(0xffffffffu, v.restart, d);
  return o;
}

__device__ __forceinline__ TileElem elem_combine(const TileElem& a, const TileElem& b) { return tile_combine(a, b); }
__device__ __forceinline__ TrajElem elem_combine(const TrajElem& a, const TrajElem& b) { return traj_combine(a, b); }
__device__ __forceinline__ TileElem elem_shfl_up(const TileElem& v, int d) { return tile_shfl_up(v, d); }
__device__ __forceinline__ TrajElem elem_shfl_up(const TrajElem& v, int d) { return traj_shfl_up(v, d); }

// Inclusive and exclusive scan of one element per thread over the CTA's
// WARPS warps, in thread order: warp shuffles, then warp 0 scans the warps'
// totals once (each thread then combines with one prefix).  `id` is the
// identity; s_tot and s_pre hold WARPS elements.
template <int WARPS, typename E>
__device__ __forceinline__ void block_scan(const E& v, const E& id, int lane, int warp, E* s_tot, E* s_pre,
                                           E& incl_out, E& excl_out) {
  E incl = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const E o = elem_shfl_up(incl, d);
    if (lane >= d) incl = elem_combine(o, incl);
  }
  const E up1 = elem_shfl_up(incl, 1);
  if (lane == 31) s_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    E t = lane < WARPS ? s_tot[lane] : id;
#pragma unroll
    for (int d = 1; d < WARPS; d <<= 1) {
      const E o = elem_shfl_up(t, d);
      if (lane >= d) t = elem_combine(o, t);
    }
    const E e = elem_shfl_up(t, 1);
    if (lane < WARPS) s_pre[lane] = (lane == 0) ? id : e;
  }
  __syncthreads();
  const E wpre = s_pre[warp];
  incl_out = elem_combine(wpre, incl);
  excl_out = (lane == 0) ? wpre : elem_combine(wpre, up1);
}

// Largest j in [0, n) with a[j] <= r (a ascending, a[0] <= r).
__device__ __forceinline__ int smem_upper_le(const int64_t* a, int n, int64_t r) {
  int lo = 0, hi = n - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (a[mid] <= r) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// The cluster form (CLUSTER; a small window of at most kClusterMaxTiles
// tiles, launched as ONE thread-block cluster of one CTA per tile, so that
// the tiles run at once): in place of the lookback through global memory,
// each tile stores its aggregate into the shared memory of every later
// tile of the cluster, and after one cluster barrier folds its
// predecessors' aggregates itself.  A second role of the barrier: the
// carried state is read before the dependency wait and written at a
// trajectory's last row, possibly by a later tile, so every CTA arrives
// once its reads are done and waits before any write.  (In the lookback
// form that order comes from the chain of published prefixes.)
constexpr int kClusterMaxTiles = 16;

template <int TILE, bool CLUSTER>
__global__ void __launch_bounds__(TILE) scan_logprobs_tile_kernel(const BatchParams p,
                                                                          const float* __restrict__ logp_s,
                                                                          const float* __restrict__ logp_t,
                                                                          int64_t n_tiles, bool validate,
                                                                          bool by_ticket) {
  constexpr int kWarps = TILE / 32;
  __shared__ int64_t s_turn_off[TILE + 1];
  __shared__ int64_t s_traj_row[TILE + 1];   // traj_row_off
  __shared__ int64_t s_traj_turn[TILE + 1];  // traj_turn_off, widened
  __shared__ int64_t s_first[2];                      // first turn, first trajectory of the tile
  __shared__ TileElem s_wtot[kWarps];
  __shared__ TileElem s_wpre[kWarps];
  __shared__ TrajElem s_ttot[kWarps];
  __shared__ TrajElem s_tpre[kWarps];
  __shared__ TileElem s_excl;  // the tile's exclusive prefix (flags unused)
  __shared__ TileElem s_agg;
  __shared__ int s_flags;  // bit 0: lookback timed out
  __shared__ double s_prof[3 * STRIDE_PROFILE_BINS];
  __shared__ int64_t s_tile;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // Launched as a programmatic dependent of the kernel that wrote the
  // log-probs (griddepcontrol.wait is a no-op otherwise).  That kernel
  // waited for its own predecessors before letting this grid be scheduled,
  // so the layout and the carried state may be read before the wait; the
  // log-probs, the tile flags and the ticket only after it.  Tiles are
  // taken in ticket order (a tile's lookback waits only on tiles taken
  // before it, which are running or done) unless the grid is small enough
  // to be resident at once, when the block index is the tile.
  if (tid < 3 * STRIDE_PROFILE_BINS) s_prof[tid] = 0.0;
  if (by_ticket) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (tid == 0) s_tile = (int64_t)atomicAdd(p.ticket, 1u);
  } else if (tid == 0) {
    s_tile = (int64_t)blockIdx.x;
  }
  __syncthreads();
  const int64_t tile = s_tile;
  if (tile >= n_tiles) return;
  const int64_t t0 = tile * TILE;           // first window row of the tile
  const int64_t n_here = min((int64_t)TILE, p.n_rows - t0);
  const int64_t r0 = p.row_begin + t0;
  const int64_t w = t0 + tid;  // this thread's window row
  const int64_t r = p.row_begin + w;
  const bool live = tid < n_here;
  // the row's log-probs, in flight while the layout is looked up (after
  // the layout, below, when this grid has not waited yet)
  float lps = 0.f, lpt = 0.f;
  if (live && by_ticket) {
    lps = __ldcg(logp_s + w);
    lpt = __ldcg(logp_t + w);
  }

  // 1. the tile's first turn (warp 0) and first trajectory (warp 1), then
  //    the offsets of the next TILE + 1 of each in shared memory (a layout
  //    of at most TILE turns and trajectories: all of them, no search --
  //    one dependent round trip less before the wait)
  if (p.n_turns <= TILE && p.n_traj <= TILE) {
    if (tid == 0) {
      s_first[0] = p.n_turns > 0 ? 0 : -1;
      s_first[1] = 0;
    }
  } else if (warp == 0) {
    const bool ok = p.n_turns > 0 && __ldg(p.turn_row_off) <= r0;
    const int64_t k0 = ok ? warp_upper_le(p.turn_row_off, 0, p.n_turns - 1, r0, lane) : 0;
    if (lane == 0) s_first[0] = ok ? k0 : -1;
  } else if (warp == 1) {
    const bool ok = __ldg(p.traj_row_off) <= r0;
    const int64_t i0 = ok ? warp_upper_le(p.traj_row_off, 0, p.n_traj - 1, r0, lane) : 0;
    if (lane == 0) s_first[1] = ok ? i0 : -1;
  }
  __syncthreads();
  const int64_t k0 = s_first[0], i0 = s_first[1];
  if (k0 >= 0 && i0 >= 0) {
    for (int j = tid; j <= TILE; j += TILE) {
      s_turn_off[j] = __ldg(p.turn_row_off + min(k0 + j, (int64_t)p.n_turns));
      s_traj_row[j] = __ldg(p.traj_row_off + min(i0 + j, (int64_t)p.n_traj));
      s_traj_turn[j] = __ldg(p.traj_turn_off + min(i0 + j, (int64_t)p.n_traj));
    }
  }
  __syncthreads();

  __shared__ TileElem s_caggs[CLUSTER ? kClusterMaxTiles : 1];  // (CLUSTER) predecessors' aggregates

  // 2. this thread's row: its turn and trajectory, and its element
  RowMeta meta;
  meta.bad = true;
  meta.traj = 0;
  meta.turn = 0;
  meta.local_turn = 0;
  meta.traj_start = meta.traj_end = meta.turn_start = meta.turn_end = 0;
  if (live && k0 >= 0 && i0 >= 0) {
    const int nk = (int)min((int64_t)TILE, (int64_t)p.n_turns - k0);
    const int j = smem_upper_le(s_turn_off, nk, r);
    const int ni = (int)min((int64_t)TILE, (int64_t)p.n_traj - i0);
    int q = smem_upper_le(s_traj_row, ni, r);
    int64_t traj = i0 + q, tr_start = s_traj_row[q], tr_end = s_traj_row[q + 1];
    int64_t tu0 = s_traj_turn[q], tu1 = s_traj_turn[q + 1];
    if (r >= tr_end && q == ni - 1 && i0 + ni < p.n_traj) {
      // past the staged trajectories (more than TILE empty ones
      // in the tile's rows): search the rest in global memory
      int64_t lo = i0 + ni, hi = p.n_traj - 1;
      while (lo < hi) {
        const int64_t mid = (lo + hi + 1) >> 1;
        if (__ldg(p.traj_row_off + mid) <= r) lo = mid; else hi = mid - 1;
      }
      traj = lo;
      tr_start = __ldg(p.traj_row_off + traj);
      tr_end = __ldg(p.traj_row_off + traj + 1);
      tu0 = __ldg(p.traj_turn_off + traj);
      tu1 = __ldg(p.traj_turn_off + traj + 1);
    }
    const int64_t turn = k0 + j;
    meta.turn = (int32_t)turn;
    meta.traj = (int32_t)traj;
    meta.turn_start = s_turn_off[j];
    meta.turn_end = s_turn_off[j + 1];
    meta.local_turn = (int32_t)(turn - tu0);
    meta.traj_start = tr_start;
    meta.traj_end = tr_end;
    meta.bad = !(meta.turn_start <= r && r < meta.turn_end) || !(tr_start <= r && r < tr_end) ||
               !(tu0 <= turn && turn < tu1);
  }
  // a seeded row's carried state, and lambda, before the wait
  const bool seeded = live && ((w == 0) || (r == meta.traj_start) || meta.bad);
  const int fturn = (live && r == meta.turn_start) ? 1 : 0;
  double cum0 = 0.0, st0 = 0.0, sd0 = 0.0, sl0 = 0.0;
  if (seeded && !meta.bad) {
    const stride_scan_state* sp = p.state + meta.traj;
    cum0 = __ldcg(&sp->cum);
    st0 = fturn ? 0.0 : __ldcg(&sp->turn_sum_t);
    sd0 = fturn ? 0.0 : __ldcg(&sp->turn_sum_d);
    sl0 = fturn ? 0.0 : __ldcg(&sp->turn_sum_l);
  }
  const float lam = (live && !meta.bad) ? (p.lambda ? __ldg(p.lambda + meta.traj) : p.lambda_all) : 0.f;
  if (CLUSTER) cluster_arrive_release();  // this CTA's reads of the carried state are done
  if (!by_ticket) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    if (live) {
      lps = __ldcg(logp_s + w);
      lpt = __ldcg(logp_t + w);
    }
  }
  TileElem x = {0.0, 0.0, 0.0, 0.0, 0};
  double c_before = 0.0, st_before = 0.0, ri_c = 0.0;
  float st_before_f = 0.f, e_sl = 0.f;
  if (live) {
    const float nan = __int_as_float(0x7fc00000);
    if (meta.bad) {
      set_status(p.dev_status, STRIDE_DEV_BAD_LAYOUT);
      lps = nan;
      lpt = nan;
      if (p.out.logp_s) p.out.logp_s[w] = nan;  // a bad row's log-probs are NaN
      if (p.out.logp_t) p.out.logp_t[w] = nan;
    }
    const float dd = lps - lpt;
    if (p.out.opd) p.out.opd[w] = dd;
    const int64_t n_k = meta.turn_end - meta.turn_start;
    // The row's terms in fp32 (logp_S * d rounded once, as the fp64 product
    // of two floats rounded to float would be); the stop-sum term in fp64,
    // a turn mean's share lpt / n_k rounded once to fp32 first (GB300 issues
    // an fp64 divide as a sequence of fp64 operations at 1/64 of the fp32
    // rate; the rounding is 6e-8 of the term).
    const float esl = lps * dd;
    const double ec =
        (p.mode == STRIDE_STOP_TURN_MEAN) ? (double)(lpt / (float)(n_k > 0 ? n_k : 1)) : (double)lpt;
    e_sl = esl;
    if (p.profile && !meta.bad) {
      const int jb = (int)((10 * (r - meta.turn_start)) / n_k);  // Observation 1 decile
      atomicAdd(s_prof + 3 * jb + 0, (double)dd);
      atomicAdd(s_prof + 3 * jb + 1, (double)lpt);
      atomicAdd(s_prof + 3 * jb + 2, 1.0);
    }
    if (seeded && !meta.bad) {
      x = TileElem{cum0 + ec, (float)(st0 + (double)lpt), (float)(sd0 + (double)dd), (float)(sl0 + (double)esl),
                   kRestartSum | kRestartTurn};
      c_before = cum0;
      st_before = st0;
      st_before_f = (float)st0;
    } else if (seeded) {
      x = TileElem{ec, lpt, dd, esl, kRestartSum | kRestartTurn};  // NaN: nothing after a bad row is meaningful
    } else {
      x = TileElem{ec, lpt, dd, esl, fturn ? kRestartTurn : 0};
    }
    if (seeded) x.flags |= 4;  // bit 2: this row's exclusive prefix is the carried state, not the scan
  }

  // 3. segmented inclusive scan over the tile
  const TileElem tile_id = {0.0, 0.f, 0.f, 0.f, 0};
  TileElem tile_incl, tile_excl;
  block_scan<kWarps>(x, tile_id, lane, warp, s_wtot, s_wpre, tile_incl, tile_excl);

  // 4. the tile's exclusive prefix: from the cluster's other tiles (CLUSTER),
  //    else publish the tile's aggregate, fold predecessors, publish its prefix
  if (CLUSTER) {
    namespace cg = cooperative_groups;
    if (tid == (int)(n_here - 1)) s_agg = tile_incl;
    __syncthreads();
    cluster_wait_acquire();  // every tile has started and read its carried state
    if (warp == 0) {
      const cg::cluster_group cl = cg::this_cluster();
      const TileElem agg = s_agg;
      for (int64_t j = tile + 1 + lane; j < n_tiles; j += 32) cl.map_shared_rank(s_caggs, (unsigned)j)[tile] = agg;
    }
    cluster_arrive_release();
    cluster_wait_acquire();  // every aggregate has arrived; nothing touches this CTA's memory after
    if (warp == 0) {
      // the predecessors' aggregates folded in tile order (a warp scan: the
      // stop sum fp64, the open-turn sums fp32 as inside a tile)
      TileElem v = {0.0, 0.f, 0.f, 0.f, 0};
      if (lane < tile) v = s_caggs[lane];
#pragma unroll
      for (int d = 1; d < kClusterMaxTiles; d <<= 1) {
        const TileElem o = tile_shfl_up(v, d);
        if (lane >= d) v = tile_combine(o, v);
      }
      if (lane == (tile > 0 ? (int)tile - 1 : 0)) {
        s_excl = tile > 0 ? TileElem{v.c, v.st, v.sd, v.sl, 0} : TileElem{0.0, 0.f, 0.f, 0.f, 0};
        s_flags = 0;
      }
    }
    __syncthreads();
  } else {
    if (tid == (int)(n_here - 1)) {
      ScanElem agg{tile_incl.c, tile_incl.st, tile_incl.sd, tile_incl.sl, tile_incl.flags & kRestartTurn};
      if (tile_incl.flags & kRestartSum) {
        publish(p.incl + tile, p.flags + tile * kFlagStride, agg, kStIncl);
      } else {
        publish(p.agg + tile, p.flags + tile * kFlagStride, agg,
                kStAgg | ((tile_incl.flags & kRestartTurn) ? kFlagTurnStart : 0u));
      }
      s_agg = tile_incl;  // the aggregate, for warp 0 below
    }
    __syncthreads();
    if (warp == 0) {
      const TileElem agg = s_agg;
      PreElem pre = {0.0, 0.0, 0.0, 0.0};
      bool timed_out = false;
      // The rows before the tile's first seeded row need the predecessors' sum
      // (a tile whose first row is seeded needs nothing).
      if (!(__shfl_sync(0xffffffffu, x.flags, 0) & kRestartSum)) {
        const ScanElem e = lookback(p, tile, lane, timed_out);
        pre = PreElem{e.c, e.st, e.sd, e.sl};
        if (lane == 0 && !(agg.flags & kRestartSum)) {
          const PreElem inc = pre_combine(pre, agg);
          ScanElem ie{inc.c, inc.st, inc.sd, inc.sl, 1};
          publish(p.incl + tile, p.flags + tile * kFlagStride, ie, kStIncl);
        }
      }
      if (lane == 0) {
        s_excl = TileElem{pre.c, (float)pre.st, (float)pre.sd, (float)pre.sl, 0};
        s_flags = timed_out ? 1 : 0;
      }
    }
    __syncthreads();
  }

  // 5. complete every row
  if (live) {
    // the row's prefixes: the stop sum fp64, the open-turn sums fp32 (the
    // tile's prefix rounded once to fp32; 6e-8 of the sums)
    const TileElem pre = s_excl;
    const TileElem ri = tile_combine(pre, tile_incl);
    if (!(x.flags & 4)) {
      const TileElem re = tile_combine(pre, tile_excl);
      c_before = re.c;
      st_before_f = fturn ? 0.f : re.st;
      st_before = (double)st_before_f;
    }
    RowCarry rc;
    rc.e = ScanElem{0.0, 0.0, 0.0, (double)e_sl, fturn};
    const ScanElem si{ri.c, (double)ri.st, (double)ri.sd, (double)ri.sl, 1};
    row_tail(p, r, meta, rc, si, c_before, st_before, (s_flags & 1) != 0, true);
    ri_c = ri.c;
  }

  // 6. the trajectories' stop records and losses, once per trajectory and
  //    tile: the first row of a trajectory here that crosses lambda records
  //    the stop (the running sum never rises, so it is the trajectory's
  //    first crossing unless an earlier tile's is lower), and the last row
  //    of a trajectory here adds its retained rows' loss and count.
  TrajElem te = {0.f, 0, 0, 1};
  bool cross = false;
  if (live && !meta.bad) {
    const int64_t n_k = meta.turn_end - meta.turn_start;
    const bool turn_last = (r == meta.turn_end - 1);
    const bool test = (p.mode == STRIDE_STOP_TOKEN_SUM) || turn_last;
    cross = test && ri_c < (double)lam;
    // retained unless the rule fired before the row (row_tail); a
    // trajectory's first token or turn always is
    const bool first = (p.mode == STRIDE_STOP_TOKEN_SUM) ? (r == meta.traj_start) : (meta.local_turn == 0);
    const double before =
        (p.mode == STRIDE_STOP_TOKEN_SUM) ? c_before : c_before - (double)(st_before_f / (float)n_k);
    const bool kept = first || !(before < (double)lam);
    te = TrajElem{kept ? e_sl : 0.f, kept ? 1 : 0, cross ? 1 : 0, r == meta.traj_start ? 1 : 0};
  }
  const TrajElem traj_id = {0.f, 0, 0, 0};
  TrajElem t_incl, t_excl;
  block_scan<kWarps>(te, traj_id, lane, warp, s_ttot, s_tpre, t_incl, t_excl);
  if (live && !meta.bad) {
    stride_scan_state* sp = p.state + meta.traj;
    if (cross && (te.restart || !t_excl.crossed)) {
      atomicMin(reinterpret_cast<unsigned long long*>(&sp->stop_row), (unsigned long long)(r - meta.traj_start));
      atomicMin(reinterpret_cast<unsigned int*>(&sp->stop_turn), (unsigned int)meta.local_turn);
      sp->stopped = 1;
    }
    if ((r == meta.traj_end - 1 || tid == (int)(n_here - 1)) && t_incl.count > 0) {
      atomicAdd(&sp->loss, t_incl.loss);
      atomicAdd(reinterpret_cast<unsigned long long*>(&sp->loss_tokens), (unsigned long long)t_incl.count);
    }
  }
  if (p.profile) {
    __syncthreads();
    if (tid < 3 * STRIDE_PROFILE_BINS && s_prof[tid] != 0.0) atomicAdd(p.profile + tid, s_prof[tid]);
  }

  // Layout checks, spread over every thread of the launch (off the path of
  // the scan: nothing above waits for them), unless the kernel that wrote
  // the log-probs made them.
  if (!validate) return;
  bool bad = false;
  const int64_t stride = n_tiles * TILE;
  for (int64_t k = t0 + tid; k < p.n_turns; k += stride)
    bad |= __ldg(p.turn_row_off + k + 1) <= __ldg(p.turn_row_off + k);
  for (int64_t i = t0 + tid; i < p.n_traj; i += stride) {
    const int32_t a = __ldg(p.traj_turn_off + i), b = __ldg(p.traj_turn_off + i + 1);
    if (a < 0 || b < a || b > p.n_turns) {
      bad = true;
    } else {
      bad |= __ldg(p.turn_row_off + a) != __ldg(p.traj_row_off + i);
      bad |= __ldg(p.turn_row_off + b) != __ldg(p.traj_row_off + i + 1);
    }
  }
  if (bad) set_status(p.dev_status, STRIDE_DEV_BAD_LAYOUT);
}

cudaError_t launch_partial_lse(const void* S, const void* T, int dtype, bool vec, int64_t ld,
                               int32_t V_shard, int64_t col0, const int32_t* tokens, int64_t rows,
                               float* partials, int32_t* dev_status, cudaStream_t stream) {
  PartialParams p{S, T, ld, V_shard, col0, 0, tokens, rows, partials, dev_status};
  const dim3 grid((unsigned)rows), block(kPartialThreads);
  if (dtype == STRIDE_DTYPE_BF16) {
    if (vec)
      partial_lse_kernel<__nv_bfloat16, true><<<grid, block, 0, stream>>>(p);
    else
      partial_lse_kernel<__nv_bfloat16, false><<<grid, block, 0, stream>>>(p);
  } else {
    if (vec)
      partial_lse_kernel<float, true><<<grid, block, 0, stream>>>(p);
    else
      partial_lse_kernel<float, false><<<grid, block, 0, stream>>>(p);
  }
  return cudaGetLastError();
}

cudaError_t launch_combine_partials(const float* parts, int32_t n_shards, int64_t rows, float* logp_s,
                                    float* logp_t, float* lse_s, float* lse_t, int32_t* dev_status,
                                    cudaStream_t stream) {
  combine_kernel<<<(unsigned)((rows + 255) / 256), 256, 0, stream>>>(parts, n_shards, rows, logp_s, logp_t,
                                                                    lse_s, lse_t, dev_status);
  return cudaGetLastError();
}

// Whether one cluster of n CTAs of the cluster form can be placed on this
// device (looked up once per device and size; sizes above 8 need the
// non-portable cluster attribute, set here first).
bool scan_cluster_fits(int dev, int n, cudaStream_t stream) {
  constexpr int kMaxDev = 64;
  static std::atomic<int> fits[kMaxDev][kClusterMaxTiles + 1];  // 0 unknown, 1 yes, 2 no
  if (dev < 0 || dev >= kMaxDev || n < 1 || n > kClusterMaxTiles) return false;
  const int known = fits[dev][n].load(std::memory_order_acquire);
  if (known) return known == 1;
  auto kern = scan_logprobs_tile_kernel<kScanTileRowsDependent, true>;
  bool ok = true;
  if (n > 8) ok = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) == cudaSuccess;
  if (ok) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)n);
    cfg.blockDim = dim3(kScanTileRowsDependent);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)n;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    ok = cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg) == cudaSuccess && clusters >= 1;
  }
  if (!ok) (void)cudaGetLastError();  // a refused size is an answer, not an error to carry
  fits[dev][n].store(ok ? 1 : 2, std::memory_order_release);
  return ok;
}

cudaError_t launch_scan_logprobs(const BatchParams& p, const float* logp_s, const float* logp_t,
                                 cudaStream_t stream, bool dependent) {
  // (the small-window path's split kernel cleared the flags of its tiles)
  const int tile_rows = dependent ? kScanTileRowsDependent : kScanTileRows;
  const int64_t n_tiles = (p.n_rows + tile_rows - 1) / tile_rows;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)n_tiles);
  cfg.blockDim = dim3((unsigned)tile_rows);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  // the small-window kernel checks the layout itself (dependent launches)
  const bool validate = !dependent;
  // A dependent grid of at most one CTA per SM is resident at once (the
  // kernel it waits on always completes), so its tiles may go by block
  // index: no ticket, and the layout is read before the wait.
  int dev = 0;
  cudaError_t qe = cudaSuccess;
  const int sms = current_device_sms(&dev, &qe);
  if (sms <= 0) return qe != cudaSuccess ? qe : cudaErrorInvalidDevice;
  const bool by_ticket = !dependent || n_tiles > sms;
  // a small dependent window runs as one cluster (the cluster form)
  const bool cluster = dependent && !by_ticket && n_tiles <= kClusterMaxTiles &&
                       scan_cluster_fits(dev, (int)n_tiles, stream);
  if (cluster) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = (unsigned)n_tiles;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
  }
  const cudaError_t e =
      !dependent ? cudaLaunchKernelEx(&cfg, scan_logprobs_tile_kernel<kScanTileRows, false>, p, logp_s, logp_t,
                                      n_tiles, validate, by_ticket)
      : cluster  ? cudaLaunchKernelEx(&cfg, scan_logprobs_tile_kernel<kScanTileRowsDependent, true>, p, logp_s,
                                      logp_t, n_tiles, validate, by_ticket)
                 : cudaLaunchKernelEx(&cfg, scan_logprobs_tile_kernel<kScanTileRowsDependent, false>, p, logp_s,
                                      logp_t, n_tiles, validate, by_ticket);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace stride
