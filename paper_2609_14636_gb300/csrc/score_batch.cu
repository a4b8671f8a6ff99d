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
// The running stop sum is a plain prefix sum over rows of a per-row term:
//   TOKEN_SUM (Sec. 5.5):   term = log pi_T(y_t)
//   TURN_MEAN (Eq. 4-5):    term = log pi_T(y_t) / n_k   (n_k = turn length)
// so that at a turn's last row the prefix equals sum_{j<=k} l_j exactly in
// real arithmetic; the stop test is applied at every row (TOKEN_SUM) or at
// turn-end rows only (TURN_MEAN).  Because every term is <= 0 the prefix is
// non-increasing, so the smallest crossing row is the first crossing.
//
// Scan protocol.  Tile t (= row row_begin + t) publishes its own row's
// element as an AGGREGATE as soon as its row is scored, then folds
// predecessors' published elements (32 at a time, by one warp) back to the
// nearest INCLUSIVE prefix, then publishes its INCLUSIVE prefix.  A tile that
// starts a trajectory, and tile 0 of the window, seed their inclusive prefix
// from the trajectory's carried state and publish it at once, so every
// lookback ends inside its own trajectory.  Tickets are taken with atomicAdd,
// so every predecessor a CTA waits on has already started and publishes its
// aggregate without waiting on anyone: the spin always ends.  It is bounded
// anyway (timeout_ns, globaltimer): on expiry the kernel sets
// STRIDE_DEV_TIMEOUT and finishes without the missing terms.
#include <math.h>

#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace stride {

constexpr int kBatchThreads = 512;
constexpr int kBatchWarps = kBatchThreads / 32;
constexpr int kBatchUnroll = 4;

constexpr uint32_t kStAgg = 1u;
constexpr uint32_t kStIncl = 2u;
constexpr uint32_t kStMask = 3u;
constexpr uint32_t kFlagTurnStart = 4u;
constexpr uint32_t kFlagTimedOut = 8u;

struct ScanElem {
  double c;   // running stop-sum terms
  double st;  // sum of log pi_T within the open turn
  double sd;  // sum of d within the open turn
  int fturn;  // the range contains a turn's first row
};

// a (earlier rows) (+) b (later rows).  c never resets inside a lookback
// (trajectory starts publish inclusive prefixes); st and sd restart at a
// turn's first row.
__device__ __forceinline__ ScanElem combine(const ScanElem& a, const ScanElem& b) {
  ScanElem r;
  r.c = a.c + b.c;
  r.st = b.fturn ? b.st : a.st + b.st;
  r.sd = b.fturn ? b.sd : a.sd + b.sd;
  r.fturn = a.fturn | b.fturn;
  return r;
}

__device__ __forceinline__ uint32_t ld_acquire_u32(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_u32(uint32_t* p, uint32_t v) {
  asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void publish(ScanSlot* slot, uint32_t* flag, const ScanElem& e,
                                        uint32_t status) {
  slot->c = e.c;
  slot->st = e.st;
  slot->sd = e.sd;
  st_release_u32(flag, status);
}

// Largest i in [lo, hi] with off[i] <= r, given off[lo] <= r (warp-wide,
// 32 probes per step).  The result stays in [lo, hi] whatever off holds.
__device__ __forceinline__ int64_t warp_upper_le(const int64_t* __restrict__ off, int64_t lo,
                                                 int64_t hi, int64_t r, int lane) {
  while (hi > lo) {
    const int64_t step = (hi - lo + 31) / 32;
    const int64_t q = lo + step * (lane + 1);
    const bool ok = (q <= hi) && (__ldg(off + q) <= r);
    const int k = __popc(__ballot_sync(0xffffffffu, ok));
    const int64_t nlo = lo + step * k;
    const int64_t nhi = (k < 32) ? min(hi, lo + step * (k + 1) - 1) : hi;
    lo = nlo;
    hi = nhi;
  }
  return lo;
}

struct RowMeta {
  int64_t traj_start, traj_end, turn_start, turn_end;
  int32_t traj, turn, local_turn;
  bool bad;
};

__device__ __forceinline__ RowMeta find_row_meta(const BatchParams& p, int64_t r, int lane) {
  RowMeta m;
  m.bad = false;
  m.traj = 0;
  m.turn = 0;
  m.local_turn = 0;
  m.traj_start = m.traj_end = m.turn_start = m.turn_end = 0;
  if (__ldg(p.traj_row_off) > r) {
    m.bad = true;
    return m;
  }
  const int64_t traj = warp_upper_le(p.traj_row_off, 0, p.n_traj - 1, r, lane);
  m.traj = (int32_t)traj;
  m.traj_start = __ldg(p.traj_row_off + traj);
  m.traj_end = __ldg(p.traj_row_off + traj + 1);
  const int32_t k0 = __ldg(p.traj_turn_off + traj);
  const int32_t k1 = __ldg(p.traj_turn_off + traj + 1);
  if (!(m.traj_start <= r && r < m.traj_end) || k0 < 0 || k1 > p.n_turns || k1 <= k0) {
    m.bad = true;
    return m;
  }
  if (__ldg(p.turn_row_off + k0) > r) {
    m.bad = true;
    return m;
  }
  const int64_t turn = warp_upper_le(p.turn_row_off, k0, k1 - 1, r, lane);
  m.turn = (int32_t)turn;
  m.local_turn = (int32_t)(turn - k0);
  m.turn_start = __ldg(p.turn_row_off + turn);
  m.turn_end = __ldg(p.turn_row_off + turn + 1);
  if (!(m.turn_start <= r && r < m.turn_end)) m.bad = true;
  return m;
}

// Checks that the CTA owning ticket t makes on the layout arrays: every turn
// is non-empty, every trajectory's turns cover exactly its rows.
__device__ __forceinline__ void validate_layout(const BatchParams& p, int64_t t) {
  bool bad = false;
  for (int64_t k = t; k < p.n_turns; k += p.n_rows)
    bad |= __ldg(p.turn_row_off + k + 1) <= __ldg(p.turn_row_off + k);
  for (int64_t i = t; i < p.n_traj; i += p.n_rows) {
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

// Folds published predecessors of `tile` back to the nearest inclusive
// prefix.  Warp-wide; every lane returns the same exclusive prefix.
__device__ ScanElem lookback(const BatchParams& p, int64_t tile, int lane, bool& timed_out) {
  ScanElem excl = {0.0, 0.0, 0.0, 0};
  int64_t j = tile - 1;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    const int64_t idx = j - lane;
    uint32_t f = kStIncl;  // before row 0: never folded (tile 0 is inclusive)
    bool valid = idx >= 0;
    if (valid) {
      f = ld_acquire_u32(p.flags + idx);
      while ((f & kStMask) == 0u) {
        if (globaltimer_ns() - t0 > p.timeout_ns) {
          f = kStIncl | kFlagTimedOut;
          break;
        }
        __nanosleep(64);
        f = ld_acquire_u32(p.flags + idx);
      }
    }
    const bool is_incl = (f & kStMask) == kStIncl;
    const unsigned inc = __ballot_sync(0xffffffffu, is_incl);
    const int stop = inc ? __ffs(inc) - 1 : 31;
    ScanElem v = {0.0, 0.0, 0.0, 0};
    if (valid && lane <= stop && !(f & kFlagTimedOut)) {
      const ScanSlot* src = is_incl ? (p.incl + idx) : (p.agg + idx);
      const double2 a = __ldcg(reinterpret_cast<const double2*>(src));
      const double2 b = __ldcg(reinterpret_cast<const double2*>(src) + 1);
      v.c = a.x;
      v.st = a.y;
      v.sd = b.x;
      v.fturn = (is_incl || (f & kFlagTurnStart)) ? 1 : 0;
    }
    if (f & kFlagTimedOut) timed_out = true;
    ScanElem win = {0.0, 0.0, 0.0, 0};
    for (int l = stop; l >= 0; --l) {
      ScanElem x;
      x.c = __shfl_sync(0xffffffffu, v.c, l);
      x.st = __shfl_sync(0xffffffffu, v.st, l);
      x.sd = __shfl_sync(0xffffffffu, v.sd, l);
      x.fturn = __shfl_sync(0xffffffffu, v.fturn, l);
      win = combine(win, x);
    }
    excl = combine(win, excl);
    if (inc) break;
    j -= 32;
  }
  timed_out = __any_sync(0xffffffffu, timed_out);
  return excl;
}

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
  const LT* trow = reinterpret_cast<const LT*>(p.T) + tile * p.ld;

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

  // ---- per-row values (lane 0) ----------------------------------------
  const int64_t n_k = meta.turn_end - meta.turn_start;
  ScanElem e = {0.0, 0.0, 0.0, 0};
  if (lane == 0) {
    const float nan = __int_as_float(0x7fc00000);
    float lps = xs - lse_s;
    float lpt = xt - lse_t;
    if (!(y >= 0 && y < p.V)) set_status(p.dev_status, STRIDE_DEV_TOKEN_RANGE);
    if (meta.bad) {
      set_status(p.dev_status, STRIDE_DEV_BAD_LAYOUT);
      lps = nan;
      lpt = nan;
    }
    const float dd = lps - lpt;
    const stride_row_outputs& o = p.out;
    if (o.logp_s) o.logp_s[tile] = lps;
    if (o.logp_t) o.logp_t[tile] = lpt;
    if (o.opd) o.opd[tile] = dd;
    if (o.lse_s) o.lse_s[tile] = lse_s;
    if (o.lse_t) o.lse_t[tile] = lse_t;
    if (o.x_s) o.x_s[tile] = xs;
    if (o.x_t) o.x_t[tile] = xt;
    e.c = (p.mode == STRIDE_STOP_TURN_MEAN) ? (double)lpt / (double)(n_k > 0 ? n_k : 1) : (double)lpt;
    e.st = (double)lpt;
    e.sd = (double)dd;
    e.fturn = (r == meta.turn_start) ? 1 : 0;
  }

  // ---- segmented scan ---------------------------------------------------
  const bool seeded = (tile == 0) || (r == meta.traj_start) || meta.bad;
  ScanElem incl;
  bool timed_out = false;
  if (seeded) {
    if (lane == 0) {
      if (meta.bad) {
        incl = e;  // NaN terms; nothing downstream of a bad row is meaningful
      } else {
        const stride_scan_state* sp = p.state + meta.traj;
        const double cum0 = __ldcg(&sp->cum);
        const double st0 = __ldcg(&sp->turn_sum_t);
        const double sd0 = __ldcg(&sp->turn_sum_d);
        incl.c = cum0 + e.c;
        incl.st = e.fturn ? e.st : st0 + e.st;
        incl.sd = e.fturn ? e.sd : sd0 + e.sd;
        incl.fturn = 1;
      }
      publish(p.incl + tile, p.flags + tile, incl, kStIncl);
    }
  } else {
    if (lane == 0) publish(p.agg + tile, p.flags + tile, e, kStAgg | (e.fturn ? kFlagTurnStart : 0u));
    const ScanElem excl = lookback(p, tile, lane, timed_out);
    if (lane == 0) {
      incl = combine(excl, e);
      publish(p.incl + tile, p.flags + tile, incl, kStIncl);
    }
  }
  if (lane != 0) return;
  if (timed_out) set_status(p.dev_status, STRIDE_DEV_TIMEOUT);
  if (meta.bad) return;

  // ---- turn statistics, stop test, carried state (lane 0) ---------------
  const bool turn_last = (r == meta.turn_end - 1);
  if (turn_last && p.turn_stats) {
    stride_turn_stats ts;
    ts.sum_t = incl.st;
    ts.sum_d = incl.sd;
    ts.cum = incl.c;
    ts.mean_t = (float)(incl.st / (double)n_k);
    ts.n = (int32_t)n_k;
    p.turn_stats[meta.turn] = ts;
  }
  const bool test = (p.mode == STRIDE_STOP_TOKEN_SUM) || turn_last;
  const float lam = p.lambda ? __ldg(p.lambda + meta.traj) : p.lambda_all;
  stride_scan_state* sp = p.state + meta.traj;
  if (test && incl.c < (double)lam) {
    atomicMin(reinterpret_cast<unsigned long long*>(&sp->stop_row),
              (unsigned long long)(r - meta.traj_start));
    atomicMin(reinterpret_cast<unsigned int*>(&sp->stop_turn), (unsigned int)meta.local_turn);
    sp->stopped = 1;
  }
  if (r == meta.traj_end - 1 || r == p.row_end - 1) {
    sp->cum = incl.c;
    sp->turn_sum_t = turn_last ? 0.0 : incl.st;
    sp->turn_sum_d = turn_last ? 0.0 : incl.sd;
    sp->rows_seen = r - meta.traj_start + 1;
    sp->turn_idx = turn_last ? meta.local_turn + 1 : meta.local_turn;
    sp->turn_tokens = turn_last ? 0 : (int32_t)(r - meta.turn_start + 1);
  }
}

BatchWorkspaceLayout batch_workspace_layout(int64_t n_rows) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  BatchWorkspaceLayout L;
  const size_t n = n_rows > 0 ? (size_t)n_rows : 0;
  L.ticket_off = 0;
  L.flags_off = 256;
  L.agg_off = L.flags_off + up(n * sizeof(uint32_t));
  L.incl_off = L.agg_off + up(n * sizeof(ScanSlot));
  L.total = L.incl_off + up(n * sizeof(ScanSlot));
  L.clear_bytes = L.agg_off;  // ticket + flags
  if (n == 0) L.total = 0;
  return L;
}

cudaError_t launch_score_batch(const BatchParams& p, int dtype, bool vec, cudaStream_t stream) {
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
