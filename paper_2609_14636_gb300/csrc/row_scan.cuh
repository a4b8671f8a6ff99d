// row_scan.cuh -- the per-row tail of the batch scoring kernels: the row's
// log-probs and outputs, its element of the decoupled-lookback segmented
// scan, turn statistics, the stop test and the carried state.
//
// The running stop sum is a plain prefix sum over rows of a per-row term:
//   TOKEN_SUM (Sec. 5.5):   term = log pi_T(y_t)
//   TURN_MEAN (Eq. 4-5):    term = log pi_T(y_t) / n_k   (n_k = turn length)
// so that at a turn's last row the prefix equals sum_{j<=k} l_j exactly in
// real arithmetic; the stop test is applied at every row (TOKEN_SUM) or at
// turn-end rows only (TURN_MEAN).  Because every term is <= 0 the prefix is
// non-increasing, so the smallest crossing row is the first crossing.
//
// Scan protocol.  Tile t (= row row_begin + t, tiles numbered in ticket
// order) publishes its own row's element as an AGGREGATE as soon as its row
// is scored, then folds predecessors' published elements (32 at a time, by
// one warp) back to the nearest INCLUSIVE prefix, then publishes its
// INCLUSIVE prefix.  A tile that starts a trajectory, and tile 0 of the
// window, seed their inclusive prefix from the trajectory's carried state and
// publish it at once, so every lookback ends inside its own trajectory.
// Tickets are taken with atomicAdd, so every predecessor a warp waits on is
// held by a running CTA that publishes its aggregate without waiting on any
// later tile: the spin always ends.  It is bounded anyway (timeout_ns,
// globaltimer): on expiry the kernel sets STRIDE_DEV_TIMEOUT and finishes
// without the missing terms.
#pragma once

#include <math.h>

#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace stride {

constexpr uint32_t kStAgg = 1u;
constexpr uint32_t kStIncl = 2u;
constexpr uint32_t kStMask = 3u;
constexpr uint32_t kFlagTurnStart = 4u;
constexpr uint32_t kFlagTimedOut = 8u;

struct ScanElem {
  double c;   // running stop-sum terms
  double st;  // sum of log pi_T within the open turn
  double sd;  // sum of d within the open turn
  double sl;  // sum of the OPD-loss terms logp_S * d within the open turn
  int fturn;  // the range contains a turn's first row
};

// a (earlier rows) (+) b (later rows).  c never resets inside a lookback
// (trajectory starts publish inclusive prefixes); st, sd and sl restart at a
// turn's first row.
__device__ __forceinline__ ScanElem combine(const ScanElem& a, const ScanElem& b) {
  ScanElem r;
  r.c = a.c + b.c;
  r.st = b.fturn ? b.st : a.st + b.st;
  r.sd = b.fturn ? b.sd : a.sd + b.sd;
  r.sl = b.fturn ? b.sl : a.sl + b.sl;
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
  slot->sl = e.sl;
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
static __device__ ScanElem lookback(const BatchParams& p, int64_t tile, int lane, bool& timed_out) {
  ScanElem excl = {0.0, 0.0, 0.0, 0.0, 0};
  int64_t j = tile - 1;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    const int64_t idx = j - lane;
    uint32_t f = kStIncl;  // before row 0: never folded (tile 0 is inclusive)
    bool valid = idx >= 0;
    if (valid) {
      f = ld_acquire_u32(p.flags + idx * kFlagStride);
      while ((f & kStMask) == 0u) {
        if (globaltimer_ns() - t0 > p.timeout_ns) {
          f = kStIncl | kFlagTimedOut;
          break;
        }
        __nanosleep(64);
        f = ld_acquire_u32(p.flags + idx * kFlagStride);
      }
    }
    const bool is_incl = (f & kStMask) == kStIncl;
    const unsigned inc = __ballot_sync(0xffffffffu, is_incl);
    const int stop = inc ? __ffs(inc) - 1 : 31;
    ScanElem v = {0.0, 0.0, 0.0, 0.0, 0};
    if (valid && lane <= stop && !(f & kFlagTimedOut)) {
      const ScanSlot* src = is_incl ? (p.incl + idx) : (p.agg + idx);
      const double2 a = __ldcg(reinterpret_cast<const double2*>(src));
      const double2 b = __ldcg(reinterpret_cast<const double2*>(src) + 1);
      v.c = a.x;
      v.st = a.y;
      v.sd = b.x;
      v.sl = b.y;
      v.fturn = (is_incl || (f & kFlagTurnStart)) ? 1 : 0;
    }
    if (f & kFlagTimedOut) timed_out = true;
    // Ordered fold of lanes stop..0 (lane l+d holds an earlier row than lane
    // l): a 5-step shuffle tree; lanes past `stop` hold the identity.
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      ScanElem o;
      o.c = __shfl_down_sync(0xffffffffu, v.c, d);
      o.st = __shfl_down_sync(0xffffffffu, v.st, d);
      o.sd = __shfl_down_sync(0xffffffffu, v.sd, d);
      o.sl = __shfl_down_sync(0xffffffffu, v.sl, d);
      o.fturn = __shfl_down_sync(0xffffffffu, v.fturn, d);
      if (lane + d < 32) v = combine(o, v);
    }
    ScanElem win;
    win.c = __shfl_sync(0xffffffffu, v.c, 0);
    win.st = __shfl_sync(0xffffffffu, v.st, 0);
    win.sd = __shfl_sync(0xffffffffu, v.sd, 0);
    win.sl = __shfl_sync(0xffffffffu, v.sl, 0);
    win.fturn = __shfl_sync(0xffffffffu, v.fturn, 0);
    excl = combine(win, excl);
    if (inc) break;
    j -= 32;
  }
  timed_out = __any_sync(0xffffffffu, timed_out);
  return excl;
}


// The part of a row's tail that waits on nobody: outputs, the row's scan
// element, the within-turn profile, and the element's publication (an
// AGGREGATE, or, for a tile that starts a trajectory or the window, the
// INCLUSIVE prefix seeded from the carried state).  Lane 0 only.  `prof`
// (30 doubles, or NULL) receives the profile: with atomics when it is the
// caller's global array, plainly when it is one writer's shared copy.
struct RowCarry {
  ScanElem e;
  ScanElem incl;      // valid for seeded tiles
  double c_before;    // running sum before this row (seeded tiles)
  double st_before;   // open-turn sum of log pi_T before this row (seeded tiles)
  int seeded;
};

__device__ __forceinline__ RowCarry row_finalize(const BatchParams& p, int64_t tile, int64_t r,
                                                 const RowMeta& meta, bool token_ok, float xs, float xt,
                                                 float lse_s, float lse_t, double* prof,
                                                 bool prof_atomic) {
  RowCarry rc;
  const int64_t n_k = meta.turn_end - meta.turn_start;
  const float nan = __int_as_float(0x7fc00000);
  float lps = xs - lse_s;
  float lpt = xt - lse_t;
  if (!token_ok) set_status(p.dev_status, STRIDE_DEV_TOKEN_RANGE);
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
  ScanElem e;
  e.c = (p.mode == STRIDE_STOP_TURN_MEAN) ? (double)lpt / (double)(n_k > 0 ? n_k : 1) : (double)lpt;
  e.st = (double)lpt;
  e.sd = (double)dd;
  e.sl = (double)lps * (double)dd;  // -log pi_S * r_t (Eq. 2)
  e.fturn = (r == meta.turn_start) ? 1 : 0;
  if (prof && !meta.bad) {
    const int j = (int)((10 * (r - meta.turn_start)) / n_k);  // Observation 1 decile
    if (prof_atomic) {
      atomicAdd(prof + 3 * j + 0, e.sd);
      atomicAdd(prof + 3 * j + 1, e.st);
      atomicAdd(prof + 3 * j + 2, 1.0);
    } else {
      prof[3 * j + 0] += e.sd;
      prof[3 * j + 1] += e.st;
      prof[3 * j + 2] += 1.0;
    }
  }
  rc.e = e;
  rc.seeded = (tile == 0) || (r == meta.traj_start) || meta.bad;
  rc.c_before = 0.0;
  rc.st_before = 0.0;
  if (rc.seeded) {
    if (meta.bad) {
      rc.incl = e;  // NaN terms; nothing downstream of a bad row is meaningful
    } else {
      const stride_scan_state* sp = p.state + meta.traj;
      const double cum0 = __ldcg(&sp->cum);
      const double st0 = __ldcg(&sp->turn_sum_t);
      const double sd0 = __ldcg(&sp->turn_sum_d);
      const double sl0 = __ldcg(&sp->turn_sum_l);
      rc.c_before = cum0;
      rc.st_before = e.fturn ? 0.0 : st0;
      rc.incl.c = cum0 + e.c;
      rc.incl.st = e.fturn ? e.st : st0 + e.st;
      rc.incl.sd = e.fturn ? e.sd : sd0 + e.sd;
      rc.incl.sl = e.fturn ? e.sl : sl0 + e.sl;
      rc.incl.fturn = 1;
    }
    publish(p.incl + tile, p.flags + tile * kFlagStride, rc.incl, kStIncl);
  } else {
    rc.incl = e;
    publish(p.agg + tile, p.flags + tile * kFlagStride, e, kStAgg | (e.fturn ? kFlagTurnStart : 0u));
  }
  return rc;
}

// The part that waits: the lookback (warp-wide) for an unseeded tile, the
// INCLUSIVE publication, then (lane 0) turn statistics, the stop test, the
// row's OPD-loss term if the row is retained, and the carried state.
//
// Retention: a row is retained when the stop rule has not fired before it.
// A trajectory's first token (token mode) or first turn (turn mode) always
// is: no test precedes it (with a prefix-buffer offset already below lambda
// that token or turn triggers the stop and is kept).  After it, in token
// mode that is "the running sum before the row is >= lambda"; in turn mode
// "the running sum through the previous turn is >= lambda", which is the
// running sum before the row minus the row's turn's terms so far
// (c_before - st_before / n_k).  The sums are monotone, so this selects
// exactly the rows up to the first crossing (its turn, in turn mode).
// rc is read in lane 0.
// row_tail is the single-thread part once the row's inclusive prefix is
// known: incl (running sum and open-turn sums through the row), c_before
// and st_before (the running sum and open turn's sum of log pi_T before it);
// of rc only rc.e.sl (the row's loss term) is read.  With defer_traj the
// trajectory's stop record and loss are left to the caller (the tiled scan
// aggregates them per trajectory and tile).
__device__ __forceinline__ void row_tail(const BatchParams& p, int64_t r, const RowMeta& meta,
                                         const RowCarry& rc, const ScanElem& incl, double c_before,
                                         double st_before, bool timed_out, bool defer_traj = false);

__device__ __forceinline__ void row_resolve(const BatchParams& p, int64_t tile, int64_t r,
                                            const RowMeta& meta, RowCarry rc, int lane) {
  const int seeded = __shfl_sync(0xffffffffu, rc.seeded, 0);
  ScanElem incl = rc.incl;
  double c_before = rc.c_before, st_before = rc.st_before;
  bool timed_out = false;
  if (!seeded) {
    const ScanElem excl = lookback(p, tile, lane, timed_out);
    if (lane == 0) {
      incl = combine(excl, rc.e);
      c_before = excl.c;
      st_before = rc.e.fturn ? 0.0 : excl.st;
      publish(p.incl + tile, p.flags + tile * kFlagStride, incl, kStIncl);
    }
  }
  if (lane != 0) return;
  row_tail(p, r, meta, rc, incl, c_before, st_before, timed_out);
}

__device__ __forceinline__ void row_tail(const BatchParams& p, int64_t r, const RowMeta& meta,
                                         const RowCarry& rc, const ScanElem& incl, double c_before,
                                         double st_before, bool timed_out, bool defer_traj) {
  if (timed_out) set_status(p.dev_status, STRIDE_DEV_TIMEOUT);
  if (meta.bad) return;
  const int64_t n_k = meta.turn_end - meta.turn_start;

  // ---- turn statistics, stop test, loss, carried state (lane 0) ---------
  const bool turn_last = (r == meta.turn_end - 1);
  if (turn_last && p.turn_stats) {
    stride_turn_stats ts;
    ts.sum_t = incl.st;
    ts.sum_d = incl.sd;
    ts.sum_l = incl.sl;
    ts.cum = incl.c;
    ts.mean_t = (float)(incl.st / (double)n_k);
    ts.n = (int32_t)n_k;
    p.turn_stats[meta.turn] = ts;
  }
  const bool test = (p.mode == STRIDE_STOP_TOKEN_SUM) || turn_last;
  const float lam = p.lambda ? __ldg(p.lambda + meta.traj) : p.lambda_all;
  stride_scan_state* sp = p.state + meta.traj;
  if (!defer_traj) {
    if (test && incl.c < (double)lam) {
      atomicMin(reinterpret_cast<unsigned long long*>(&sp->stop_row),
                (unsigned long long)(r - meta.traj_start));
      atomicMin(reinterpret_cast<unsigned int*>(&sp->stop_turn), (unsigned int)meta.local_turn);
      sp->stopped = 1;
    }
    const bool first = (p.mode == STRIDE_STOP_TOKEN_SUM) ? (r == meta.traj_start) : (meta.local_turn == 0);
    const double before = (p.mode == STRIDE_STOP_TOKEN_SUM) ? c_before : c_before - st_before / (double)n_k;
    if (first || !(before < (double)lam)) {  // the previous test did not fire (a NaN lambda never does)
      atomicAdd(&sp->loss, rc.e.sl);
      atomicAdd(reinterpret_cast<unsigned long long*>(&sp->loss_tokens), 1ull);
    }
  }
  if (r == meta.traj_end - 1 || r == p.row_end - 1) {
    sp->cum = incl.c;
    sp->turn_sum_t = turn_last ? 0.0 : incl.st;
    sp->turn_sum_d = turn_last ? 0.0 : incl.sd;
    sp->turn_sum_l = turn_last ? 0.0 : incl.sl;
    sp->rows_seen = r - meta.traj_start + 1;
    sp->turn_idx = turn_last ? meta.local_turn + 1 : meta.local_turn;
    sp->turn_tokens = turn_last ? 0 : (int32_t)(r - meta.turn_start + 1);
  }
}

// Warp-wide: everything a row needs once its two log-sum-exps are known.
// lse_s, lse_t and meta are valid in every lane; y, xs, xt in lane 0.
__device__ __forceinline__ void finish_row(const BatchParams& p, int64_t tile, int64_t r,
                                           const RowMeta& meta, int32_t y, float xs, float xt,
                                           float lse_s, float lse_t, int lane) {
  RowCarry rc;
  if (lane == 0) rc = row_finalize(p, tile, r, meta, y >= 0 && y < p.V, xs, xt, lse_s, lse_t, p.profile, true);
  row_resolve(p, tile, r, meta, rc, lane);
}

}  // namespace stride
