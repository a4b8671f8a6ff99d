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
// (scan_logprobs_kernel), one warp per row with the same decoupled-lookback
// protocol as the fused kernels (row_scan.cuh).
#include <math.h>

#include "row_scan.cuh"
#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

namespace stride {

constexpr int kPartialThreads = 256;
constexpr int kPartialWarps = kPartialThreads / 32;

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
__global__ void __launch_bounds__(kPartialThreads) partial_lse_kernel(const PartialParams p) {
  __shared__ float s_red[4][kPartialWarps];
  const int64_t r = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const LT* srow = reinterpret_cast<const LT*>(p.S) + r * p.ld;
  const LT* trow = reinterpret_cast<const LT*>(p.T) + r * p.ld;
  float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
  stream_pair<LT, VEC, 4>(srow, trow, 0, p.V_shard, tid, kPartialThreads, mS, sS, mT, sT);
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

// One warp per row, rows taken in ticket order: trajectory/turn lookup, the
// row's element (from the given log-probs), the lookback and the row tail.
constexpr int kScanWarpsPerCta = 8;
__global__ void __launch_bounds__(32 * kScanWarpsPerCta) scan_logprobs_kernel(const BatchParams p,
                                                                             const float* logp_s,
                                                                             const float* logp_t) {
  const int lane = threadIdx.x & 31;
  uint32_t t = 0;
  if (lane == 0) t = atomicAdd(p.ticket, 1u);
  t = __shfl_sync(0xffffffffu, t, 0);
  if ((int64_t)t >= p.n_rows) return;
  const int64_t tile = t;
  const int64_t r = p.row_begin + tile;
  float ls = 0.f, lt = 0.f;
  if (lane == 0) {
    ls = __ldg(logp_s + tile);
    lt = __ldg(logp_t + tile);
    validate_layout(p, tile);
  }
  const RowMeta meta = find_row_meta(p, r, lane);
  RowCarry rc;
  if (lane == 0) rc = row_finalize(p, tile, r, meta, true, ls, lt, 0.f, 0.f, p.profile, true);
  row_resolve(p, tile, r, meta, rc, lane);
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

cudaError_t launch_scan_logprobs(const BatchParams& p, const float* logp_s, const float* logp_t,
                                 cudaStream_t stream) {
  const unsigned grid = (unsigned)((p.n_rows + kScanWarpsPerCta - 1) / kScanWarpsPerCta);
  scan_logprobs_kernel<<<grid, 32 * kScanWarpsPerCta, 0, stream>>>(p, logp_s, logp_t);
  return cudaGetLastError();
}

}  // namespace stride
