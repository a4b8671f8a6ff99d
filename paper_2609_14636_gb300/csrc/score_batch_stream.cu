// score_batch_stream.cu -- persistent, warp-specialised batch scoring kernel
// for 16-byte-aligned rows (sm_103a).
//
// One CTA per SM runs until the window's rows are exhausted.  Its warps have
// fixed roles:
//
//   warp 0, producer   takes row tickets (atomicAdd, so rows are processed in
//                      ticket order) and streams each row's student and
//                      teacher logits, chunk by chunk, into a ring of
//                      kStages shared-memory stages with 1-D bulk async copies
//                      (cp.async.bulk ... mbarrier::complete_tx).  The ring
//                      keeps kStages x 2 x kChunk bytes in flight per SM
//                      without spending registers on them.
//   warps 6..21,       read each stage from shared memory into single-pass
//   consumers          online log-sum-exp pairs (stride_device.cuh), release
//                      the stage, and at a row's last chunk merge their pairs
//                      for the row warp.
//   warp 1, row warp   per row, while the row streams: trajectory/turn lookup,
//                      token, gathered logits, the ragged tail (V mod 8
//                      logits); once the row's pairs land: log-probs, outputs,
//                      and the row's scan element published at once
//                      (row_finalize).  It never waits on another CTA, so
//                      every row's AGGREGATE appears as soon as the row is
//                      scored, which keeps every lookback short.
//   warps 2..5, scan   rows taken round-robin (row n by scan warp n mod 4):
//                      the decoupled lookback, the INCLUSIVE publication,
//                      turn statistics, stop test and carried state
//                      (row_resolve).  Four lookbacks can be in flight per
//                      SM, and the scan warps may lag the row warp by up to
//                      kSlots rows without stalling the stream.
//
// Hand-offs inside the CTA use mbarriers only (no named barriers): full/empty
// per stage, and per row slot (kSlots rows in flight) start / red_done /
// lse_ready / agg_ready / slot_free.  Every wait is bounded by a
// %globaltimer budget; on expiry the CTA sets STRIDE_DEV_TIMEOUT, stops
// issuing, waits (bounded) for the copies it has in flight, and returns.
#include <math.h>

#include <atomic>

#include "mbarrier.cuh"
#include "row_scan.cuh"
#include "stride.h"
#include "stride_device.cuh"
#include "stride_internal.h"

// Ring shape: 3 stages of 32 KB per tensor (192 KB in flight per SM).  A
// sweep on GB300 over stages x chunk bytes at up to 218 KB of ring (the
// batch-scoring workload, two boxes, alternating runs) put 3 x 32 KB 0.4-
// 0.5 % ahead of 6 x 16 KB and 3 x 36 KB level with it; 2 x 48 KB, 4 x 27 KB,
// 5 x 20 KB and 8 x 12 KB were slower, 12 x 8 KB 14 % slower.
#ifndef STRIDE_BULK_STAGES
#define STRIDE_BULK_STAGES 3
#endif
#ifndef STRIDE_BULK_CHUNK
#define STRIDE_BULK_CHUNK 32768
#endif
#ifndef STRIDE_BULK_EVICT_FIRST
#define STRIDE_BULK_EVICT_FIRST 1
#endif

namespace stride {

constexpr int kStages = STRIDE_BULK_STAGES;   // ring depth
constexpr int kChunk = STRIDE_BULK_CHUNK;     // bytes per tensor per stage
constexpr int kSlots = 8;                     // rows in flight per CTA
constexpr int kConsumerWarps = 16;
constexpr int kConsumers = kConsumerWarps * 32;
constexpr int kScanWarps = 4;
constexpr int kFirstConsumerWarp = 2 + kScanWarps;
constexpr int kStreamThreads = 32 * kFirstConsumerWarp + kConsumers;
constexpr int kInfoEnd = -1;
constexpr int kInfoLast = 1 << 16;
static_assert(kChunk % 16 == 0, "bulk copies move multiples of 16 bytes");

struct alignas(128) StreamShared {
  uint64_t full[kStages];
  uint64_t empty[kStages];
  uint64_t start[kSlots];
  uint64_t lse_ready[kSlots];
  uint64_t slot_free[kSlots];
  uint64_t red_done[kSlots];
  uint64_t agg_ready[kSlots];
  int32_t stage_info[kStages];
  uint32_t stage_bytes[kStages];
  int64_t slot_tile[kSlots];
  float slot_pair[kSlots][4];
  float red[kSlots][kConsumerWarps][4];
  RowMeta slot_meta[kSlots];
  RowCarry slot_carry[kSlots];
  double prof[3 * STRIDE_PROFILE_BINS];  // this CTA's within-turn profile (row warp only)
  int64_t end_seq;  // first row sequence number without a row (set by the row warp)
  int32_t abort;
};

constexpr size_t kStreamHeader = (sizeof(StreamShared) + 127) & ~size_t(127);
constexpr size_t kStreamSmem = kStreamHeader + 2 * (size_t)kStages * kChunk;
static_assert(kStreamSmem <= 227 * 1024, "ring and header exceed the shared memory of one CTA");

__device__ __forceinline__ void raise_abort(StreamShared& sh, const BatchParams& p) {
  *reinterpret_cast<volatile int32_t*>(&sh.abort) = 1;
  set_status(p.dev_status, STRIDE_DEV_TIMEOUT);
}

template <typename LT>
__global__ void __launch_bounds__(kStreamThreads, 1) score_batch_stream_kernel(const BatchParams p) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  StreamShared& sh = *reinterpret_cast<StreamShared*>(smem_raw);
  unsigned char* bufS = smem_raw + kStreamHeader;
  unsigned char* bufT = bufS + (size_t)kStages * kChunk;
  volatile int32_t* abort = &sh.abort;

  constexpr int P = LogitTraits<LT>::kPerVec;
  const int tid = threadIdx.x;
  const int lane = tid & 31;
  const int warp = tid >> 5;
  const int v_body = p.V / P;  // 16-byte vectors per row streamed by bulk copies
  const uint32_t row_bytes = (uint32_t)v_body * 16u;
  const int n_chunks = (int)((row_bytes + kChunk - 1) / kChunk);
  const uint64_t tmo = p.timeout_ns;

  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&sh.full[s], 1);
      mbar_init(&sh.empty[s], kConsumerWarps);
    }
    for (int q = 0; q < kSlots; ++q) {
      mbar_init(&sh.start[q], 1);
      mbar_init(&sh.lse_ready[q], 1);
      mbar_init(&sh.slot_free[q], 1);
      mbar_init(&sh.red_done[q], kConsumerWarps);
      mbar_init(&sh.agg_ready[q], 1);
    }
    sh.abort = 0;
    sh.end_seq = INT64_MAX;
    for (int i = 0; i < 3 * STRIDE_PROFILE_BINS; ++i) sh.prof[i] = 0.0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  // Launched as a programmatic dependent of the workspace clear: the set-up
  // above may overlap the previous kernel's end; nothing global is touched
  // before the clear (and everything before it) has completed.  Dependents
  // may be scheduled at once: they wait for this grid in turn.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      uint64_t policy;
#if STRIDE_BULK_EVICT_FIRST
      asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
#else
      asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(policy));
#endif
      uint32_t it = 0;  // stages issued
      int64_t seq = 0;  // rows started by this CTA
      bool ok = true;
      while (ok) {
        const int q = (int)(seq % kSlots);
        const uint32_t use = (uint32_t)(seq / kSlots);
        if (use > 0 && !mbar_wait(&sh.slot_free[q], (use - 1) & 1u, tmo, abort)) {
          ok = false;
          break;
        }
        const uint32_t t = atomicAdd(p.ticket, 1u);
        const bool done = (int64_t)t >= p.n_rows;
        sh.slot_tile[q] = done ? -1 : (int64_t)t;
        mbar_arrive(&sh.start[q]);
        if (done) break;
        const unsigned char* srow = reinterpret_cast<const unsigned char*>(p.S) + (int64_t)t * p.ld * sizeof(LT);
        const unsigned char* trow = reinterpret_cast<const unsigned char*>(teacher_row<LT>(p, (int64_t)t));
        for (int c = 0; c < n_chunks; ++c) {
          const int s = (int)(it % kStages);
          const uint32_t k = it / kStages;
          if (k > 0 && !mbar_wait(&sh.empty[s], (k - 1) & 1u, tmo, abort)) {
            ok = false;
            break;
          }
          const uint32_t off = (uint32_t)c * kChunk;
          const uint32_t bytes = min((uint32_t)kChunk, row_bytes - off);
          sh.stage_info[s] = q | (c == n_chunks - 1 ? kInfoLast : 0);
          sh.stage_bytes[s] = bytes;
          mbar_arrive_expect_tx(&sh.full[s], 2u * bytes);
          bulk_g2s(bufS + (size_t)s * kChunk, srow + off, bytes, &sh.full[s], policy);
          bulk_g2s(bufT + (size_t)s * kChunk, trow + off, bytes, &sh.full[s], policy);
          ++it;
        }
        ++seq;
      }
      if (ok) {
        // end marker for the consumers in the next stage
        const int s = (int)(it % kStages);
        const uint32_t k = it / kStages;
        if (k == 0 || mbar_wait(&sh.empty[s], (k - 1) & 1u, tmo, abort)) {
          sh.stage_info[s] = kInfoEnd;
          sh.stage_bytes[s] = 0;
          mbar_arrive(&sh.full[s]);
        } else {
          ok = false;
        }
      }
      if (!ok) {
        raise_abort(sh, p);
        // wait (bounded) for the last copies issued into each stage
        for (int s = 0; s < kStages; ++s) {
          const uint32_t uses = it / kStages + ((uint32_t)s < it % kStages ? 1u : 0u);
          if (uses > 0) {
            const uint64_t t0 = globaltimer_ns();
            while (!mbar_try_wait(&sh.full[s], (uses - 1) & 1u) && globaltimer_ns() - t0 < tmo) {
            }
          }
        }
      }
    }
    return;
  }

  if (warp >= kFirstConsumerWarp) {
    // ----------------------------------------------------------- consumers
    const int cw = warp - kFirstConsumerWarp;
    const int ct = tid - 32 * kFirstConsumerWarp;
    uint32_t it = 0;
    int64_t seq = 0;  // rows finished, in the producer's order
    float mS = kMaxStart, sS = 0.f, mT = kMaxStart, sT = 0.f;
    while (true) {
      const int s = (int)(it % kStages);
      const uint32_t k = it / kStages;
      if (!mbar_wait_warp(&sh.full[s], k & 1u, tmo, abort)) {
        raise_abort(sh, p);
        break;
      }
      const int info = sh.stage_info[s];
      if (info == kInfoEnd) break;
      const int nvec = (int)(sh.stage_bytes[s] >> 4);
      const uint4* vs = reinterpret_cast<const uint4*>(bufS + (size_t)s * kChunk);
      const uint4* vt = reinterpret_cast<const uint4*>(bufT + (size_t)s * kChunk);
      int v = ct;
      for (; v + kConsumers < nvec; v += 2 * kConsumers) {
        const uint4 a[2] = {vs[v], vs[v + kConsumers]};
        const uint4 b[2] = {vt[v], vt[v + kConsumers]};
        LogitTraits<LT>::template chunk<2>(a, mS, sS);
        LogitTraits<LT>::template chunk<2>(b, mT, sT);
      }
      for (; v < nvec; v += kConsumers) {
        const uint4 a[1] = {vs[v]};
        const uint4 b[1] = {vt[v]};
        LogitTraits<LT>::template chunk<1>(a, mS, sS);
        LogitTraits<LT>::template chunk<1>(b, mT, sT);
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sh.empty[s]);
      ++it;
      if (info & kInfoLast) {
        // Row end: each warp posts its pair under the row's slot; warp 0
        // merges them once all 16 have arrived.  red[q] is reused only after
        // the scan warp has released slot q, which follows warp 0's read.
        const int q = info & 0xffff;
        const uint32_t use = (uint32_t)(seq / kSlots);
        warp_merge2(mS, sS, mT, sT);
        if (lane == 0) {
          sh.red[q][cw][0] = mS;
          sh.red[q][cw][1] = sS;
          sh.red[q][cw][2] = mT;
          sh.red[q][cw][3] = sT;
          mbar_arrive(&sh.red_done[q]);
        }
        if (cw == 0) {
          if (!mbar_wait_warp(&sh.red_done[q], use & 1u, tmo, abort)) {
            raise_abort(sh, p);
            break;
          }
          mS = lane < kConsumerWarps ? sh.red[q][lane][0] : kMaxStart;
          sS = lane < kConsumerWarps ? sh.red[q][lane][1] : 0.f;
          mT = lane < kConsumerWarps ? sh.red[q][lane][2] : kMaxStart;
          sT = lane < kConsumerWarps ? sh.red[q][lane][3] : 0.f;
          warp_merge2(mS, sS, mT, sT);
          if (lane == 0) {
            sh.slot_pair[q][0] = mS;
            sh.slot_pair[q][1] = sS;
            sh.slot_pair[q][2] = mT;
            sh.slot_pair[q][3] = sT;
            mbar_arrive(&sh.lse_ready[q]);
          }
        }
        ++seq;
        mS = kMaxStart;
        sS = 0.f;
        mT = kMaxStart;
        sT = 0.f;
      }
    }
    return;
  }

  if (warp == 1) {
    // ------------------------------------------------------------ row warp
    int64_t seq = 0;
    const float nan = __int_as_float(0x7fc00000);
    while (true) {
      const int q = (int)(seq % kSlots);
      const uint32_t use = (uint32_t)(seq / kSlots);
      if (!mbar_wait_warp(&sh.start[q], use & 1u, tmo, abort)) {
        if (lane == 0) raise_abort(sh, p);
        break;
      }
      const int64_t tile = sh.slot_tile[q];
      if (tile < 0) {
        __syncwarp();
        if (lane == 0) {
          *reinterpret_cast<volatile int64_t*>(&sh.end_seq) = seq;  // every scan warp stops here
          mbar_arrive(&sh.agg_ready[q]);
        }
        break;
      }
      const int64_t r = p.row_begin + tile;
      const LT* srow = reinterpret_cast<const LT*>(p.S) + tile * p.ld;
      const LT* trow = teacher_row<LT>(p, tile);
      int32_t y = 0;
      float xs = nan, xt = nan;
      if (lane == 0) {
        y = __ldg(p.tokens + tile);
        if (y >= 0 && y < p.V) {
          xs = to_f32(srow[y]);
          xt = to_f32(trow[y]);
        }
        validate_layout(p, tile);
      }
      const RowMeta meta = find_row_meta(p, r, lane);
      // ragged tail: the logits past the last whole 16-byte vector
      float tmS = kMaxStart, tsS = 0.f, tmT = kMaxStart, tsT = 0.f;
      for (int j = v_body * P + lane; j < p.V; j += 32) {
        lse_one(to_f32(srow[j]), tmS, tsS);
        lse_one(to_f32(trow[j]), tmT, tsT);
      }
      warp_merge2(tmS, tsS, tmT, tsT);
      if (!mbar_wait_warp(&sh.lse_ready[q], use & 1u, tmo, abort)) {
        if (lane == 0) raise_abort(sh, p);
        break;
      }
      float mS = sh.slot_pair[q][0], sS = sh.slot_pair[q][1];
      float mT = sh.slot_pair[q][2], sT = sh.slot_pair[q][3];
      lse_merge(mS, sS, tmS, tsS);
      lse_merge(mT, sT, tmT, tsT);
      if (lane == 0) {
        sh.slot_carry[q] = row_finalize(p, tile, r, meta, y >= 0 && y < p.V, xs, xt, lse_finish(mS, sS),
                                        lse_finish(mT, sT), p.profile ? sh.prof : nullptr, false);
        sh.slot_meta[q] = meta;
        mbar_arrive(&sh.agg_ready[q]);
      }
      __syncwarp();
      ++seq;
    }
    if (lane == 0 && p.profile) {
      for (int i = 0; i < 3 * STRIDE_PROFILE_BINS; ++i)
        if (sh.prof[i] != 0.0) atomicAdd(p.profile + i, sh.prof[i]);
    }
    return;
  }

  // --------------------------------------------------------------- scan warps
  volatile int64_t* end_seq = &sh.end_seq;
  for (int64_t seq = warp - 2;; seq += kScanWarps) {
    const int q = (int)(seq % kSlots);
    const uint32_t use = (uint32_t)(seq / kSlots);
    // Wait for row `seq`, unless the rows ran out before it.  The slots
    // past the last row never fill, so the wait polls (test_wait and a short
    // sleep) and looks at the end marker in between: a blocking try_wait
    // kept each scan warp suspended about 7.5 us after the row warp had
    // marked the end (probe timeline of 16,384-row windows: every CTA left
    // 7.4-7.7 us after its scan warps began their last wait).
    if (*end_seq <= seq) break;
    bool ready = mbar_test_wait(&sh.agg_ready[q], use & 1u);
    if (!ready) {
      const uint64_t t0 = globaltimer_ns();
      while (!(ready = mbar_test_wait(&sh.agg_ready[q], use & 1u))) {
        __nanosleep(100);
        if (*end_seq <= seq || *abort) break;
        if (globaltimer_ns() - t0 > tmo) {
          if (lane == 0) raise_abort(sh, p);
          break;
        }
      }
    }
    // the warp leaves together (lanes whose waits ended differently agree)
    ready = __all_sync(0xffffffffu, ready);
    if (!ready) break;
    const int64_t tile = sh.slot_tile[q];
    if (tile < 0) break;
    const RowMeta meta = sh.slot_meta[q];
    const RowCarry rc = sh.slot_carry[q];
    row_resolve(p, tile, p.row_begin + tile, meta, rc, lane);
    __syncwarp();
    if (lane == 0) mbar_arrive(&sh.slot_free[q]);
  }
}

size_t stream_smem_bytes() { return kStreamSmem; }

cudaError_t launch_score_batch_stream(const BatchParams& p, int dtype, cudaStream_t stream) {
  // The dynamic shared-memory limit is a per-device function attribute: set
  // once per device and dtype (setting it again is harmless, so two threads
  // racing here both succeed).
  static std::atomic<bool> attr_done[64][2];
  int dev = 0;
  cudaError_t e = cudaSuccess;
  const int sms = current_device_sms(&dev, &e);
  if (sms <= 0) return e != cudaSuccess ? e : cudaErrorInvalidDevice;
  const int di = dtype == STRIDE_DTYPE_BF16 ? 0 : 1;
  if (!attr_done[dev][di].load(std::memory_order_acquire)) {
    e = dtype == STRIDE_DTYPE_BF16
            ? cudaFuncSetAttribute(score_batch_stream_kernel<__nv_bfloat16>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kStreamSmem)
            : cudaFuncSetAttribute(score_batch_stream_kernel<float>,
                                   cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kStreamSmem);
    if (e != cudaSuccess) return e;
    attr_done[dev][di].store(true, std::memory_order_release);
  }
  const int64_t grid = p.n_rows < sms ? p.n_rows : sms;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kStreamThreads);
  cfg.dynamicSmemBytes = kStreamSmem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = dtype == STRIDE_DTYPE_BF16 ? cudaLaunchKernelEx(&cfg, score_batch_stream_kernel<__nv_bfloat16>, p)
                                 : cudaLaunchKernelEx(&cfg, score_batch_stream_kernel<float>, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace stride
