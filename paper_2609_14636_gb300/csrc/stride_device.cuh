// stride_device.cuh -- device helpers shared by the STRIDE scoring kernels
// (sm_103a).  Streaming loads, bf16 unpacking, the single-pass online
// log-sum-exp, and (m, s) merges.
//
// Log-sum-exp convention: a running pair (m, s) stands for
//   LSE = m + ln(s),  s = sum_j 2^((x_j - m) * log2 e)
// m starts at kMaxStart, a finite value below any realistic logit, so that
// x - m is -inf (never NaN) for -inf entries, which contribute exactly 0.  A
// row whose largest logit is below kMaxStart is treated as fully masked
// (LSE = -inf).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace stride {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kMaxStart = -2.0e38f;

// 16-byte streaming load: read-only path, no L1 allocation (each logit byte
// is touched once), 256-byte L2 prefetch granule.
__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0,%1,%2,%3}, [%4];"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "l"(p));
  return v;
}

// 2^x on the SFU (PTX ex2.approx.ftz.f32: relative error ~2^-22, subnormal
// results flush to 0, 2^-inf = 0).
__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ __nv_bfloat162 as_bf162(uint32_t w) {
  __nv_bfloat162 h;
  *reinterpret_cast<uint32_t*>(&h) = w;
  return h;
}

__device__ __forceinline__ float to_f32(__nv_bfloat16 h) { return __bfloat162float(h); }
__device__ __forceinline__ float to_f32(float x) { return x; }

// Adds 2^((x - m) log2e) for a pair of logits to a packed accumulator.
// x - m is exact for bf16 inputs (and 0 for the maximum itself, so a row's
// largest logit contributes exactly 1); one rounding follows in the scale.
__device__ __forceinline__ float2 exp_pair_acc(float2 acc, float2 x, float2 nm) {
  const float2 l2 = make_float2(kLog2e, kLog2e);
  const float2 t = __fmul2_rn(__fadd2_rn(x, nm), l2);
  return __fadd2_rn(acc, make_float2(ex2(t.x), ex2(t.y)));
}

// One chunk of U 16-byte vectors of bf16 logits (8 per vector) into (m, s).
// The chunk maximum is taken on packed bf16x2 (exact), the running pair is
// rescaled at most once per chunk, and each element costs one unpack, half a
// packed subtract, half a packed multiply, one ex2 and half a packed add.
template <int U>
__device__ __forceinline__ void lse_chunk_bf16(const uint4 (&v)[U], float& m, float& s) {
  __nv_bfloat162 mx = __hmax2(as_bf162(v[0].x), as_bf162(v[0].y));
  mx = __hmax2(mx, __hmax2(as_bf162(v[0].z), as_bf162(v[0].w)));
#pragma unroll
  for (int u = 1; u < U; ++u) {
    mx = __hmax2(mx, __hmax2(as_bf162(v[u].x), as_bf162(v[u].y)));
    mx = __hmax2(mx, __hmax2(as_bf162(v[u].z), as_bf162(v[u].w)));
  }
  const float cm = fmaxf(__low2float(mx), __high2float(mx));
  if (cm > m) {
    s *= ex2((m - cm) * kLog2e);
    m = cm;
  }
  const float nmv = -m;
  const float2 nm = make_float2(nmv, nmv);
  float2 acc = make_float2(0.f, 0.f);
#pragma unroll
  for (int u = 0; u < U; ++u) {
    acc = exp_pair_acc(acc, make_float2(bf16_lo(v[u].x), bf16_hi(v[u].x)), nm);
    acc = exp_pair_acc(acc, make_float2(bf16_lo(v[u].y), bf16_hi(v[u].y)), nm);
    acc = exp_pair_acc(acc, make_float2(bf16_lo(v[u].z), bf16_hi(v[u].z)), nm);
    acc = exp_pair_acc(acc, make_float2(bf16_lo(v[u].w), bf16_hi(v[u].w)), nm);
  }
  s += acc.x + acc.y;
}

// Same for fp32 logits (4 per vector).
template <int U>
__device__ __forceinline__ void lse_chunk_f32(const uint4 (&v)[U], float& m, float& s) {
  float cm = fmaxf(fmaxf(__uint_as_float(v[0].x), __uint_as_float(v[0].y)),
                   fmaxf(__uint_as_float(v[0].z), __uint_as_float(v[0].w)));
#pragma unroll
  for (int u = 1; u < U; ++u) {
    cm = fmaxf(cm, fmaxf(fmaxf(__uint_as_float(v[u].x), __uint_as_float(v[u].y)),
                         fmaxf(__uint_as_float(v[u].z), __uint_as_float(v[u].w))));
  }
  if (cm > m) {
    s *= ex2((m - cm) * kLog2e);
    m = cm;
  }
  const float nmv = -m;
  const float2 nm = make_float2(nmv, nmv);
  float2 acc = make_float2(0.f, 0.f);
#pragma unroll
  for (int u = 0; u < U; ++u) {
    acc = exp_pair_acc(acc, make_float2(__uint_as_float(v[u].x), __uint_as_float(v[u].y)), nm);
    acc = exp_pair_acc(acc, make_float2(__uint_as_float(v[u].z), __uint_as_float(v[u].w)), nm);
  }
  s += acc.x + acc.y;
}

// A single logit into (m, s).
__device__ __forceinline__ void lse_one(float x, float& m, float& s) {
  if (x > m) {
    s *= ex2((m - x) * kLog2e);
    m = x;
  }
  s += ex2((x - m) * kLog2e);
}

// (m, s) <- (m, s) (+) (m2, s2): the pair for the union of both element sets.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float M = fmaxf(m, m2);
  s = s * ex2((m - M) * kLog2e) + s2 * ex2((m2 - M) * kLog2e);
  m = M;
}

__device__ __forceinline__ float lse_finish(float m, float s) { return m + logf(s); }

template <typename LT>
struct LogitTraits;
template <>
struct LogitTraits<__nv_bfloat16> {
  static constexpr int kPerVec = 8;
  template <int U>
  __device__ __forceinline__ static void chunk(const uint4 (&v)[U], float& m, float& s) {
    lse_chunk_bf16<U>(v, m, s);
  }
};
template <>
struct LogitTraits<float> {
  static constexpr int kPerVec = 4;
  template <int U>
  __device__ __forceinline__ static void chunk(const uint4 (&v)[U], float& m, float& s) {
    lse_chunk_f32<U>(v, m, s);
  }
};

// Streams logit columns [c0, c1) of one student row and one teacher row
// (both read once, interleaved) into two running pairs.  VEC requires both
// row pointers 16-byte aligned and c0, c1 multiples of kPerVec, except that
// c1 may equal the row length V (the ragged tail is read with scalar loads).
// Threads tid = 0..nthreads-1 of the caller share the range.
template <typename LT, bool VEC, int U>
__device__ __forceinline__ void stream_pair(const LT* __restrict__ srow, const LT* __restrict__ trow,
                                            int c0, int c1, int tid, int nthreads, float& mS,
                                            float& sS, float& mT, float& sT) {
  constexpr int P = LogitTraits<LT>::kPerVec;
  if (VEC) {
    const uint4* sv = reinterpret_cast<const uint4*>(srow);
    const uint4* tv = reinterpret_cast<const uint4*>(trow);
    const int v0 = c0 / P;
    const int v1 = c1 / P;  // full vectors end here
    int v = v0 + tid;
    for (; v + (U - 1) * nthreads < v1; v += U * nthreads) {
      uint4 a[U], b[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        a[u] = ld_stream(sv + v + u * nthreads);
        b[u] = ld_stream(tv + v + u * nthreads);
      }
      LogitTraits<LT>::template chunk<U>(a, mS, sS);
      LogitTraits<LT>::template chunk<U>(b, mT, sT);
    }
    for (; v < v1; v += nthreads) {
      uint4 a[1] = {ld_stream(sv + v)};
      uint4 b[1] = {ld_stream(tv + v)};
      LogitTraits<LT>::template chunk<1>(a, mS, sS);
      LogitTraits<LT>::template chunk<1>(b, mT, sT);
    }
    for (int j = v1 * P + tid; j < c1; j += nthreads) {
      lse_one(to_f32(srow[j]), mS, sS);
      lse_one(to_f32(trow[j]), mT, sT);
    }
  } else {
    // Rows that are not 16-byte aligned.  When S and T share the row's
    // misalignment (row stride and bases alike), the logits up to the next
    // 16-byte boundary are read one by one and the rest as 16-byte vectors,
    // then the ragged tail; otherwise every logit is read on its own.
    // (A typed pointer is element-aligned, so the distance to the boundary
    // is a whole number of elements.)
    const uintptr_t as = reinterpret_cast<uintptr_t>(srow + c0), at = reinterpret_cast<uintptr_t>(trow + c0);
    const bool same = ((as ^ at) & 15u) == 0;
    int head = c1 - c0;
    if (same) {
      const int h = (int)(((16u - (unsigned)(as & 15u)) & 15u) / sizeof(LT));
      head = h < head ? h : head;
    }
    for (int j = c0 + tid; j < c0 + head; j += nthreads) {
      lse_one(to_f32(srow[j]), mS, sS);
      lse_one(to_f32(trow[j]), mT, sT);
    }
    if (same && c0 + head < c1) {
      const LT* s2 = srow + c0 + head;  // 16-byte aligned
      const LT* t2 = trow + c0 + head;
      const int n2 = c1 - (c0 + head);
      const int nvec = n2 / P;
      const uint4* sv = reinterpret_cast<const uint4*>(s2);
      const uint4* tv = reinterpret_cast<const uint4*>(t2);
      int v = tid;
      for (; v + (U - 1) * nthreads < nvec; v += U * nthreads) {
        uint4 a[U], b[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          a[u] = ld_stream(sv + v + u * nthreads);
          b[u] = ld_stream(tv + v + u * nthreads);
        }
        LogitTraits<LT>::template chunk<U>(a, mS, sS);
        LogitTraits<LT>::template chunk<U>(b, mT, sT);
      }
      for (; v < nvec; v += nthreads) {
        uint4 a[1] = {ld_stream(sv + v)};
        uint4 b[1] = {ld_stream(tv + v)};
        LogitTraits<LT>::template chunk<1>(a, mS, sS);
        LogitTraits<LT>::template chunk<1>(b, mT, sT);
      }
      for (int j = nvec * P + tid; j < n2; j += nthreads) {
        lse_one(to_f32(s2[j]), mS, sS);
        lse_one(to_f32(t2[j]), mT, sT);
      }
    }
  }
}

// Warp-wide merge of two running pairs; every lane ends with the warp total
// (bit for bit the same in every lane: each butterfly step adds or takes the
// larger of the same two values).  The warp's largest m first, then each
// lane rescales its s to it once and the rescaled sums are added: two
// exponentials per lane instead of one per pair and step.
__device__ __forceinline__ void warp_merge2(float& mS, float& sS, float& mT, float& sT) {
  float MS = mS, MT = mT;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    MS = fmaxf(MS, __shfl_xor_sync(0xffffffffu, MS, o));
    MT = fmaxf(MT, __shfl_xor_sync(0xffffffffu, MT, o));
  }
  sS *= ex2((mS - MS) * kLog2e);
  sT *= ex2((mT - MT) * kLog2e);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sS += __shfl_xor_sync(0xffffffffu, sS, o);
    sT += __shfl_xor_sync(0xffffffffu, sT, o);
  }
  mS = MS;
  mT = MT;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
  return t;
}

// Cluster barrier halves (PTX barrier.cluster, executed by every thread of
// the CTA): a wait returns once all non-exited threads of the cluster have
// arrived.  Arriving at kernel start and waiting before the first remote
// shared-memory store guarantees the target CTA has started.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ void set_status(int32_t* dev_status, int bits) {
  if (dev_status) atomicOr(dev_status, bits);
}

}  // namespace stride
