// Register-staged scan of one chunk of a vocabulary row.
//
// A row of V logits is split across the C CTAs of a thread-block cluster;
// CTA c owns elements [c0, c1).  Each of the 256 threads issues all of its
// 16-byte loads up front (8 vectors: 64 bf16 or 32 fp32 elements), so one
// CTA keeps 32 KB of reads in flight and the whole grid saturates HBM with a
// single pass.  Element (i, j) of a thread is vector i, lane j, at row
// position c0 + (i * 256 + threadIdx.x) * VW + j: positions increase with
// (i, j), so "first in scan order" is "lowest token id".  Positions past c1
// are loaded as -inf, which no max, exp or threshold test can pick.
//
// The per-element work is kept to what the math needs: the thread max uses
// packed bf16x2 max (half an instruction per element), the exp-sum is taken
// relative to the thread's own max (no block barrier in between), and
// positions are only materialised for the few elements that can win.
#pragma once

#include "common.cuh"

namespace tg {

constexpr int kScanThreads = 256;
constexpr int kScanVecs = 8;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

template <typename T>
struct ScanTraits;
template <>
struct ScanTraits<__nv_bfloat16> {
  static constexpr int kVW = 8;  // elements per 16-byte vector
  static constexpr uint32_t kNegInfWord = 0xFF80FF80u;
};
template <>
struct ScanTraits<float> {
  static constexpr int kVW = 4;
  static constexpr uint32_t kNegInfWord = 0xFF800000u;
};

template <typename T>
constexpr int scan_elems_per_cta() {
  return kScanThreads * kScanVecs * ScanTraits<T>::kVW;
}

__device__ __forceinline__ uint32_t vec_word(const uint4& v, int w) {
  return w == 0 ? v.x : (w == 1 ? v.y : (w == 2 ? v.z : v.w));
}

// element j (compile-time after unrolling) of a 16-byte vector
template <typename T>
__device__ __forceinline__ float vec_elem(const uint4& v, int j);
template <>
__device__ __forceinline__ float vec_elem<__nv_bfloat16>(const uint4& v, int j) {
  const uint32_t w = vec_word(v, j >> 1);
  return (j & 1) ? bf16_hi(w) : bf16_lo(w);
}
template <>
__device__ __forceinline__ float vec_elem<float>(const uint4& v, int j) {
  return __uint_as_float(vec_word(v, j));
}

__device__ __forceinline__ int scan_pos(int c0, int i, int j, int vw) {
  return c0 + (i * kScanThreads + (int)threadIdx.x) * vw + j;
}

// One 16-byte vector at an edge of the chunk: elements [pos, pos + VW) that
// lie below c1 are read one by one, the rest read as -inf.  A rolled loop:
// only the threads at a chunk edge run it, and it stays small in the
// instruction cache.
template <typename T>
__device__ __forceinline__ uint4 load_edge_vec(const T* __restrict__ row, int pos, int c1) {
  constexpr int VW = ScanTraits<T>::kVW;
  constexpr int EB = 16 / VW * 8;  // bits per element
  uint64_t val[2] = {0ull, 0ull}, got[2] = {0ull, 0ull};
#pragma unroll 1
  for (int j = 0; j < VW; ++j) {
    if (pos + j < c1) {
      uint64_t x;
      if constexpr (VW == 8) x = reinterpret_cast<const uint16_t*>(row)[pos + j];
      else x = reinterpret_cast<const uint32_t*>(row)[pos + j];
      const int half = j / (VW / 2), sh = EB * (j % (VW / 2));
      const uint64_t fm = (EB == 64 ? ~0ull : ((1ull << EB) - 1ull)) << sh;
      if (half) { val[1] |= x << sh; got[1] |= fm; } else { val[0] |= x << sh; got[0] |= fm; }
    }
  }
  const uint64_t neg = (uint64_t)ScanTraits<T>::kNegInfWord * 0x100000001ull;
  const uint64_t lo = val[0] | (neg & ~got[0]), hi = val[1] | (neg & ~got[1]);
  return make_uint4((uint32_t)lo, (uint32_t)(lo >> 32), (uint32_t)hi, (uint32_t)(hi >> 32));
}

// Load this thread's elements of [c0, c1); positions past c1 read as -inf.
// kAligned: the row start is 16-byte aligned (c0 is a multiple of VW).
// Whole vectors take one 16-byte load each; the few vectors that straddle
// c1 (or every vector of an unaligned row) are filled afterwards by one
// rolled fix-up loop, which keeps the unrolled fast path small.
template <typename T, bool kAligned>
__device__ __forceinline__ void scan_load(const T* __restrict__ row, int c0, int c1,
                                          uint4 (&buf)[kScanVecs]) {
  constexpr int VW = ScanTraits<T>::kVW;
  constexpr uint32_t kNeg = ScanTraits<T>::kNegInfWord;
  uint32_t partial = 0;  // vectors that start below c1 but are not loaded whole
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i) {
    const int pos = scan_pos(c0, i, 0, VW);
    if (kAligned && pos + VW <= c1) {
      buf[i] = ld_stream_v4(row + pos);
    } else {
      buf[i] = make_uint4(kNeg, kNeg, kNeg, kNeg);
      if (pos < c1) partial |= 1u << i;
    }
  }
  while (partial) {
    const int i = __ffs(partial) - 1;
    partial &= partial - 1;
    const uint4 v = load_edge_vec<T>(row, scan_pos(c0, i, 0, VW), c1);
#pragma unroll
    for (int j = 0; j < kScanVecs; ++j)
      if (i == j) buf[j] = v;
  }
}

// vector i of the thread's buffer for a run-time i (a select chain: keeps
// the buffer in registers)
__device__ __forceinline__ uint4 buf_vec(const uint4 (&buf)[kScanVecs], int i) {
  uint4 q = buf[0];
#pragma unroll
  for (int j = 1; j < kScanVecs; ++j)
    if (i == j) q = buf[j];
  return q;
}

// value of element (i, j) of a thread's chunk read back from global memory
// (rare paths re-read instead of holding code for every register slot)
template <typename T>
__device__ __forceinline__ float load_elem(const T* __restrict__ row, int pos) {
  if constexpr (ScanTraits<T>::kVW == 8)
    return __uint_as_float((uint32_t)reinterpret_cast<const uint16_t*>(row)[pos] << 16);
  else
    return reinterpret_cast<const float*>(row)[pos];
}

// Largest element of this thread (-inf if it has none).
template <typename T>
__device__ __forceinline__ float scan_thread_max(const uint4 (&buf)[kScanVecs]);
template <>
__device__ __forceinline__ float scan_thread_max<__nv_bfloat16>(const uint4 (&buf)[kScanVecs]) {
  __nv_bfloat162 m[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    uint32_t x = vec_word(buf[0], w);
    m[w] = *reinterpret_cast<__nv_bfloat162*>(&x);
  }
#pragma unroll
  for (int i = 1; i < kScanVecs; ++i)
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      uint32_t x = vec_word(buf[i], w);
      m[w] = __hmax2(m[w], *reinterpret_cast<__nv_bfloat162*>(&x));
    }
  const __nv_bfloat162 a = __hmax2(__hmax2(m[0], m[1]), __hmax2(m[2], m[3]));
  return fmaxf(__low2float(a), __high2float(a));
}
template <>
__device__ __forceinline__ float scan_thread_max<float>(const uint4 (&buf)[kScanVecs]) {
  float m = __uint_as_float(buf[0].x);
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) m = fmaxf(m, __uint_as_float(vec_word(buf[i], j)));
  return m;
}

// elements 2w, 2w+1 of a 16-byte vector as a float pair
template <typename T>
__device__ __forceinline__ float2 vec_pair(const uint4& v, int w);
template <>
__device__ __forceinline__ float2 vec_pair<__nv_bfloat16>(const uint4& v, int w) {
  const uint32_t x = vec_word(v, w);
  return make_float2(bf16_lo(x), bf16_hi(x));
}
template <>
__device__ __forceinline__ float2 vec_pair<float>(const uint4& v, int w) {
  return make_float2(__uint_as_float(vec_word(v, 2 * w)), __uint_as_float(vec_word(v, 2 * w + 1)));
}

// sum_t 2^((x_t - m) * log2 e) over this thread's elements, m = its max, on
// the MUFU unit (one ex2 per element; after the load the scan kernels are
// bound by latency, not by MUFU throughput, and a share of polynomial
// exponentials on the FMA pipe measured slower)
template <typename T>
__device__ __forceinline__ float scan_thread_sumexp(const uint4 (&buf)[kScanVecs], float m) {
  if (m == __int_as_float(0xff800000)) return 0.f;
  constexpr int VW = ScanTraits<T>::kVW;
  const float mb = -m * kLog2e;
  const float2 l2e = make_float2(kLog2e, kLog2e), nb = make_float2(mb, mb);
  float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
    for (int w = 0; w < VW / 2; ++w) {
      const float2 y = __ffma2_rn(vec_pair<T>(buf[i], w), l2e, nb);
      const float2 e = make_float2(ex2(y.x), ex2(y.y));
      if (i & 1) acc1 = __fadd2_rn(acc1, e); else acc0 = __fadd2_rn(acc0, e);
    }
  return (acc0.x + acc0.y) + (acc1.x + acc1.y);
}

// Lowest position in [c0, c1) whose value equals v (INT_MAX if none).
// Positions grow in scan order (vector, then lane), so the first match in
// that order is the lowest; a match at or past c1 means none below c1.
template <typename T>
__device__ __forceinline__ int scan_first_pos(const uint4 (&buf)[kScanVecs], int c0, int c1,
                                              float v);
template <>
__device__ __forceinline__ int scan_first_pos<float>(const uint4 (&buf)[kScanVecs], int c0, int c1,
                                                     float v) {
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (vec_elem<float>(buf[i], j) == v) {
        const int pos = scan_pos(c0, i, j, 4);
        return pos < c1 ? pos : 0x7FFFFFFF;
      }
  return 0x7FFFFFFF;
}
template <>
__device__ __forceinline__ int scan_first_pos<__nv_bfloat16>(const uint4 (&buf)[kScanVecs], int c0,
                                                             int c1, float v) {
  // v is an element value, so it is exact in bf16: one packed compare per pair
  const __nv_bfloat162 v2 = __float2bfloat162_rn(v);
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const uint32_t x = vec_word(buf[i], w);
      const uint32_t mk = __heq2_mask(*reinterpret_cast<const __nv_bfloat162*>(&x), v2);
      if (mk) {
        const int pos = scan_pos(c0, i, 2 * w, 8) + ((mk & 0xFFFFu) ? 0 : 1);
        return pos < c1 ? pos : 0x7FFFFFFF;
      }
    }
  return 0x7FFFFFFF;
}

// Combine two (max, sum of 2^(x - max)) pairs.
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  const float NEG_INF = __int_as_float(0xff800000);
  const float M = fmaxf(m, m2);
  if (M == NEG_INF) {
    m = M;
    s = 0.f;
    return;
  }
  s = (m == NEG_INF ? 0.f : s * ex2((m - M) * kLog2e)) +
      (m2 == NEG_INF ? 0.f : s2 * ex2((m2 - M) * kLog2e));
  m = M;
}

}  // namespace tg
