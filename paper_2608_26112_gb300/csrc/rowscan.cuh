// Register-staged scan of one chunk of a vocabulary row.
//
// A row of V logits is split across the C CTAs of a thread-block cluster;
// CTA c owns elements [c0, c1).  Each of the 256 threads issues all of its
// 16-byte loads up front (8 vectors: 64 bf16 or 32 fp32 elements), so one
// CTA keeps 32 KB of reads in flight and the whole grid saturates HBM with a
// single pass.  Element (i, j) of a thread is vector i, lane j, at row
// position c0 + (i * 256 + threadIdx.x) * VW + j: positions increase with
// (i, j), so "first in scan order" is "lowest token id".
#pragma once

#include "common.cuh"

namespace tg {

constexpr int kScanThreads = 256;
constexpr int kScanVecs = 8;

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

// Load this thread's elements of [c0, c1); positions past c1 read as -inf.
// kAligned: the row start is 16-byte aligned (c0 is a multiple of VW).
template <typename T, bool kAligned>
__device__ __forceinline__ void scan_load(const T* __restrict__ row, int c0, int c1,
                                          uint4 (&buf)[kScanVecs]) {
  constexpr int VW = ScanTraits<T>::kVW;
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i) {
    const int pos = c0 + (i * kScanThreads + (int)threadIdx.x) * VW;
    if (kAligned && pos + VW <= c1) {
      buf[i] = ld_stream_v4(row + pos);
    } else {
      uint32_t w[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) w[q] = ScanTraits<T>::kNegInfWord;
      if (pos < c1) {
        if constexpr (VW == 8) {
          const uint16_t* r16 = reinterpret_cast<const uint16_t*>(row);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (pos + j < c1) {
              const uint32_t h = r16[pos + j];
              w[j >> 1] = (j & 1) ? ((w[j >> 1] & 0x0000FFFFu) | (h << 16))
                                  : ((w[j >> 1] & 0xFFFF0000u) | h);
            }
          }
        } else {
          const uint32_t* r32 = reinterpret_cast<const uint32_t*>(row);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (pos + j < c1) w[j] = r32[pos + j];
        }
      }
      buf[i] = make_uint4(w[0], w[1], w[2], w[3]);
    }
  }
}

// Largest element of this thread and its lowest position (-inf elements
// count; a thread without elements returns pos = -1).
template <typename T>
__device__ __forceinline__ void scan_thread_max(const uint4 (&buf)[kScanVecs], int c0, int c1,
                                                float& vmax, int& pmax) {
  constexpr int VW = ScanTraits<T>::kVW;
  vmax = __int_as_float(0xff800000);
  pmax = -1;
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i) {
    const int base = c0 + (i * kScanThreads + (int)threadIdx.x) * VW;
#pragma unroll
    for (int j = 0; j < VW; ++j) {
      const float v = vec_elem<T>(buf[i], j);
      const int pos = base + j;
      if (pos < c1 && (pmax < 0 || v > vmax)) {
        vmax = v;
        pmax = pos;
      }
    }
  }
}

}  // namespace tg
