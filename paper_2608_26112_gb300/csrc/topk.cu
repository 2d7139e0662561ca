// expand_topk: per-node log-softmax, exact top-k child tokens and cumulative
// path scores (Sec. 3.1 edge score p(u) and s(u) = s(v) p(u); Top_m of
// Algorithms 1 and 2), one HBM pass over the logits.
//
// Grid (C, rows) with clusters of C CTAs along x: the C CTAs of a cluster
// split one row.  Each CTA
//   1. stages its chunk in registers and takes per-thread (max, sum of
//      exp(x - max)) - packed bf16x2 max, one exp per element - merged per
//      warp with shuffles;
//   2. sorts the 256 thread maxima per warp; after one barrier each of the
//      top-k lanes of every warp counts, by binary search in the eight
//      sorted lists, how many maxima reach its own value, and the largest
//      value with a count >= k is the threshold t = the k-th largest thread
//      maximum.  At least k elements reach t, and only threads whose max
//      reaches t can hold elements that do, so candidates are collected by a
//      handful of threads only, which visit just the 16-byte vectors whose
//      packed max reaches t;
//   3. ranks the candidates by 64-bit keys (value desc, token asc - exact
//      on ties) by counting larger keys.  Heavily tied chunks can overflow
//      the candidate buffer; they fall back to an exact key threshold (the
//      k-th largest per-thread (max, first position) key), which bounds the
//      candidates by 64 * k;
//   4. the ranking threads store the chunk's top-k (descending) straight
//      into the cluster leader's shared memory (DSMEM), each warp adds its
//      (max, sum), and the cluster meets one barrier.
// In the leader every received key finds its row rank as its index in its
// own sorted list plus, by binary search, the number of larger keys in each
// other list; the k keys of rank < k write the outputs, and their warps fold
// the C * 8 (max, sum) pairs into the lse.  No global scratch and no second
// launch.
//
// These kernels are latency-bound, and several CTAs share an SM: the code
// keeps dependency chains short and the executed code small (rare paths are
// rolled loops), so the instruction cache holds the hot path.
#include <cooperative_groups.h>

#include "launch.h"
#include "rowscan.cuh"

namespace cg = cooperative_groups;

namespace tg {
namespace {

constexpr int kMaxK = 32;
constexpr int kCandMax = 2048;  // >= 64 elements/thread * kMaxK
constexpr int kMaxCluster = 16;
static_assert(kCandMax >= kScanVecs * 8 * kMaxK, "exact fallback must fit the buffer");

struct TopkSmem {
  uint64_t cand[kCandMax];
  uint64_t recv_top[kMaxCluster * kMaxK];  // leader only: each CTA's sorted top-k
  float recv_m[kMaxCluster * 8];           // leader only: each warp's (max, sum)
  float recv_s[kMaxCluster * 8];
  float warp_v[8 * 32];  // each warp's 32 thread maxima, sorted descending
  uint64_t warp_k[8 * kMaxK];
  uint64_t thr_key;
  uint32_t thr_ord;
  int ncand;
};

// Entries >= x in the eight descending 32-float lists L[w * 32 ..]: eight
// branch-free binary searches run in lockstep (5 halving steps and a final
// probe), so each step issues eight independent shared loads.
__device__ __forceinline__ int count_ge_8x32(const float* L, float x) {
  int pos[8];
#pragma unroll
  for (int w = 0; w < 8; ++w) pos[w] = 0;
#pragma unroll
  for (int step = 16; step > 0; step >>= 1)
#pragma unroll
    for (int w = 0; w < 8; ++w) pos[w] += (L[w * 32 + pos[w] + step - 1] >= x) ? step : 0;
  int cnt = 0;
#pragma unroll
  for (int w = 0; w < 8; ++w) cnt += pos[w] + ((L[w * 32 + pos[w]] >= x) ? 1 : 0);
  return cnt;
}

// Keys > x in the C descending lists of n <= 32 keys at L[c * n ..], list
// `skip` excluded: the C binary searches run in lockstep.
__device__ __forceinline__ int count_gt_lists(const uint64_t* L, int C, int n, int skip,
                                              uint64_t x) {
  int pos[kMaxCluster];
#pragma unroll
  for (int c = 0; c < kMaxCluster; ++c) pos[c] = 0;
#pragma unroll
  for (int step = 16; step > 0; step >>= 1)
#pragma unroll
    for (int c = 0; c < kMaxCluster; ++c) {
      const int i = pos[c] + step - 1;
      if (c < C && i < n && L[c * n + i] > x) pos[c] += step;
    }
  int cnt = 0;
#pragma unroll
  for (int c = 0; c < kMaxCluster; ++c)
    if (c < C && c != skip) cnt += pos[c] + ((pos[c] < n && L[c * n + pos[c]] > x) ? 1 : 0);
  return cnt;
}

// descending bitonic sort of one value per lane; lane j ends with the j-th largest
template <typename K>
__device__ __forceinline__ K warp_sort_desc(K x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const K y = __shfl_xor_sync(0xffffffffu, x, stride);
      const bool take_max = (((lane & stride) == 0) == ((lane & size) == 0));
      x = take_max ? (x > y ? x : y) : (x < y ? x : y);
    }
  }
  return x;
}

__device__ __forceinline__ void push_cand(TopkSmem& sm, uint64_t key) {
  const int slot = atomicAdd(&sm.ncand, 1);
  if (slot < kCandMax) sm.cand[slot] = key;
}

// Elements >= tv of this thread's chunk into the candidate buffer.  Only the
// vectors whose packed max reaches tv are visited (typically one).
template <typename T>
__device__ __forceinline__ void collect_candidates(const uint4 (&buf)[kScanVecs], int c0, int c1,
                                                   float tv, TopkSmem& sm) {
  constexpr int VW = ScanTraits<T>::kVW;
  uint32_t hit = 0;
  if constexpr (VW == 8) {
    // tv is a thread max, so it is exactly representable in bf16
    const __nv_bfloat162 tv2 = __float2bfloat162_rn(tv);
#pragma unroll
    for (int i = 0; i < kScanVecs; ++i) {
      const uint4 q = buf[i];
      const __nv_bfloat162 m2 =
          __hmax2(__hmax2(*reinterpret_cast<const __nv_bfloat162*>(&q.x),
                          *reinterpret_cast<const __nv_bfloat162*>(&q.y)),
                  __hmax2(*reinterpret_cast<const __nv_bfloat162*>(&q.z),
                          *reinterpret_cast<const __nv_bfloat162*>(&q.w)));
      hit |= (__hge2_mask(m2, tv2) ? 1u : 0u) << i;
    }
  } else {
#pragma unroll
    for (int i = 0; i < kScanVecs; ++i) {
      const uint4 q = buf[i];
      const float m = fmaxf(fmaxf(__uint_as_float(q.x), __uint_as_float(q.y)),
                            fmaxf(__uint_as_float(q.z), __uint_as_float(q.w)));
      hit |= (m >= tv ? 1u : 0u) << i;
    }
  }
  while (hit) {
    const int i = __ffs(hit) - 1;
    hit &= hit - 1;
    const uint4 q = buf_vec(buf, i);
    // bit j: element j of the vector reaches tv (independent compares)
    uint32_t em = 0;
    if constexpr (VW == 8) {
      const __nv_bfloat162 tv2 = __float2bfloat162_rn(tv);
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const uint32_t x = vec_word(q, w);
        const uint32_t mk = __hge2_mask(*reinterpret_cast<const __nv_bfloat162*>(&x), tv2);
        em |= ((mk & 1u) | ((mk >> 15) & 2u)) << (2 * w);
      }
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) em |= (__uint_as_float(vec_word(q, j)) >= tv ? 1u : 0u) << j;
    }
    while (em) {
      const int j = __ffs(em) - 1;
      em &= em - 1;
      const uint32_t w = vec_word(q, VW == 8 ? (j >> 1) : j);
      const float v = VW == 8 ? ((j & 1) ? bf16_hi(w) : bf16_lo(w)) : __uint_as_float(w);
      const int pos = scan_pos(c0, i, j, VW);
      if (pos < c1) push_cand(sm, make_key(v, (uint32_t)pos));
    }
  }
}

// Heavy ties (the candidate buffer overflowed): exact key threshold = the
// k-th largest per-thread (max, first position) key; candidates are the
// elements whose key reaches it (at most 64 * k).  The chunk is re-read from
// global memory in rolled loops: this path is rare and stays out of the hot
// code.  Called by every thread of the CTA; returns the candidate count.
template <typename T>
__device__ __noinline__ int tie_fallback(const T* __restrict__ rowp, int c0, int c1, int k,
                                         float tmax, TopkSmem& sm) {
  constexpr int VW = ScanTraits<T>::kVW;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __syncthreads();  // every thread has read ncand before it is reset below
  int fp = 0x7FFFFFFF;
#pragma unroll 1
  for (int e = 0; e < kScanVecs * VW && fp == 0x7FFFFFFF; ++e) {
    const int pos = scan_pos(c0, e / VW, e % VW, VW);
    if (pos < c1 && load_elem<T>(rowp, pos) == tmax) fp = pos;
  }
  const uint64_t tk = (fp == 0x7FFFFFFF) ? 0ull : make_key(tmax, (uint32_t)fp);
  const uint64_t sk = warp_sort_desc<uint64_t>(tk);
  if (lane < k) sm.warp_k[warp * k + lane] = sk;
  if (tid == 0) {
    sm.thr_key = 0ull;
    sm.ncand = 0;
  }
  __syncthreads();
  if (tid < 8 * k) {
    const uint64_t mine = sm.warp_k[tid];
    int rank = 0;
    for (int i = 0; i < 8 * k; ++i) rank += (sm.warp_k[i] > mine) ? 1 : 0;
    if (mine != 0ull && rank == k - 1) sm.thr_key = mine;
  }
  __syncthreads();
  const uint64_t thr = sm.thr_key;
  if (tk >= thr && tk != 0ull) {
#pragma unroll 1
    for (int e = 0; e < kScanVecs * VW; ++e) {
      const int pos = scan_pos(c0, e / VW, e % VW, VW);
      if (pos < c1) {
        const uint64_t key = make_key(load_elem<T>(rowp, pos), (uint32_t)pos);
        if (key >= thr) push_cand(sm, key);
      }
    }
  }
  __syncthreads();
  return min(sm.ncand, kCandMax);
}

template <typename T, bool kAligned>
__global__ void __launch_bounds__(kScanThreads, 4) expand_topk_kernel(TopkArgs a) {
  __shared__ TopkSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int row = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k;
  const int V = a.V;
  constexpr int VW = ScanTraits<T>::kVW;
  const float NEG_INF = __int_as_float(0xff800000);

  pdl_launch_dependents();
  pdl_wait();
  // physical row (uniform over the cluster: every CTA reads the same index)
  int r = row;
  if (a.row_idx) r = a.row_idx[row];
  if (r < 0 || r >= a.logit_rows) {
    if (crank == 0 && tid == 0) raise_status(a.status, kStIndex);
    return;
  }
  cluster_arrive_relaxed();
  // the leader's threads fetch the parent's path score now, while the
  // logits are in flight (one broadcast request per warp)
  float parent_score = 0.f;
  if (crank == 0) parent_score = __ldg(a.parent_score + row);
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)r * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);
  if (tid == 0) {
    sm.ncand = 0;
    sm.thr_ord = 0u;
  }

  // 1. per-thread max and exp-sum, warp-combined
  const float tmax = scan_thread_max<T>(buf);
  float m = tmax, s = scan_thread_sumexp<T>(buf, tmax);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_merge(m, s, m2, s2);
  }
  // 2. value threshold: the k-th largest of the 256 thread maxima.  It is
  //    among the top k of some warp's sorted list; each such entry counts
  //    the maxima >= itself in all eight lists, and the largest entry with
  //    a count >= k is the k-th largest.
  const float sv = warp_sort_desc<float>(tmax);
  sm.warp_v[warp * 32 + lane] = sv;
  __syncthreads();
  if (lane < k && count_ge_8x32(sm.warp_v, sv) >= k) atomicMax(&sm.thr_ord, ord_f32(sv));
  __syncthreads();
  const float tv = unord_f32(sm.thr_ord);
  // 3. candidates (only threads whose max reaches the threshold have any)
  if (tmax >= tv) collect_candidates<T>(buf, c0, c1, tv, sm);
  __syncthreads();
  int nc = sm.ncand;
  if (nc > kCandMax) nc = tie_fallback<T>(rowp, c0, c1, k, tmax, sm);

  // 4. rank the candidates and store the chunk's top-k (descending) straight
  //    into the leader's receive slots; slots past the candidates get 0
  cluster_wait();  // every CTA of the cluster is running: DSMEM is addressable
  TopkSmem* lead = cluster.map_shared_rank(&sm, 0);
  uint64_t* dst = lead->recv_top + crank * k;
  for (int i = tid; i < nc; i += kScanThreads) {
    const uint64_t mine = sm.cand[i];
    int rank = 0;
#pragma unroll 4
    for (int j = 0; j < nc; ++j) rank += (sm.cand[j] > mine) ? 1 : 0;
    if (rank < k) dst[rank] = mine;
  }
  if (tid >= nc && tid < k) dst[tid] = 0ull;
  if (lane == 0) {
    lead->recv_m[crank * 8 + warp] = m;
    lead->recv_s[crank * 8 + warp] = s;
  }
  cluster.sync();
  if (crank != 0) return;

  // ---- leader: key t (list c = t / k, index j = t % k) has row rank
  // j + the number of larger keys in the other lists (keys are unique; empty
  // slots are 0 and never reach rank k, as the row has >= k real keys)
  const int ck = C * k;
  if (warp * 32 >= ck) return;
  float M = NEG_INF, S = 0.f;
  for (int i = lane; i < C * 8; i += 32) lse_merge(M, S, sm.recv_m[i], sm.recv_s[i]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, M, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, S, o);
    lse_merge(M, S, m2, s2);
  }
  const float lse = (M == NEG_INF) ? M : M + log2f(S) * kLn2;
  for (int t = tid; t < ck; t += kScanThreads) {
    const uint64_t key = sm.recv_top[t];
    const int c = t / k;
    const int rank = t - c * k + count_gt_lists(sm.recv_top, C, k, c, key);
    if (key != 0ull && rank < k) {
      const float v = key_value(key);
      const float lp = (lse == NEG_INF) ? lse : (v - lse);
      const size_t o = (size_t)row * k + rank;
      a.tok[o] = (int32_t)key_index(key);
      a.logprob[o] = lp;
      a.score[o] = __fadd_rn(parent_score, lp);
      if (rank == 0 && a.lse_out) a.lse_out[row] = lse;
    }
  }
}

template <typename T, bool kAligned>
cudaError_t launch_topk_t(const TopkArgs& a, int C, cudaStream_t s) {
  auto kern = expand_topk_kernel<T, kAligned>;
  if (C > 8) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  for (int r0 = 0; r0 < a.rows; r0 += 65535) {
    TopkArgs b = a;
    const int nr = min(65535, a.rows - r0);
    b.rows = nr;
    if (b.row_idx) {
      b.row_idx += r0;
    } else {
      b.logits = static_cast<const char*>(a.logits) + (size_t)r0 * (size_t)a.ld * (a.is_bf16 ? 2 : 4);
      b.logit_rows = a.logit_rows - r0;
    }
    b.parent_score += r0;
    b.tok += (size_t)r0 * a.k;
    b.logprob += (size_t)r0 * a.k;
    b.score += (size_t)r0 * a.k;
    if (b.lse_out) b.lse_out += r0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C, nr, 1);
    cfg.blockDim = dim3(kScanThreads, 1, 1);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, b);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

// Cluster size for a row scan: enough CTAs to cover V with <= 64 elements
// per thread, more when there are few rows, at most 16.
int scan_cluster_size(int V, int is_bf16, int rows, int num_sms) {
  const int epc = is_bf16 ? scan_elems_per_cta<__nv_bfloat16>() : scan_elems_per_cta<float>();
  int C = (V + epc - 1) / epc;
  if (C < 1) C = 1;
  const int vw = is_bf16 ? 8 : 4;
  while (C < kMaxCluster && (long long)rows * C < num_sms && (V + 2 * C - 1) / (2 * C) >= 256 * vw)
    C *= 2;
  return C > kMaxCluster ? kMaxCluster : C;
}

cudaError_t launch_expand_topk(const TopkArgs& a, cudaStream_t s) {
  const int C = scan_cluster_size(a.V, a.is_bf16, a.rows, device_sm_count());
  const int esz = a.is_bf16 ? 2 : 4;
  const bool aligned = ((reinterpret_cast<uintptr_t>(a.logits) & 15) == 0) &&
                       (((a.ld * esz) & 15) == 0);
  if (a.is_bf16)
    return aligned ? launch_topk_t<__nv_bfloat16, true>(a, C, s)
                   : launch_topk_t<__nv_bfloat16, false>(a, C, s);
  return aligned ? launch_topk_t<float, true>(a, C, s) : launch_topk_t<float, false>(a, C, s);
}

}  // namespace tg
