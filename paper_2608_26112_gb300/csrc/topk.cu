// expand_topk: per-node log-softmax, exact top-k child tokens and cumulative
// path scores (Sec. 3.1 edge score p(u) and s(u) = s(v) p(u); Top_m of
// Algorithms 1 and 2), one HBM pass over the logits.
//
// Grid (C, rows) with clusters of C CTAs along x: the C CTAs of a cluster
// split one row.  Each CTA
//   1. stages its chunk in registers and takes per-thread (max, sum of
//      exp(x - max)) - packed bf16x2 max, one exp per element;
//   2. sorts the 256 thread maxima per warp and picks the value threshold
//      t = the largest value v with at least k thread maxima >= v.  At
//      least k elements reach t, and only threads whose max reaches t can
//      hold elements that do, so candidates are collected by a handful of
//      threads only;
//   3. ranks the candidates by 64-bit keys (value desc, token asc - exact
//      on ties) into its local top-k.  Heavily tied chunks can overflow the
//      candidate buffer; they fall back to an exact key threshold (the k-th
//      largest per-thread (max, first position) key), which bounds the
//      candidates by 64 * k;
//   4. pushes (max, sum, top-k) into the cluster leader's shared memory
//      (DSMEM stores) and meets the cluster barrier once.
// The leader merges the C partials into lse and the row's top-k and writes
// the outputs.  No global scratch and no second launch.
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
  uint64_t top[kMaxK];
  uint64_t recv_top[kMaxCluster * kMaxK];  // leader only: partials pushed by the cluster
  float recv_m[kMaxCluster];
  float recv_s[kMaxCluster];
  float warp_v[8 * kMaxK];
  uint64_t warp_k[8 * kMaxK];
  float red_m[8], red_s[8];
  uint32_t thr_ord;
  uint64_t thr_key;
  int ncand;
  float lse;
};

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
  // the leader's output threads fetch the parent's path score now, while
  // the logits are in flight
  float parent_score = 0.f;
  if (crank == 0 && tid < k) parent_score = __ldg(a.parent_score + row);
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)r * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);
  if (tid == 0) {
    sm.thr_ord = 0u;
    sm.ncand = 0;
  }
  if (tid < kMaxK) sm.top[tid] = 0ull;

  // 1. per-thread max and exp-sum, warp-combined
  const float tmax = scan_thread_max<T>(buf);
  float m = tmax, s = scan_thread_sumexp<T>(buf, tmax);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    lse_merge(m, s, m2, s2);
  }
  // 2. value threshold from the sorted thread maxima
  const float sv = warp_sort_desc<float>(tmax);
  if (lane < k) sm.warp_v[warp * k + lane] = sv;
  if (lane == 0) {
    sm.red_m[warp] = m;
    sm.red_s[warp] = s;
  }
  __syncthreads();
  if (tid < 8 * k) {
    const float v = sm.warp_v[tid];
    int ge = 0;
    for (int i = 0; i < 8 * k; ++i) ge += (sm.warp_v[i] >= v) ? 1 : 0;
    if (ge >= k && v == v) atomicMax(&sm.thr_ord, ord_f32(v));
  }
  __syncthreads();
  const float tv = unord_f32(sm.thr_ord);
  // 3. candidates (only threads whose max reaches the threshold have any)
  if (tmax >= tv) {
    auto push = [&](float v, int pos) {
      if (pos < c1) {
        const int slot = atomicAdd(&sm.ncand, 1);
        if (slot < kCandMax) sm.cand[slot] = make_key(v, (uint32_t)pos);
      }
    };
    if constexpr (VW == 8) {
      // one packed compare per element pair; tv is a thread max, so it is
      // exactly representable in bf16
      const __nv_bfloat162 tv2 = __float2bfloat162_rn(tv);
#pragma unroll
      for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const uint32_t x = vec_word(buf[i], w);
          const uint32_t mk = __hge2_mask(*reinterpret_cast<const __nv_bfloat162*>(&x), tv2);
          if (mk) {
            const int pos = scan_pos(c0, i, 2 * w, VW);
            if (mk & 0xFFFFu) push(bf16_lo(x), pos);
            if (mk >> 16) push(bf16_hi(x), pos + 1);
          }
        }
    } else {
#pragma unroll
      for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
        for (int j = 0; j < VW; ++j) {
          const float v = vec_elem<T>(buf[i], j);
          if (v >= tv) push(v, scan_pos(c0, i, j, VW));
        }
    }
  }
  __syncthreads();
  int nc = sm.ncand;
  if (nc > kCandMax) {
    // heavy ties: exact key threshold = k-th largest (thread max, first position)
    __syncthreads();  // every thread has read ncand before it is reset below
    const int fp = (c0 + (int)tid * VW >= c1) ? 0x7FFFFFFF : scan_first_pos<T>(buf, c0, c1, tmax);
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
#pragma unroll
      for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
        for (int j = 0; j < VW; ++j) {
          const int pos = scan_pos(c0, i, j, VW);
          const uint64_t key = make_key(vec_elem<T>(buf[i], j), (uint32_t)pos);
          if (pos < c1 && key >= thr) {
            const int slot = atomicAdd(&sm.ncand, 1);
            if (slot < kCandMax) sm.cand[slot] = key;
          }
        }
    }
    __syncthreads();
    nc = min(sm.ncand, kCandMax);
  }
  for (int i = tid; i < nc; i += kScanThreads) {
    const uint64_t mine = sm.cand[i];
    int rank = 0;
    for (int j = 0; j < nc; ++j) rank += (sm.cand[j] > mine) ? 1 : 0;
    if (rank < k) sm.top[rank] = mine;
  }
  __syncthreads();

  // 4. push the partial into the leader's shared memory
  cluster_wait();
  TopkSmem* lead = cluster.map_shared_rank(&sm, 0);
  if (tid < k) lead->recv_top[crank * k + tid] = sm.top[tid];
  if (tid == 0) {
    float M = sm.red_m[0], S = sm.red_s[0];
#pragma unroll
    for (int w = 1; w < 8; ++w) lse_merge(M, S, sm.red_m[w], sm.red_s[w]);
    lead->recv_m[crank] = M;
    lead->recv_s[crank] = S;
  }
  cluster.sync();
  if (crank != 0) return;

  // ---- leader: merge the C partials
  if (warp == 0) {
    // lse over the C partials: one (max, sum) per lane, shuffle tree
    float M = lane < C ? sm.recv_m[lane] : __int_as_float(0xff800000);
    float S = lane < C ? sm.recv_s[lane] : 0.f;
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, M, o);
      const float s2 = __shfl_xor_sync(0xffffffffu, S, o);
      lse_merge(M, S, m2, s2);
    }
    if (lane == 0) {
      const float lse = (M == __int_as_float(0xff800000)) ? M : M + log2f(S) * kLn2;
      sm.lse = lse;
      if (a.lse_out) a.lse_out[row] = lse;
    }
  }
  for (int t = tid; t < C * k; t += kScanThreads) {
    const uint64_t mine = sm.recv_top[t];
    int rank = 0;
    for (int j = 0; j < C * k; ++j) rank += (sm.recv_top[j] > mine) ? 1 : 0;
    if (rank < k) sm.top[rank] = mine;
  }
  __syncthreads();
  if (tid < k) {
    const uint64_t key = sm.top[tid];
    const float v = key_value(key);
    const float lse = sm.lse;
    const float lp = (lse == __int_as_float(0xff800000)) ? lse : (v - lse);
    const size_t o = (size_t)row * k + tid;
    a.tok[o] = (int32_t)key_index(key);
    a.logprob[o] = lp;
    a.score[o] = __fadd_rn(parent_score, lp);
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
