// expand_topk: per-node log-softmax, exact top-k child tokens and cumulative
// path scores (Sec. 3.1 edge score p(u) and s(u) = s(v) p(u); Top_m of
// Algorithms 1 and 2), one HBM pass over the logits.
//
// Grid (C, rows) with clusters of C CTAs along x: the C CTAs of a cluster
// split one row.  Each CTA
//   1. stages its chunk in registers (rowscan.cuh),
//   2. reduces the chunk max m_c and sum_t exp(l_t - m_c),
//   3. finds an exact threshold key: the k-th largest of the 256 per-thread
//      maxima (a warp bitonic sort, then a rank count over 8 * k keys).  At
//      least k elements reach it and only the k threads owning the top-k
//      maxima can hold elements above it, so at most 64 * k candidates pass,
//   4. collects the candidates in shared memory and ranks them to its local
//      top-k (64-bit keys: value desc, token asc - exact on ties).
// The cluster leader then pulls every CTA's (m_c, s_c, top-k) over DSMEM,
// merges them into lse and the row's top-k, and writes the outputs.  No
// global scratch and no second launch.
#include <cooperative_groups.h>

#include "launch.h"
#include "rowscan.cuh"

namespace cg = cooperative_groups;

namespace tg {
namespace {

constexpr int kMaxK = 32;
constexpr int kCandMax = kMaxK * kScanVecs * 8;  // 64 elements/thread * k
constexpr int kMaxCluster = 16;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct TopkSmem {
  uint64_t cand[kCandMax];
  uint64_t warp_top[8 * kMaxK];
  uint64_t top[kMaxK];
  uint64_t merged[kMaxCluster * kMaxK];
  float merged_m[kMaxCluster];
  float merged_s[kMaxCluster];
  float red_f[8];
  float part_m, part_s;
  uint64_t thr;
  int ncand;
  int bad_row;
};

// descending bitonic sort of one 64-bit key per lane; lane j ends with the
// j-th largest
__device__ __forceinline__ uint64_t warp_sort_desc(uint64_t x) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const uint64_t y = __shfl_xor_sync(0xffffffffu, x, stride);
      const bool asc_block = (lane & size) == 0;
      const bool lower = (lane & stride) == 0;
      const bool take_max = (lower == asc_block);
      x = take_max ? (x > y ? x : y) : (x < y ? x : y);
    }
  }
  return x;
}

template <typename T, bool kAligned>
__global__ void __launch_bounds__(kScanThreads) expand_topk_kernel(TopkArgs a) {
  __shared__ TopkSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int row = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k;
  const int V = a.V;

  // physical row (uniform over the cluster: every CTA reads the same index)
  int r = row;
  if (a.row_idx) r = a.row_idx[row];
  if (r < 0 || r >= a.logit_rows) {
    if (crank == 0 && tid == 0) raise_status(a.status, kStIndex);
    return;
  }
  constexpr int VW = ScanTraits<T>::kVW;
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)r * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);

  if (tid == 0) {
    sm.thr = 0;
    sm.ncand = 0;
  }
  if (tid < kMaxK) sm.top[tid] = 0;

  // 1. thread max (first position on ties) and chunk max
  float tmax;
  int tpos;
  scan_thread_max<T>(buf, c0, c1, tmax, tpos);
  float wm = warp_max_f32(tmax);
  if (lane == 0) sm.red_f[warp] = wm;
  __syncthreads();
  float m_c = sm.red_f[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) m_c = fmaxf(m_c, sm.red_f[w]);

  // 2. sum of exp(l - m_c)
  float ssum = 0.f;
  if (m_c != __int_as_float(0xff800000)) {
    const float mb = -m_c * kLog2e;
#pragma unroll
    for (int i = 0; i < kScanVecs; ++i) {
#pragma unroll
      for (int j = 0; j < VW; ++j) ssum += ex2(fmaf(vec_elem<T>(buf[i], j), kLog2e, mb));
    }
  }
  ssum = warp_sum_f32(ssum);
  __syncthreads();  // red_f reuse
  if (lane == 0) sm.red_f[warp] = ssum;

  // 3. threshold = k-th largest per-thread max key
  const uint64_t tkey = (tpos < 0) ? 0ull : make_key(tmax, (uint32_t)tpos);
  const uint64_t sorted = warp_sort_desc(tkey);
  if (lane < k) sm.warp_top[warp * k + lane] = sorted;
  __syncthreads();
  if (tid == 0) {
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s += sm.red_f[w];
    sm.part_m = m_c;
    sm.part_s = s;
  }
  if (tid < 8 * k) {
    const uint64_t mine = sm.warp_top[tid];
    int rank = 0;
    for (int i = 0; i < 8 * k; ++i) rank += (sm.warp_top[i] > mine) ? 1 : 0;
    if (mine != 0ull && rank == k - 1) sm.thr = mine;
  }
  __syncthreads();

  // 4. candidates: elements whose key reaches the threshold
  {
    const uint64_t thr = sm.thr;
    const bool take_all = (thr == 0ull);
    const float tv = key_value(thr);
    const int tp = (int)key_index(thr);
#pragma unroll
    for (int i = 0; i < kScanVecs; ++i) {
      const int base = c0 + (i * kScanThreads + tid) * VW;
#pragma unroll
      for (int j = 0; j < VW; ++j) {
        const float v = vec_elem<T>(buf[i], j);
        const int pos = base + j;
        if (pos < c1 && (take_all || v > tv || (v == tv && pos <= tp))) {
          const int slot = atomicAdd(&sm.ncand, 1);
          if (slot < kCandMax) sm.cand[slot] = make_key(v, (uint32_t)pos);
        }
      }
    }
  }
  __syncthreads();
  {
    const int nc = min(sm.ncand, kCandMax);
    for (int i = tid; i < nc; i += kScanThreads) {
      const uint64_t mine = sm.cand[i];
      int rank = 0;
      for (int j = 0; j < nc; ++j) rank += (sm.cand[j] > mine) ? 1 : 0;
      if (rank < k) sm.top[rank] = mine;
    }
  }

  // 5. cluster merge at rank 0
  cluster.sync();
  if (crank == 0) {
    for (int t = tid; t < C * k; t += kScanThreads) {
      const TopkSmem* peer = cluster.map_shared_rank(&sm, t / k);
      sm.merged[t] = peer->top[t % k];
    }
    if (tid < C) {
      const TopkSmem* peer = cluster.map_shared_rank(&sm, tid);
      sm.merged_m[tid] = peer->part_m;
      sm.merged_s[tid] = peer->part_s;
    }
  }
  cluster.sync();
  if (crank != 0) return;

  __shared__ float lse_s;
  if (tid == 0) {
    float M = sm.merged_m[0];
    for (int c = 1; c < C; ++c) M = fmaxf(M, sm.merged_m[c]);
    float lse;
    if (M == __int_as_float(0xff800000)) {
      lse = M;
    } else {
      float S = 0.f;
      for (int c = 0; c < C; ++c) {
        const float mc = sm.merged_m[c];
        if (mc != __int_as_float(0xff800000)) S += sm.merged_s[c] * ex2((mc - M) * kLog2e);
      }
      lse = M + log2f(S) * kLn2;
    }
    lse_s = lse;
    if (a.lse_out) a.lse_out[row] = lse;
  }
  __syncthreads();
  for (int t = tid; t < C * k; t += kScanThreads) {
    const uint64_t mine = sm.merged[t];
    int rank = 0;
    for (int j = 0; j < C * k; ++j) rank += (sm.merged[j] > mine) ? 1 : 0;
    if (rank < k) sm.top[rank] = mine;  // own top[] is no longer read by peers
  }
  __syncthreads();
  if (tid < k) {
    const uint64_t key = sm.top[tid];
    const float v = key_value(key);
    const float lse = lse_s;
    const float lp = (lse == __int_as_float(0xff800000)) ? lse : (v - lse);
    const size_t o = (size_t)row * k + tid;
    a.tok[o] = (int32_t)key_index(key);
    a.logprob[o] = lp;
    a.score[o] = __fadd_rn(a.parent_score[row], lp);
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
    if (b.row_idx) b.row_idx += r0;
    else b.logits = static_cast<const char*>(a.logits) +
                    (size_t)r0 * (size_t)a.ld * (a.is_bf16 ? 2 : 4);
    if (!b.row_idx) b.logit_rows = a.logit_rows - r0;
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
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = C;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
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
  // with few rows, spread each row over more CTAs (at least ~1 CTA per SM)
  const int vw = is_bf16 ? 8 : 4;
  while (C < kMaxCluster && (long long)rows * C < num_sms && (V + 2 * C - 1) / (2 * C) >= 256 * vw)
    C *= 2;
  return C > kMaxCluster ? -1 : C;
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
