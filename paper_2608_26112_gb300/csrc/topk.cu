// expand_topk: per-node log-softmax, exact top-k child tokens and cumulative
// path scores (Sec. 3.1 edge score p(u) and s(u) = s(v) p(u); Top_m of
// Algorithms 1 and 2), one HBM pass over the logits.
//
// Grid (C, rows) with clusters of C CTAs along x: the C CTAs of a cluster
// split one row.  The selection uses no block barrier, only three phases of
// the cluster barrier:
//   0. every CTA stages its chunk in registers (eight 16-byte loads per
//      thread, all in flight at once) and takes its thread maxima; each warp
//      finds its top r lane maxima (r = ceil(k / (8 C)), so the row pushes at
//      least k values) and stores them into EVERY CTA of the cluster (DSMEM);
//   1. while the other CTAs finish, each thread takes the sum of exp(x - max)
//      over its elements (packed bf16x2 max, one exp per element), each warp
//      folds its lanes' (max, sum) with one exponential per lane and pushes
//      the pair to the leader.  After the barrier every
//      warp holds the same 8 C r pushed maxima and takes their k-th largest
//      T: k distinct elements of the row reach T, so the row's top-k all do.
//      Only threads whose max reaches T hold elements that do; they visit
//      the 16-byte vectors whose packed max reaches T and push those
//      elements' 64-bit keys (value desc, token asc - exact on ties) into the
//      leader's candidate buffer (DSMEM atomics);
//   2. the leader ranks the few candidates by counting larger keys, folds
//      the C * 8 (max, sum) pairs into the lse, and writes token, logprob =
//      x - lse and score = fp32(parent_score + logprob).  A tie-heavy row that
//      overflows the candidate buffer is ranked exactly by the leader alone
//      from global memory (k rounds of a block-wide key max) - slow, rare.
// No global scratch and no second launch.  The kernels are latency-bound
// after the load, so the code keeps dependency chains short and the
// executed code small (rare paths are rolled loops).
#include <cooperative_groups.h>

#include "launch.h"
#include "rowscan.cuh"

namespace cg = cooperative_groups;

namespace tg {
namespace {

constexpr int kMaxK = 32;  // TG_MAX_TOPK
constexpr int kMaxCluster = 16;
constexpr int kMaxPush = 128;   // pushed lane maxima per row: 8 C r <= 128
// r = ceil(k / (8 C)) <= 4 lane maxima per warp give 8 C r >= k pushed values
static_assert(kMaxK <= 8 * 4 && 8 * kMaxCluster <= kMaxPush, "push sizes");
constexpr int kCandMax = 2048;  // the leader's candidate buffer

struct TopkSmem {
  uint64_t cand[kCandMax];        // leader: candidate keys of the whole row
  float push_v[kMaxPush];         // every CTA: the row's pushed lane maxima
  float recv_m[kMaxCluster * 8];  // leader: each warp's (max, sum)
  float recv_s[kMaxCluster * 8];
  uint64_t red_k[8];              // leader fallback: block reduction
  int ncand;                      // leader: candidate count
};

// (max, sum of exp(x - max)) of the 32 lanes' pairs, in every lane: the max
// by one warp-wide integer max, one exponential per lane, a shuffle sum.
__device__ __forceinline__ void warp_lse_pair(float& m, float& s) {
  const float NEG_INF = __int_as_float(0xff800000);
  const float M = unord_f32(__reduce_max_sync(0xffffffffu, ord_f32(m)));
  float t = (m == NEG_INF) ? 0.f : s * ex2((m - M) * kLog2e);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  m = M;
  s = t;
}

// r rounds of warp-wide max extraction: lane i < r ends with the i-th
// largest of the 32 lane values (each round pops one lane holding the max;
// ties are popped one at a time, lowest lane first).
__device__ __forceinline__ float warp_top_r(float x, int r) {
  const int lane = threadIdx.x & 31;
  float out = __int_as_float(0xff800000);
  uint32_t h = ord_f32(x);
  for (int i = 0; i < r; ++i) {
    const uint32_t mx = __reduce_max_sync(0xffffffffu, h);
    const uint32_t who = __ffs(__ballot_sync(0xffffffffu, h == mx)) - 1;
    if (lane == i) out = unord_f32(mx);
    if (lane == (int)who) h = 0u;  // below every ordered value (ord(-inf) > 0)
  }
  return out;
}

// k-th largest (with multiplicity) of the n <= 128 values at v[]: each lane
// sorts its 4 values, then rounds of warp-wide max extraction count them
// down.  Every lane returns the same value.
__device__ __forceinline__ float kth_largest_128(const float* v, int n, int k) {
  const int lane = threadIdx.x & 31;
  const float NEG_INF = __int_as_float(0xff800000);
  float a0 = lane < n ? v[lane] : NEG_INF;
  float a1 = lane + 32 < n ? v[lane + 32] : NEG_INF;
  float a2 = lane + 64 < n ? v[lane + 64] : NEG_INF;
  float a3 = lane + 96 < n ? v[lane + 96] : NEG_INF;
  auto cas = [](float& x, float& y) {
    const float hi = fmaxf(x, y), lo = fminf(x, y);
    x = hi;
    y = lo;
  };
  cas(a0, a1);
  cas(a2, a3);
  cas(a0, a2);
  cas(a1, a3);
  cas(a1, a2);
  int cnt = 0;
  for (int round = 0; round < kMaxPush; ++round) {  // ends after at most k rounds
    const uint32_t h = ord_f32(a0);
    const uint32_t mx = __reduce_max_sync(0xffffffffu, h);
    const bool mine = h == mx;
    cnt += __popc(__ballot_sync(0xffffffffu, mine));
    if (cnt >= k) return unord_f32(mx);
    if (mine) {
      a0 = a1;
      a1 = a2;
      a2 = a3;
      a3 = NEG_INF;
    }
  }
  return NEG_INF;
}

// Elements >= tv of this thread's chunk into the leader's candidate buffer
// (DSMEM atomics for the slots).  Only the vectors whose packed max reaches
// tv are visited (typically one).
template <typename T>
__device__ __forceinline__ void push_candidates(const uint4 (&buf)[kScanVecs], int c0, int c1,
                                                float tv, TopkSmem* lead) {
  constexpr int VW = ScanTraits<T>::kVW;
  uint32_t hit = 0;
  if constexpr (VW == 8) {
    // tv is an element value, so it is exactly representable in bf16
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
      if (pos < c1) {
        const int slot = atomicAdd(&lead->ncand, 1);
        if (slot < kCandMax) lead->cand[slot] = make_key(v, (uint32_t)pos);
      }
    }
  }
}

// Leader only, when the candidate buffer overflowed (heavy ties): the row's
// exact top-k by k rounds of a block-wide max over the keys below the last
// one found, read from global memory.  Returns in smem cand[0..k).
template <typename T>
__device__ __noinline__ void exact_topk_fallback(const T* __restrict__ rowp, int V, int k,
                                                 TopkSmem& sm) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  uint64_t last = ~0ull;
#pragma unroll 1
  for (int r = 0; r < k; ++r) {
    uint64_t best = 0ull;
#pragma unroll 1
    for (int pos = tid; pos < V; pos += kScanThreads) {
      const uint64_t key = make_key(load_elem<T>(rowp, pos), (uint32_t)pos);
      if (key < last && key > best) best = key;
    }
    best = warp_max_u64(best);
    if (lane == 0) sm.red_k[warp] = best;
    __syncthreads();
    best = sm.red_k[0];
#pragma unroll
    for (int w = 1; w < 8; ++w) best = sm.red_k[w] > best ? sm.red_k[w] : best;
    __syncthreads();
    if (tid == 0) sm.cand[r] = best;
    last = best;
  }
  __syncthreads();
}

// kTree: the tree-batch row mapping and the append of children (grow step),
// compiled out of the plain kernel.
// kMinCtas: resident CTAs per SM the registers are fitted to.  At batches
// of many rows (more than one wave of four CTAs per SM) each CTA holds its
// slot through the cluster phases after its load, so five resident CTAs (48
// registers, a few spilled) keep more bytes in flight: 6 % faster at 8 K
// rows.  In one wave the spills only lengthen the chain after the load
// (+1.1 us at 60 rows), so small batches keep four (62 registers).
template <typename T, bool kAligned, bool kTree, int kMinCtas>
__global__ void __launch_bounds__(kScanThreads, kMinCtas) expand_topk_kernel(TopkArgs a) {
  __shared__ TopkSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int row = a.row0 + (int)blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = a.k;
  const int V = a.V;
  constexpr int VW = ScanTraits<T>::kVW;
  const float NEG_INF = __int_as_float(0xff800000);

  pdl_launch_dependents();
  pdl_wait();
  // physical row (uniform over the cluster: every CTA reads the same index)
  int r = row;
  if (a.row_idx) {
    r = a.row_idx[row];
    if (kTree && a.idx_local) {  // a local node id of tree row / gdiv (graft)
      const int bt = row / a.gdiv;
      r = (r >= 0 && r < a.app_n) ? bt * a.gcap + r : -1;
    }
  } else if (kTree && a.gdiv) {
    const int bt = row / a.gdiv;
    r = bt * a.gcap + a.goff + (row - bt * a.gdiv);
  }
  if (r < 0 || r >= a.logit_rows) {
    if (crank == 0 && tid == 0) raise_status(a.status, kStIndex);
    return;
  }
  if (crank == 0 && tid == 0) sm.ncand = 0;
  // phase 0: the leader's counter is initialised before any CTA can push
  cluster_arrive_release();
  // the leader's threads fetch the parent's path score now, while the
  // logits are in flight (one broadcast request per warp)
  float parent_score = 0.f;
  if (crank == 0 && a.parent_score)
    parent_score = __ldg(a.parent_score + ((kTree && a.ps_gather) ? r : row));
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)r * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);
  const float tmax = scan_thread_max<T>(buf);
  // each warp's top rp lane maxima go to every CTA of the cluster
  const int rp = min(4, (k + 8 * C - 1) / (8 * C));
  const int npush = 8 * C * rp;
  const float top = warp_top_r(tmax, rp);
  cluster_wait_acquire();
  TopkSmem* lead = cluster.map_shared_rank(&sm, 0);
  if (lane < rp) {
    const int slot = (crank * 8 + warp) * rp + lane;
    for (int c = 0; c < C; ++c) cluster.map_shared_rank(&sm, c)->push_v[slot] = top;
  }
  // phase 1: the pushed maxima become visible; the exp-sum runs while the
  // other CTAs finish their loads
  cluster_arrive_release();
  float m = tmax, s = scan_thread_sumexp<T>(buf, tmax);
  warp_lse_pair(m, s);
  if (lane == 0) {
    lead->recv_m[crank * 8 + warp] = m;
    lead->recv_s[crank * 8 + warp] = s;
  }
  cluster_wait_acquire();
  const float tv = kth_largest_128(sm.push_v, npush, k);
  if (tmax >= tv) push_candidates<T>(buf, c0, c1, tv, lead);
  // phase 2: every candidate and (max, sum) has reached the leader
  cluster_arrive_release();
  cluster_wait_acquire();
  if (crank != 0) return;

  // ---- leader: lse and the row's top-k from the candidates
  const int nc = sm.ncand;
  if (nc > kCandMax) exact_topk_fallback<T>(rowp, V, k, sm);
  const int nr = nc > kCandMax ? k : nc;  // keys to rank; the fallback's are already in order
  if (warp * 32 >= nr) return;
  float M = NEG_INF, S = 0.f;
  for (int i = lane; i < C * 8; i += 32) lse_merge(M, S, sm.recv_m[i], sm.recv_s[i]);
  warp_lse_pair(M, S);
  const float lse = (M == NEG_INF) ? M : M + log2f(S) * kLn2;
  for (int t = tid; t < nr; t += kScanThreads) {
    const uint64_t key = sm.cand[t];
    int rank = t;
    if (nc <= kCandMax) {
      rank = 0;
#pragma unroll 4
      for (int j = 0; j < nr; ++j) rank += (sm.cand[j] > key) ? 1 : 0;
    }
    if (rank < k) {
      const float v = key_value(key);
      const float lp = (lse == NEG_INF) ? lse : (v - lse);
      if (kTree && a.app_token) {  // children appended to the tree (grow step)
        const int bt = row / a.gdiv;
        const size_t u = (size_t)bt * a.gcap + a.app_n + (size_t)(row - bt * a.gdiv) * k + rank;
        a.app_parent[u] = r - bt * a.gcap;
        a.app_token[u] = (int32_t)key_index(key);
        a.app_edge[u] = lp;
        a.app_score[u] = __fadd_rn(parent_score, lp);
      } else {
        const size_t o = (size_t)row * k + rank;
        a.tok[o] = (int32_t)key_index(key);
        a.logprob[o] = lp;
        if (a.score) a.score[o] = __fadd_rn(parent_score, lp);
      }
      if (rank == 0 && a.lse_out) a.lse_out[row] = lse;
    }
  }
}

template <typename T, bool kAligned>
cudaError_t launch_topk_t(const TopkArgs& a, int C, int num_sms, cudaStream_t s) {
  const bool tree = a.gdiv || a.app_token;
  const bool many = (long long)a.rows * C > 4LL * num_sms;
  auto kern = tree ? (many ? expand_topk_kernel<T, kAligned, true, 5>
                           : expand_topk_kernel<T, kAligned, true, 4>)
                   : (many ? expand_topk_kernel<T, kAligned, false, 5>
                           : expand_topk_kernel<T, kAligned, false, 4>);
  if (C > 8) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  for (int r0 = 0; r0 < a.rows; r0 += 65535) {
    TopkArgs b = a;
    const int nr = min(65535, a.rows - r0);
    b.rows = nr;
    b.row0 = r0;  // the kernel indexes rows, parent scores and outputs by r0 + blockIdx.y
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
  const int nsm = device_sm_count();
  const int C = scan_cluster_size(a.V, a.is_bf16, a.rows, nsm);
  const int esz = a.is_bf16 ? 2 : 4;
  const bool aligned = ((reinterpret_cast<uintptr_t>(a.logits) & 15) == 0) &&
                       (((a.ld * esz) & 15) == 0);
  if (a.is_bf16)
    return aligned ? launch_topk_t<__nv_bfloat16, true>(a, C, nsm, s)
                   : launch_topk_t<__nv_bfloat16, false>(a, C, nsm, s);
  return aligned ? launch_topk_t<float, true>(a, C, nsm, s)
                 : launch_topk_t<float, false>(a, C, nsm, s);
}

}  // namespace tg
