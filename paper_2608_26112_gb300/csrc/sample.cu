// accept_sample: stochastic tree verification at temperature T > 0 (the
// rejection-sampling verification of Algorithms 1 and 2, which keeps the
// target's output distribution, Sec. 3.2).  Children are deterministic
// proposals, so the rule at node v with p = softmax(l_v / T) is: visit the
// children in ascending id; child c (token x) is accepted iff
// u[c, 0] * R_c < r(x), where r is p with the tokens of the children
// rejected before c removed and R_c = sum(r) = 1 - (their p); a child whose
// token repeats an earlier sibling's has r(x) = 0.  The walk follows the
// first accepted child; where all are rejected (or at a leaf) the bonus
// token is drawn from the residual by inversion with u[a*, 1].
//
// Every child's decision depends only on its parent's row and its earlier
// siblings (the walk reaches c only after rejecting them all), so all of
// them are taken in parallel:
//   sample_walk   grid (C, n_total), clusters of C CTAs per node row: the
//                 row's (max, sum of 2^((l - max) log2e / T)), then, in the
//                 leader, p of every child's token, an exclusive scan of
//                 the siblings' p in id order (duplicates count zero) and
//                 each child's flag; a ticket per tree, and the CTA that
//                 draws the last one walks the tree along the first flagged
//                 child of every node and writes path, A and a*;
//   sample_bonus  grid (C, B): row a* split over the cluster, each thread a
//                 contiguous run of tokens; the residual mass per thread
//                 (the tokens of a*'s children, all rejected, count zero),
//                 a cluster-wide scan in token order, and the one thread
//                 whose range holds u * sum(r) finds the token.
// The scan values are built so that neighbouring ranges share their bound
// bit for bit: the ranges partition [0, sum(r)) and exactly one thread
// claims the draw.
#include <cooperative_groups.h>

#include "launch.h"
#include "rowscan.cuh"

namespace cg = cooperative_groups;

namespace tg {
namespace {

struct WalkSmem {
  float red_m[8], red_s[8];
  float recv_m[16], recv_s[16];  // leader only: per-CTA (max, sum) of the row
  float wsum[8];
  int last;
  int par[256];
  int tok[256];
  int next[256];
};

// sum over this thread's elements of 2^((x - m) * c), m = the thread max
template <typename T>
__device__ __forceinline__ float thread_sumexp_scaled(const uint4 (&buf)[kScanVecs], float m,
                                                      float c) {
  if (m == __int_as_float(0xff800000)) return 0.f;
  constexpr int VW = ScanTraits<T>::kVW;
  // (x - m) first, then the scale: at small T the scale is large and
  // x * c - m * c would lose the difference to rounding
  const float2 c2 = make_float2(c, c), nm2 = make_float2(-m, -m);
  float2 acc0 = make_float2(0.f, 0.f), acc1 = make_float2(0.f, 0.f);
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
    for (int w = 0; w < VW / 2; ++w) {
      const float2 y = __fmul2_rn(__fadd2_rn(vec_pair<T>(buf[i], w), nm2), c2);
      const float2 e = make_float2(ex2(y.x), ex2(y.y));
      if (i & 1) acc1 = __fadd2_rn(acc1, e); else acc0 = __fadd2_rn(acc0, e);
    }
  return (acc0.x + acc0.y) + (acc1.x + acc1.y);
}

// (m, s) merge with the exponent scale c
__device__ __forceinline__ void merge_scaled(float& m, float& s, float m2, float s2, float c) {
  const float NEG_INF = __int_as_float(0xff800000);
  const float M = fmaxf(m, m2);
  if (M == NEG_INF) {
    m = M;
    s = 0.f;
    return;
  }
  s = (m == NEG_INF ? 0.f : s * ex2((m - M) * c)) + (m2 == NEG_INF ? 0.f : s2 * ex2((m2 - M) * c));
  m = M;
}

// Scan over the CTA's 256 threads in thread order: returns the inclusive
// value and sets excl to the previous thread's inclusive value (0 for
// thread 0), bit for bit: a warp's offset is accumulated so that it is the
// same float as the previous warp's last inclusive value.
__device__ __forceinline__ float block_scan(float x, float* wsum, float& excl) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  float off = 0.f;
  for (int w = 0; w < warp; ++w) off = off + wsum[w];
  __syncthreads();
  const float incl = warp == 0 ? x : off + x;
  const float prev = __shfl_up_sync(0xffffffffu, incl, 1);
  excl = lane == 0 ? off : prev;
  return incl;
}


template <typename T, bool kAligned>
__global__ void __launch_bounds__(kScanThreads, 4) sample_walk_kernel(SampleArgs a, int row_base) {
  __shared__ WalkSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int row = row_base + (int)blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int VW = ScanTraits<T>::kVW;
  const int V = a.V;
  const float cs = a.scale_log2;
  pdl_launch_dependents();
  pdl_wait();
  cluster_arrive_relaxed();
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)row * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);

  // the leader resolves the row's tree and fetches its parent / token arrays
  // while the logits are in flight
  int b = 0, off = 0, n = 0, v_par = -1, v_tok = 0;
  if (crank == 0) {
    int lo = 0, hi = a.B - 1;  // last b with node_off[b] <= row
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(a.node_off + mid) <= row) lo = mid; else hi = mid - 1;
    }
    b = lo;
    off = __ldg(a.node_off + b);
    n = __ldg(a.node_off + b + 1) - off;
    if (n >= 1 && n <= 256 && off >= 0 && off + n <= a.n_total && tid < n) {
      v_par = __ldg(a.parent + off + tid);
      v_tok = __ldg(a.token + off + tid);
    }
  }
  // (max, sum of 2^((x - max) * cs)) of the chunk
  float m = scan_thread_max<T>(buf);
  float sx = thread_sumexp_scaled<T>(buf, m, cs);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, sx, o);
    merge_scaled(m, sx, m2, s2, cs);
  }
  if (lane == 0) {
    sm.red_m[warp] = m;
    sm.red_s[warp] = sx;
  }
  __syncthreads();
  cluster_wait();
  if (tid == 0) {
    float cm = sm.red_m[0], csum = sm.red_s[0];
    for (int w = 1; w < 8; ++w) merge_scaled(cm, csum, sm.red_m[w], sm.red_s[w], cs);
    WalkSmem* lead = cluster.map_shared_rank(&sm, 0);
    lead->recv_m[crank] = cm;
    lead->recv_s[crank] = csum;
  }
  cluster.sync();
  if (crank != 0) return;

  // ---- leader: the row's (M, S), then its children's flags
  const bool bad_tree = (n < 1 || n > 256 || off < 0 || off + n > a.n_total);
  if (tid == 0) {
    float M = sm.recv_m[0], S = sm.recv_s[0];
    for (int c = 1; c < C; ++c) merge_scaled(M, S, sm.recv_m[c], sm.recv_s[c], cs);
    a.stat[row] = make_float2(M, S);
    sm.red_m[0] = M;
    sm.red_s[0] = S;
  }
  sm.par[tid] = v_par;
  sm.tok[tid] = v_tok;
  __syncthreads();
  const float M = sm.red_m[0], S = sm.red_s[0];
  const int v = row - off;
  const bool child = !bad_tree && tid < n && tid > v && v_par == v;
  float p = 0.f;
  bool dup = false;
  if (child) {
    if (v_tok < 0 || v_tok >= V) {
      raise_status(a.status, kStIndex);
      dup = true;  // no mass: never accepted
    } else {
      p = __fdiv_rn(ex2((load_elem<T>(rowp, v_tok) - M) * cs), S);
      for (int j = v + 1; j < tid && !dup; ++j) dup = (sm.par[j] == v && sm.tok[j] == v_tok);
    }
  }
  const float q = (child && !dup) ? p : 0.f;
  float before;
  block_scan(q, sm.wsum, before);   // mass of the earlier siblings, in id order
  if (child) {
    const float R = 1.f - before;
    const bool flag = !dup && (__ldg(a.u + 2 * (size_t)(off + tid)) * R < p);
    a.flag[off + tid] = flag ? 1 : 0;
    __threadfence();
  }
  __syncthreads();
  if (tid == 0) {
    if (bad_tree) {
      sm.last = 0;  // a malformed extent never touches the ticket
      raise_status(a.status, kStTree);
    } else {
      // release: the flags above reach the CTA that draws the last ticket;
      // acquire: that CTA sees every other row's flags
      const int t = atom_add_acq_rel_gpu(&a.tickets[b], 1);
      sm.last = (t == n - 1);
      if (sm.last) a.tickets[b] = 0;  // ready for the next call
    }
  }
  __syncthreads();
  if (!sm.last) return;

  // ---- walk of tree b along the first flagged child of every node
  const bool bad = (tid < n) && (tid == 0 ? (v_par != -1) : (v_par < 0 || v_par >= tid));
  if (__syncthreads_or(bad)) {
    if (tid == 0) {
      raise_status(a.status, kStTree);
      a.astar[b] = -1;
    }
    return;
  }
  sm.next[tid] = 0x7FFFFFFF;
  const int f = (tid > 0 && tid < n) ? __ldcg(a.flag + off + tid) : 0;
  __syncthreads();
  if (f) atomicMin(&sm.next[v_par], tid);
  __syncthreads();
  int32_t* path = a.path + (size_t)b * a.path_cap;
  if (tid == 0) {
    int w = 0, A = 0;
    while (sm.next[w] != 0x7FFFFFFF && A < n) {  // ids grow along the walk: at most n steps
      w = sm.next[w];
      ++A;
    }
    if (A + 1 > a.path_cap) {
      raise_status(a.status, kStIndex);
      a.astar[b] = -1;
      sm.last = -1;
    } else {
      int x = w;
      for (int d = A; d >= 0; --d) {
        path[d] = x;
        x = sm.par[x];
      }
      a.accept_len[b] = A;
      a.astar[b] = w;
      sm.last = A;
    }
  }
  __syncthreads();
  if (sm.last < 0) return;
  for (int d = sm.last + 1 + tid; d < a.path_cap; d += kScanThreads) path[d] = -1;
}


struct BonusSmem {
  unsigned long long excl[256];  // per thread: its elements that are a*'s children's tokens
  float tot[16];                 // per-CTA residual mass, in cluster rank order
  float wsum[8];
  int ch_tok[256];
  int nch;
};

// Thread t of CTA `crank` owns the contiguous tokens [c0 + t * E, + E) of
// row a*; element k sits in vector k / VW, lane k % VW.
template <typename T, bool kAligned>
__global__ void __launch_bounds__(kScanThreads) sample_bonus_kernel(SampleArgs a) {
  __shared__ BonusSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int b = blockIdx.y;
  const int tid = threadIdx.x;
  constexpr int VW = ScanTraits<T>::kVW;
  constexpr uint32_t kNeg = ScanTraits<T>::kNegInfWord;
  const int V = a.V;
  const float cs = a.scale_log2;
  pdl_launch_dependents();
  pdl_wait();
  cluster_arrive_relaxed();
  const int off = __ldg(a.node_off + b);
  const int n = __ldg(a.node_off + b + 1) - off;
  const int astar = __ldcg(a.astar + b);
  if (n < 1 || n > 256 || off < 0 || off + n > a.n_total || astar < 0 || astar >= n) {
    cluster_wait();
    return;  // the walk raised the status (uniform over the cluster)
  }
  const int row = off + astar;
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const int E = ((per + kScanThreads - 1) / kScanThreads + VW - 1) / VW * VW;  // <= 8 vectors
  const int nv = E / VW;
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)row * (size_t)a.ld;
  const int pos0 = c0 + tid * E;
  uint4 buf[kScanVecs];
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i) {
    const int pos = pos0 + i * VW;
    if (i < nv && pos < c1) {
      if (kAligned && pos + VW <= c1) buf[i] = *reinterpret_cast<const uint4*>(rowp + pos);
      else buf[i] = load_edge_vec<T>(rowp, pos, c1);
    } else {
      buf[i] = make_uint4(kNeg, kNeg, kNeg, kNeg);
    }
  }
  const float M = __ldcg(&a.stat[row].x);
  sm.excl[tid] = 0ull;
  if (tid == 0) sm.nch = 0;
  __syncthreads();
  // a*'s children (all rejected by the walk) leave the residual
  if (tid < n && __ldg(a.parent + off + tid) == astar) {
    const int x = __ldg(a.token + off + tid);
    sm.ch_tok[atomicAdd(&sm.nch, 1)] = x;
    if (x >= c0 && x < c1) {
      const int t = (x - c0) / E, k = (x - c0) - t * E;
      atomicOr(&sm.excl[t], 1ull << k);
    }
  }
  __syncthreads();
  const unsigned long long mask = sm.excl[tid];
  float own = 0.f;
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
    for (int j = 0; j < VW; ++j) {
      const float x = vec_elem<T>(buf[i], j);
      const bool out = ((mask >> (i * VW + j)) & 1ull) || x == __int_as_float(0xff800000);
      own = own + (out ? 0.f : ex2((x - M) * cs));
    }
  float excl;
  const float incl = block_scan(own, sm.wsum, excl);
  cluster_wait();  // every CTA of the cluster is running: remote stores are safe
  if (tid == kScanThreads - 1)
    for (int r = 0; r < C; ++r) cluster.map_shared_rank(&sm, r)->tot[crank] = incl;
  cluster_arrive_release();
  cluster_wait_acquire();
  float offset = 0.f;
  for (int r = 0; r < crank; ++r) offset = offset + sm.tot[r];
  float R = offset;
  for (int r = crank; r < C; ++r) R = R + sm.tot[r];
  const float g0 = offset + excl, g1 = offset + incl;
  if (R > 0.f) {
    float tau = __ldg(a.u + 2 * (size_t)row + 1) * R;
    if (tau >= R) tau = __int_as_float(__float_as_int(R) - 1);  // the largest float below R
    if (g0 <= tau && tau < g1) {  // exactly one thread of the cluster
      float run = g0;
      int chosen = -1, last = -1;
#pragma unroll
      for (int i = 0; i < kScanVecs; ++i)
#pragma unroll
        for (int j = 0; j < VW; ++j) {
          const float x = vec_elem<T>(buf[i], j);
          const bool out = ((mask >> (i * VW + j)) & 1ull) || x == __int_as_float(0xff800000);
          const float e = out ? 0.f : ex2((x - M) * cs);
          if (chosen < 0 && e > 0.f) {
            last = pos0 + i * VW + j;
            run = run + e;
            if (tau < run) chosen = last;
          }
        }
      a.bonus[b] = chosen >= 0 ? chosen : last;
    }
  } else if (crank == 0 && tid == 0) {
    // no residual mass in fp32 (the rejected children held all of it): the
    // token of the most likely child, as exact arithmetic would have
    // accepted it
    int best = -1;
    float bl = 0.f;
    for (int i = 0; i < sm.nch; ++i) {
      const int x = sm.ch_tok[i];
      if (x < 0 || x >= V) continue;
      const float l = load_elem<T>(rowp, x);
      if (best < 0 || l > bl || (l == bl && x < best)) {
        best = x;
        bl = l;
      }
    }
    a.bonus[b] = best;
  }
}

template <typename T, bool kAligned>
cudaError_t launch_sample_t(const SampleArgs& a, int C, int Cb, cudaStream_t s) {
  auto walk = sample_walk_kernel<T, kAligned>;
  auto bon = sample_bonus_kernel<T, kAligned>;
  if (C > 8 || Cb > 8) {
    cudaError_t e = cudaFuncSetAttribute(walk, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(bon, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kScanThreads, 1, 1);
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  attr[0].val.clusterDim.x = C;
  for (int r0 = 0; r0 < a.n_total; r0 += 65535) {
    cfg.gridDim = dim3(C, min(65535, a.n_total - r0), 1);
    cudaError_t e = cudaLaunchKernelEx(&cfg, walk, a, r0);
    if (e != cudaSuccess) return e;
  }
  attr[0].val.clusterDim.x = Cb;
  cfg.gridDim = dim3(Cb, a.B, 1);
  return cudaLaunchKernelEx(&cfg, bon, a);
}

}  // namespace

size_t sample_ws_bytes(int B, int n_total) {
  const size_t a8 = ((size_t)n_total * 8 + 255) / 256 * 256;
  const size_t a4 = ((size_t)n_total * 4 + 255) / 256 * 256;
  const size_t b4 = ((size_t)B * 4 + 255) / 256 * 256;
  return a8 + a4 + 2 * b4;
}

void sample_ws_carve(SampleArgs& a, void* ws, int B, int n_total) {
  const size_t a8 = ((size_t)n_total * 8 + 255) / 256 * 256;
  const size_t a4 = ((size_t)n_total * 4 + 255) / 256 * 256;
  const size_t b4 = ((size_t)B * 4 + 255) / 256 * 256;
  char* p = static_cast<char*>(ws);
  a.stat = reinterpret_cast<float2*>(p);
  a.flag = reinterpret_cast<int32_t*>(p + a8);
  a.astar = reinterpret_cast<int32_t*>(p + a8 + a4);
  a.tickets = reinterpret_cast<int32_t*>(p + a8 + a4 + b4);
}

cudaError_t launch_accept_sample(const SampleArgs& a, cudaStream_t s) {
  const int sms = device_sm_count();
  const int C = scan_cluster_size(a.V, a.is_bf16, a.n_total, sms);
  const int Cb = scan_cluster_size(a.V, a.is_bf16, a.B, sms);
  const int esz = a.is_bf16 ? 2 : 4;
  const bool aligned = ((reinterpret_cast<uintptr_t>(a.logits) & 15) == 0) &&
                       (((a.ld * esz) & 15) == 0);
  if (a.is_bf16)
    return aligned ? launch_sample_t<__nv_bfloat16, true>(a, C, Cb, s)
                   : launch_sample_t<__nv_bfloat16, false>(a, C, Cb, s);
  return aligned ? launch_sample_t<float, true>(a, C, Cb, s)
                 : launch_sample_t<float, false>(a, C, Cb, s);
}

}  // namespace tg

