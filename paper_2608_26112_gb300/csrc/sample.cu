// accept_sample: stochastic tree verification at temperature T > 0 (the
// rejection-sampling verification of Algorithms 1 and 2, which keeps the
// target's output distribution, Sec. 3.2).  Children are deterministic
// proposals, so the rule at node v with p = softmax(l_v / T) is: visit the
// children in ascending id; child c (token x) is accepted iff
// u[c, 0] * R_c < r(x), where r is p with the tokens of the children
// rejected before c removed and R_c = sum(r); a child whose token repeats
// an earlier sibling's has r(x) = 0.  The walk follows the first accepted
// child; where all are rejected (or at a leaf) the bonus token is drawn from
// the residual by inversion with u[a*, 1].
//
// One launch, grid (C, n_total), clusters of C CTAs per node row.  Every
// child's decision depends only on its parent's row and its earlier
// siblings (the walk reaches c only after rejecting them all), and the
// bonus draw at v only on v's row and v's children (all rejected if the
// walk ends at v), so each row's cluster takes all of them at once:
//   masses  w(t) = 2^((l_t - max) log2e / T), summed in fp32 per 16-byte
//           vector and then taken as 40-bit fixed point, so every sum above
//           a vector is exact and independent of its order: the cluster's
//           residual mass R (v's children's tokens left out) and
//           S = R + the children's masses;
//   flags   child c is accepted iff u[c, 0] (S - w of its earlier distinct
//           siblings) < w(x_c);
//   bonus   the token holding fixed-point mass floor(u[v, 1] R) in token
//           order, found by a cluster-wide prefix of per-CTA totals, then
//           the CTA's per-vector totals, then a scan over its threads;
// and the CTA that draws a tree's last ticket (two per row: the flags and
// the bonus candidate) walks the tree along the first accepted child of
// every node and reads the bonus of a*.
#include <cooperative_groups.h>

#include "launch.h"
#include "rowscan.cuh"

namespace cg = cooperative_groups;

namespace tg {
namespace {

constexpr int kMaxC = 16;

struct SampleSmem {
  float cmax[kMaxC];                          // per-CTA max of the row (every CTA)
  unsigned long long ctot[kMaxC];             // per-CTA residual mass (every CTA)
  unsigned long long sv[kScanVecs][kScanThreads];  // per vector, per thread residual mass
  unsigned long long vtot[kScanVecs];         // this CTA's per-vector residual mass
  unsigned long long wsc[8];                  // warp totals of a scan
  unsigned long long excl[kScanThreads];      // per thread: its elements that are v's children
  unsigned long long best;                    // leader: most likely child (no residual mass)
  float red_m[8];
  int par[256];
  int tok[256];
  int next[256];
  int last;
};

// A non-negative float below 16 (a mass w = 2^((x - M) cs) <= 1, or the sum
// of one vector's masses) as a fixed-point integer in units of 2^-40
// (truncated), taken from the float's exponent and mantissa with shifts:
// w = m 2^(e - 150) for the 24-bit mantissa m and biased exponent e.  A row
// of at most 2^18 tokens sums below 2^59.  Monotone in w.
__device__ __forceinline__ unsigned long long to_fixed(float w) {
  const uint32_t bits = __float_as_uint(w);
  const int e = (int)(bits >> 23);
  const uint32_t m = (bits & 0x7FFFFFu) | 0x800000u;
  const int sh = e - 110;
  if (e == 0) return 0ull;  // zero (masses flush denormals)
  if (sh >= 0) return (unsigned long long)m << sh;
  return sh > -32 ? (unsigned long long)(m >> -sh) : 0ull;
}

static_assert(kScanThreads / 32 == kScanVecs, "warp i sums vector i of the CTA");

__device__ __forceinline__ unsigned long long warp_sum_u64(unsigned long long x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// inclusive scan over the CTA's 256 threads in thread order (exact: integers)
__device__ __forceinline__ unsigned long long block_scan_u64(unsigned long long x,
                                                             unsigned long long* wsc) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsc[warp] = x;
  __syncthreads();
  unsigned long long off = 0;
  for (int w = 0; w < warp; ++w) off += wsc[w];
  __syncthreads();
  return off + x;
}

template <typename T, bool kAligned>
__global__ void __launch_bounds__(kScanThreads, 4) sample_kernel(SampleArgs a, int row_base) {
  __shared__ SampleSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int row = row_base + (int)blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int VW = ScanTraits<T>::kVW;
  const int V = a.V;
  const float cs = a.scale_log2;
  const float NEG_INF = __int_as_float(0xff800000);
  pdl_launch_dependents();
  pdl_wait();
  cluster_arrive_relaxed();
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)row * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);

  // the row's tree, fetched while the logits are in flight: every CTA needs
  // the tokens of v's children (they leave its chunk of the residual)
  int b;
  {
    int lo = 0, hi = a.B - 1;  // last b with node_off[b] <= row
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (__ldg(a.node_off + mid) <= row) lo = mid; else hi = mid - 1;
    }
    b = lo;
  }
  const int off = __ldg(a.node_off + b);
  const int n = __ldg(a.node_off + b + 1) - off;
  // a row outside its tree's own extent belongs to no tree and draws no ticket
  const bool bad_tree = (n < 1 || n > 256 || off < 0 || off + n > a.n_total || row < off ||
                         row >= off + n);
  int v_par = -1, v_tok = 0;
  if (!bad_tree && tid < n) {
    v_par = __ldg(a.parent + off + tid);
    v_tok = __ldg(a.token + off + tid);
  }
  const int v = row - off;
  const bool child = !bad_tree && tid < n && tid > v && v_par == v;
  const bool tok_ok = v_tok >= 0 && v_tok < V;
  // leader: the child's own logit, in flight during the exchanges below
  float l_child = 0.f;
  if (crank == 0 && child && tok_ok) l_child = load_elem<T>(rowp, v_tok);
  sm.excl[tid] = 0ull;
  sm.par[tid] = v_par;
  sm.tok[tid] = v_tok;
  if (tid == 0) sm.best = 0ull;
  const float wm = warp_max_f32(scan_thread_max<T>(buf));
  if (lane == 0) sm.red_m[warp] = wm;
  __syncthreads();
  if (child && v_tok >= c0 && v_tok < c1) {  // this CTA holds the child's token
    const int rel = v_tok - c0, vi = rel / VW;
    const int i = vi / kScanThreads, t = vi - i * kScanThreads, j = rel - vi * VW;
    atomicOr(&sm.excl[t], 1ull << (i * VW + j));
  }
  float cm = sm.red_m[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) cm = fmaxf(cm, sm.red_m[w]);
  cluster_wait();  // every CTA of the cluster runs: remote stores are safe
  if (tid == 0)
    for (int r = 0; r < C; ++r) cluster.map_shared_rank(&sm, r)->cmax[crank] = cm;
  cluster_arrive_release();
  cluster_wait_acquire();
  float M = sm.cmax[0];
  for (int r = 1; r < C; ++r) M = fmaxf(M, sm.cmax[r]);
  if (M == NEG_INF) M = 0.f;  // every mass is then 0

  // Residual masses.  One vector's masses are summed in fp32 in lane order
  // and then taken as fixed point: the exact integer prefix runs over
  // (CTA, vector, thread), and inside a vector the draw compares against the
  // same fp32 running sums, so the ranges still partition the residual
  // exactly.  2^(-inf) = 0 covers the padding; only the few threads that
  // hold a child's token test the exclusion bits.
  const unsigned long long mask = sm.excl[tid];
  auto vec_masses = [&](const uint4& q, int i, float (&e)[VW]) {
    const float2 nm2 = make_float2(-M, -M), c2 = make_float2(cs, cs);
#pragma unroll
    for (int w = 0; w < VW / 2; ++w) {
      const float2 y = __fmul2_rn(__fadd2_rn(vec_pair<T>(q, w), nm2), c2);
      e[2 * w] = ex2(y.x);
      e[2 * w + 1] = ex2(y.y);
    }
    if (mask != 0ull) {
#pragma unroll
      for (int j = 0; j < VW; ++j)
        if ((mask >> (i * VW + j)) & 1ull) e[j] = 0.f;
    }
  };
  auto vec_mass = [&](const uint4& q, int i) -> unsigned long long {
    float e[VW];
    vec_masses(q, i, e);
    float acc = 0.f;
#pragma unroll
    for (int j = 0; j < VW; ++j) acc += e[j];
    return to_fixed(acc);
  };
  unsigned long long own = 0ull;
#pragma unroll
  for (int i = 0; i < kScanVecs; ++i) {
    const unsigned long long w = vec_mass(buf[i], i);
    sm.sv[i][tid] = w;
    own += w;
  }
  const unsigned long long wtot = warp_sum_u64(own);
  if (lane == 0) sm.wsc[warp] = wtot;
  __syncthreads();
  unsigned long long ctotal = 0ull;
#pragma unroll
  for (int w = 0; w < 8; ++w) ctotal += sm.wsc[w];
  if (tid == 0)
    for (int r = 0; r < C; ++r) cluster.map_shared_rank(&sm, r)->ctot[crank] = ctotal;
  cluster_arrive_release();
  cluster_wait_acquire();
  unsigned long long R = 0ull, coff = 0ull;
  for (int r = 0; r < C; ++r) {
    if (r == crank) coff = R;
    R += sm.ctot[r];
  }

  // ---- bonus draw at v (used if the walk ends at v): the token holding
  //      residual mass floor(u[v, 1] R) in token order
  bool owner = false;  // this CTA holds the draw (uniform over it)
  if (R > 0ull) {
    const double t = floor((double)__ldg(a.u + 2 * (size_t)row + 1) * (double)R);
    const unsigned long long tgt =
        !(t > 0.0) ? 0ull : (t >= (double)R ? R - 1ull : (unsigned long long)t);
    owner = tgt >= coff && tgt - coff < sm.ctot[crank];
    if (owner) {
      // this CTA's per-vector totals (warp i sums vector i), then the vector
      // holding the draw
      {
        unsigned long long t = 0ull;
#pragma unroll
        for (int k = 0; k < kScanThreads / 32; ++k) t += sm.sv[warp][lane + 32 * k];
        t = warp_sum_u64(t);
        if (lane == 0) sm.vtot[warp] = t;
      }
      __syncthreads();
      unsigned long long rem = tgt - coff;
      int vi = 0;
      while (vi < kScanVecs - 1 && rem >= sm.vtot[vi]) rem -= sm.vtot[vi++];
      const uint4 q = buf_vec(buf, vi);
      const unsigned long long x = sm.sv[vi][tid];
      const unsigned long long incl = block_scan_u64(x, sm.wsc);
      if (x > 0ull && rem >= incl - x && rem < incl) {  // exactly one thread
        const unsigned long long base = incl - x;
        float e[VW];
        vec_masses(q, vi, e);
        float acc = 0.f;
        int pos = -1;
#pragma unroll
        for (int j = 0; j < VW; ++j) {
          acc += e[j];
          if (pos < 0 && rem < base + to_fixed(acc)) pos = c0 + (vi * kScanThreads + tid) * VW + j;
        }
        a.bcand[row] = pos;
        __threadfence();
      }
    }
  }

  // ---- leader: the decisions of v's children
  if (crank == 0) {
    unsigned long long wc = 0ull;
    bool dup = false;
    if (child) {
      if (!tok_ok) {
        raise_status(a.status, kStIndex);
        dup = true;  // no mass: never accepted
      } else {
        wc = to_fixed(ex2((l_child - M) * cs));
        for (int j = v + 1; j < tid && !dup; ++j) dup = (sm.par[j] == v && sm.tok[j] == v_tok);
        if (R == 0ull && !dup) atomicMax(&sm.best, make_key(l_child, (uint32_t)v_tok));
      }
    }
    const unsigned long long q = (child && !dup) ? wc : 0ull;
    const unsigned long long before = block_scan_u64(q, sm.wsc) - q;  // earlier siblings
    unsigned long long chs = 0ull;  // the distinct children's mass (warp totals of the scan)
#pragma unroll
    for (int w = 0; w < 8; ++w) chs += sm.wsc[w];
    const unsigned long long S = R + chs;  // the row's full mass
    if (child) {
      const bool flag = !dup && ((double)__ldg(a.u + 2 * (size_t)(off + tid)) *
                                     (double)(S - before) <
                                 (double)wc);
      a.flag[off + tid] = flag ? 1 : 0;
      __threadfence();
    }
    // no residual mass in fixed point (the children hold all of it): the
    // most likely child's token, as exact arithmetic would have accepted it
    if (R == 0ull && tid == 0) {
      a.bcand[row] = sm.best ? (int)key_index(sm.best) : -1;
      __threadfence();
    }
  }
  // Two tickets per row: the leader's (its children's flags) and the owner
  // CTA's (the bonus candidate; the leader's too when there is no residual
  // mass).  The CTA that draws the tree's last one walks it.
  const int mine = (crank == 0 ? 1 : 0) + (owner ? 1 : 0) + (crank == 0 && R == 0ull ? 1 : 0);
  if (mine == 0) return;
  if (bad_tree) {
    if (crank == 0 && tid == 0) raise_status(a.status, kStTree);
    return;  // a malformed extent never touches the tickets
  }
  __syncthreads();
  if (tid == 0) {
    // release: this CTA's flags / candidate (fenced above) reach the CTA
    // that draws the last ticket; acquire: that CTA sees every other row's
    const int t = atom_add_acq_rel_gpu(&a.tickets[b], mine);
    sm.last = (t + mine == 2 * n);
    if (sm.last) a.tickets[b] = 0;  // ready for the next call
  }
  __syncthreads();
  if (!sm.last) return;

  // this tree's flags and candidates; their slots go back to zero, so that
  // with the ticket the whole workspace is zero again for the next call
  const int f = (tid > 0 && tid < n) ? __ldcg(a.flag + off + tid) : 0;
  const int cand = tid < n ? __ldcg(a.bcand + off + tid) : 0;
  if (tid < n) {
    a.flag[off + tid] = 0;
    a.bcand[off + tid] = 0;
  }
  // ---- walk of tree b along the first accepted child of every node
  const bool bad = (tid < n) && (tid == 0 ? (v_par != -1) : (v_par < 0 || v_par >= tid));
  if (__syncthreads_or(bad)) {
    if (tid == 0) raise_status(a.status, kStTree);
    return;
  }
  sm.next[tid] = 0x7FFFFFFF;
  if (tid < n) sm.tok[tid] = cand;  // the tokens are not needed any more
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
      sm.last = -1;
    } else {
      int x = w;
      for (int d = A; d >= 0; --d) {
        path[d] = x;
        x = sm.par[x];
      }
      a.accept_len[b] = A;
      a.bonus[b] = sm.tok[w];
      sm.last = A;
    }
  }
  __syncthreads();
  if (sm.last < 0) return;
  for (int d = sm.last + 1 + tid; d < a.path_cap; d += kScanThreads) path[d] = -1;
}

template <typename T, bool kAligned>
cudaError_t launch_sample_t(const SampleArgs& a, int C, cudaStream_t s) {
  auto kern = sample_kernel<T, kAligned>;
  if (C > 8) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kScanThreads, 1, 1);
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  for (int r0 = 0; r0 < a.n_total; r0 += 65535) {
    cfg.gridDim = dim3(C, min(65535, a.n_total - r0), 1);
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, a, r0);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}
}  // namespace

size_t sample_ws_bytes(int B, int n_total) {
  const size_t a4 = ((size_t)n_total * 4 + 255) / 256 * 256;
  const size_t b4 = ((size_t)B * 4 + 255) / 256 * 256;
  return 2 * a4 + b4;
}

void sample_ws_carve(SampleArgs& a, void* ws, int B, int n_total) {
  const size_t a4 = ((size_t)n_total * 4 + 255) / 256 * 256;
  char* p = static_cast<char*>(ws);
  a.flag = reinterpret_cast<int32_t*>(p);
  a.bcand = reinterpret_cast<int32_t*>(p + a4);
  a.tickets = reinterpret_cast<int32_t*>(p + 2 * a4);
  (void)B;
}

cudaError_t launch_accept_sample(const SampleArgs& a, cudaStream_t s) {
  const int C = scan_cluster_size(a.V, a.is_bf16, a.n_total, device_sm_count());
  const int esz = a.is_bf16 ? 2 : 4;
  const bool aligned = ((reinterpret_cast<uintptr_t>(a.logits) & 15) == 0) &&
                       (((a.ld * esz) & 15) == 0);
  if (a.is_bf16)
    return aligned ? launch_sample_t<__nv_bfloat16, true>(a, C, s)
                   : launch_sample_t<__nv_bfloat16, false>(a, C, s);
  return aligned ? launch_sample_t<float, true>(a, C, s) : launch_sample_t<float, false>(a, C, s);
}

}  // namespace tg
