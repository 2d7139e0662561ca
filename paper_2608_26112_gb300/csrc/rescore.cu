// rescore_select: stronger-drafter rescoring of the candidate pool and the
// global top-N reselection of grafting positions (Sec. 3.2 expanded
// grafting-position selection; Algorithm 2, middle-drafter branch).
//
// One CTA of 256 threads per tree, one thread per node:
//   edge[v]  = strong_lp[pa(v), token(v)] for unvisited non-root v, else the
//              stored edge; the root's edge is 0 and s(root) = 0 (log of 1);
//   score[v] = score[pa(v)] + edge[v] in fp32, filled level by level so every
//              node adds onto its parent's final value - the same rounding
//              as the root-first definition;
//   selected = top-N of the unvisited nodes by (score desc, id asc): each
//              candidate counts the candidates with a larger 64-bit key, and
//              that count is its output slot.
// The work is a 64-value gather plus a few hundred shared-memory ops: the
// kernel is latency bound.
#include "common.cuh"
#include "launch.h"

namespace tg {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads) rescore_select_kernel(RescoreArgs a) {
  __shared__ int par_s[256];
  __shared__ float score_s[256];
  __shared__ uint64_t key_s[256];
  __shared__ int red_i[8];
  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_launch_dependents();
  pdl_wait();
  const int o_lo = a.node_off[b], o_hi = a.node_off[b + 1];
  const int off = o_lo;
  const int n = o_hi - o_lo;
  if (n < 1 || n > 256 || off < 0 || off + n > a.n_total) {
    if (tid == 0) raise_status(a.status, kStTree);
    return;
  }
  // rows outside every tree (node_off[0] > 0 or node_off[B] < n_total)
  // belong to no result; the trees themselves are still computed
  if (tid == 0 && ((b == 0 && o_lo != 0) || (b == a.B - 1 && o_hi != a.n_total)))
    raise_status(a.status, kStTree);
  const int v = tid;
  // every per-node input is requested at once; only the strong-row gather
  // depends on them (parent and token)
  int p = -1, bad = 0, t = 0;
  float e = 0.f, w_edge = 0.f;
  bool cand = false;
  if (v < n) {
    p = a.parent[off + v];
    cand = a.visited[off + v] == 0;
    t = a.token[off + v];
    w_edge = a.weak_edge[off + v];
    bad = (v == 0) ? (p != -1) : (p < 0 || p >= v);
    par_s[v] = p;
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) raise_status(a.status, kStTree);
    return;
  }
  int bad_tok = 0;
  if (v > 0 && v < n) {
    if (cand) {
      if (t < 0 || t >= a.V) {
        bad_tok = 1;
      } else {
        e = a.strong_lp[(size_t)(off + p) * (size_t)a.ld + t];
      }
    } else {
      e = w_edge;
    }
  }
  if (__syncthreads_or(bad_tok)) {
    if (tid == 0) raise_status(a.status, kStIndex);
    return;
  }
  // depth by walking up (parent[v] < v bounds the walk)
  int d = 0;
  if (v < n) {
    int w = v;
    while (w != 0) {
      w = par_s[w];
      ++d;
    }
    if (v == 0) score_s[0] = 0.f;
  }
  int dmax = d;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) dmax = max(dmax, __shfl_xor_sync(0xffffffffu, dmax, o));
  if (lane == 0) red_i[warp] = dmax;
  __syncthreads();
  dmax = red_i[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) dmax = max(dmax, red_i[w]);
  for (int lvl = 1; lvl <= dmax; ++lvl) {
    if (v < n && d == lvl) score_s[v] = __fadd_rn(score_s[p], e);
    __syncthreads();
  }
  float s = 0.f;
  if (v < n) {
    s = score_s[v];
    a.edge_out[off + v] = e;
    a.score_out[off + v] = s;
  }
  key_s[v] = cand ? make_key(s, (uint32_t)v) : 0ull;
  const int ncand = __syncthreads_count(cand);
  if (cand) {
    const uint64_t mine = key_s[v];
    int rank = 0;
    for (int u = 0; u < n; ++u) rank += (key_s[u] > mine) ? 1 : 0;
    if (rank < a.N) a.selected[(size_t)b * a.N + rank] = v;
  }
  for (int i = ncand + tid; i < a.N; i += kThreads) a.selected[(size_t)b * a.N + i] = -1;
  if (tid == 0) a.n_selected[b] = min(ncand, a.N);
}

}  // namespace

cudaError_t launch_rescore_select(const RescoreArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.B, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, rescore_select_kernel, a);
}

}  // namespace tg
