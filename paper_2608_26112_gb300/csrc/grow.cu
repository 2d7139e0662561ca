// grow: one drafting step of TreeGraft's shared-tree construction
// (Algorithm 2; a schedule of small-drafter steps only is Algorithm 1).
//
// Every tree of the batch grows in lock step (one schedule), so the node
// count n, the candidate pool [pool_lo, n) and the frontier size
// |F| = min(W, n - pool_lo) are known on the host.  The pool is a contiguous
// range in both branches of Algorithm 2: a small step pools the nodes the
// previous step made, N_k = [new_lo, n); a middle step pools V(T) \ P, and
// P is always a prefix [0, |P|) of the node ids - P only grows at middle
// steps, where it becomes P u (V \ P) = V, and nodes are only ever appended.
//
// Small step (a = 0), two launches:
//   grow_select   Top_W of the pool by (s desc, id asc) -> frontier F, and the
//                 expansion rows with their path scores;
//   expand_topk   Top_m of each frontier row of the small drafter's table
//                 (log-softmax, token ids, fp32(s(v) + p(u))), the children
//                 appended straight into the tree at n, n + 1, ... in
//                 frontier order, then child rank.
// Middle step (a = 1), two launches:
//   expand_topk   log-sum-exp and Top_m of every pool row (the drafter's
//                 forward over C, whose logits are then reused for F), the
//                 rows of each tree's pool [pool_lo, n) mapped in the kernel;
//   grow_select   caches each pool row's lse, rescores every non-root pool
//                 node p(v) = l_m[pa(v), token(v)] - lse_m[pa(v)], recomputes
//                 s root-first, takes Top_W of the pool and appends the
//                 frontier's children; P u= C is the caller's |P| = n.
// One CTA of up to 1024 threads per tree (one thread per node) for select
// and append.  Latency-bound: the scans of expand_topk move the bytes.
#include "common.cuh"
#include "launch.h"

namespace tg {
namespace {

constexpr int kGrowThreads = 1024;

__device__ __forceinline__ float logit_at(const void* logits, int is_bf16, int64_t ld, size_t row,
                                          int col) {
  if (is_bf16) {
    const uint16_t h = reinterpret_cast<const uint16_t*>(logits)[row * (size_t)ld + col];
    return __uint_as_float((uint32_t)h << 16);
  }
  return reinterpret_cast<const float*>(logits)[row * (size_t)ld + col];
}

__global__ void __launch_bounds__(kGrowThreads) grow_select_kernel(GrowArgs a) {
  __shared__ float score_s[kGrowThreads];
  __shared__ int par_s[kGrowThreads];
  __shared__ uint64_t key_s[kGrowThreads];
  __shared__ int front_s[kGrowThreads];
  __shared__ int red_i[32];
  const int b = blockIdx.x;
  const int v = threadIdx.x, lane = v & 31, warp = v >> 5;
  const int n = a.n, lo = a.pool_lo, nc = n - lo;
  const int nf = min(a.W, nc);
  const size_t base = (size_t)b * a.cap;
  pdl_launch_dependents();
  pdl_wait();
  const bool in_tree = v < n, in_pool = v >= lo && v < n;
  int p = -1, bad = 0;
  float s = 0.f;
  if (in_tree) {
    p = a.parent[base + v];
    s = a.score[base + v];
    bad = (v == 0) ? (p != -1) : (p < 0 || p >= v);
    par_s[v] = p;
  }
  if (__syncthreads_or(bad)) {
    if (v == 0) raise_status(a.status, kStTree);
    return;
  }
  if (a.mode == 1) {
    // cache the pool rows' log-sum-exp (the middle drafter's forward over C)
    if (in_pool) a.lse_mid[base + v] = a.ws_lse[(size_t)b * nc + (v - lo)];
    __syncthreads();
    // rescore every non-root pool node from its parent's middle row
    float e = 0.f;
    int bad_tok = 0;
    if (in_pool && v > 0) {
      const int t = a.token[base + v];
      if (t < 0 || t >= a.V) {
        bad_tok = 1;
      } else {
        const float l = logit_at(a.logits, a.is_bf16, a.ld, base + p, t);
        e = __fsub_rn(l, a.lse_mid[base + p]);
        a.edge[base + v] = e;
      }
    }
    if (__syncthreads_or(bad_tok)) {
      if (v == 0) raise_status(a.status, kStIndex);
      return;
    }
    // s(v) = fp32(s(pa(v)) + p(v)) root-first for the pool; nodes below the
    // pool keep theirs.  Depth by walking up; one barrier per level.
    int d = 0;
    if (in_pool) {
      for (int w = v; w != 0; w = par_s[w]) ++d;
    }
    int dmax = d;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dmax = max(dmax, __shfl_xor_sync(0xffffffffu, dmax, o));
    if (lane == 0) red_i[warp] = dmax;
    if (in_tree) score_s[v] = s;
    __syncthreads();
    dmax = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) dmax = max(dmax, red_i[w]);
    for (int lvl = 1; lvl <= dmax; ++lvl) {
      if (in_pool && v > 0 && d == lvl) score_s[v] = __fadd_rn(score_s[p], e);
      __syncthreads();
    }
    if (in_pool) {
      s = score_s[v];
      a.score[base + v] = s;
    }
  } else {
    if (in_tree) score_s[v] = s;
  }
  // Top_W of the pool: each candidate counts the candidates with a larger
  // (score, -id) key; that count is its frontier slot
  key_s[v] = in_pool ? make_key(s, (uint32_t)v) : 0ull;
  __syncthreads();
  if (in_pool) {
    const uint64_t mine = key_s[v];
    int rank = 0;
    for (int w = lo; w < n; ++w) rank += (key_s[w] > mine) ? 1 : 0;
    if (rank < nf) {
      front_s[rank] = v;
      a.frontier[(size_t)b * a.W + rank] = v;
      if (a.mode == 0) {
        a.ws_row[(size_t)b * nf + rank] = (int)(base + v);
        a.ws_ps[(size_t)b * nf + rank] = s;
      }
    }
  }
  for (int r = nf + v; r < a.W; r += blockDim.x) a.frontier[(size_t)b * a.W + r] = -1;
  if (a.mode == 0) return;
  // middle step: append the frontier's children from the pool rows' Top_m
  __syncthreads();
  const int m = a.m;
  for (int item = v; item < nf * m; item += blockDim.x) {
    const int i = item / m, r = item - i * m;
    const int f = front_s[i];
    const size_t src = ((size_t)b * nc + (f - lo)) * m + r;
    const size_t u = base + n + item;
    const float e = a.ws_lp[src];
    a.parent[u] = f;
    a.token[u] = a.ws_tok[src];
    a.edge[u] = e;
    a.score[u] = __fadd_rn(score_s[f], e);
  }
}

cudaError_t launch_pdl(const void* fn, dim3 grid, dim3 block, const GrowArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {const_cast<GrowArgs*>(&a)};
  return cudaLaunchKernelExC(&cfg, fn, args);
}

}  // namespace

size_t grow_ws_bytes(int B, int cap, int m) {
  const size_t rows = (size_t)B * cap;
  const size_t a = (rows * 4 + 255) / 256 * 256;       // int32 row list / fp32 per row
  const size_t am = (rows * m * 4 + 255) / 256 * 256;  // per (row, child)
  return 3 * a + 3 * am;                               // row, ps, lse; tok, lp, sc
}

void grow_ws_carve(GrowArgs& a, void* ws, int B, int cap, int m) {
  const size_t rows = (size_t)B * cap;
  const size_t sa = (rows * 4 + 255) / 256 * 256;
  const size_t sam = (rows * m * 4 + 255) / 256 * 256;
  char* p = static_cast<char*>(ws);
  a.ws_row = reinterpret_cast<int32_t*>(p);
  a.ws_ps = reinterpret_cast<float*>(p + sa);
  a.ws_lse = reinterpret_cast<float*>(p + 2 * sa);
  a.ws_tok = reinterpret_cast<int32_t*>(p + 3 * sa);
  a.ws_lp = reinterpret_cast<float*>(p + 3 * sa + sam);
  a.ws_sc = reinterpret_cast<float*>(p + 3 * sa + 2 * sam);
}

cudaError_t launch_grow_step(const GrowArgs& a, cudaStream_t s) {
  const int nc = a.n - a.pool_lo, nf = min(a.W, nc);
  TopkArgs t = {};
  t.logits = a.logits;
  t.is_bf16 = a.is_bf16;
  t.logit_rows = a.B * a.cap;
  t.V = a.V;
  t.ld = a.ld;
  t.k = a.m;
  t.status = a.status;
  t.gcap = a.cap;
  const dim3 sel_grid(a.B), sel_block((unsigned)((a.n + 31) / 32 * 32));
  cudaError_t e;
  if (a.mode == 0) {
    e = launch_pdl(reinterpret_cast<const void*>(grow_select_kernel), sel_grid, sel_block, a, s);
    if (e != cudaSuccess) return e;
    // row b * nf + i = frontier node i of tree b (ws_row), its children
    // appended to the tree
    t.rows = a.B * nf;
    t.row_idx = a.ws_row;
    t.parent_score = a.ws_ps;
    t.gdiv = nf;
    t.app_n = a.n;
    t.app_parent = a.parent;
    t.app_token = a.token;
    t.app_edge = a.edge;
    t.app_score = a.score;
    return launch_expand_topk(t, s);
  }
  // row b * nc + j = pool node pool_lo + j of tree b; zero parent scores (the
  // children's scores come from the rescored s in grow_select)
  t.rows = a.B * nc;
  t.gdiv = nc;
  t.goff = a.pool_lo;
  t.tok = a.ws_tok;
  t.logprob = a.ws_lp;
  t.lse_out = a.ws_lse;
  e = launch_expand_topk(t, s);
  if (e != cudaSuccess) return e;
  return launch_pdl(reinterpret_cast<const void*>(grow_select_kernel), sel_grid, sel_block, a, s);
}

}  // namespace tg
