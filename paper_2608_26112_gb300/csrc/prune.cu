// global_prune: global score-based pruning with ancestor closure and the
// verification buffers (Algorithm 3).
//
// One CTA of 1024 threads per tree, one thread per node:
//   1. depth d(v) by walking parent pointers (parent[v] < v bounds the walk);
//   2. the non-root nodes ranked under (-s(v), d(v), id(v)) by a bitonic
//      sort of exact 64-bit keys (score order as an unsigned image, then
//      1023 - depth, then 1023 - id) in shared memory;
//   3. the greedy closure over the ranked nodes: the chain from v up to the
//      first kept node is added whole when |K| + |chain| <= M, and the loop
//      stops at |K| = M.  When every node ranks after its parent - its score
//      does not exceed its parent's, as for sums of log-probabilities -
//      every chain is the node alone and the result is the root plus the
//      first M - 1 ranked nodes, marked in parallel; otherwise thread 0 runs
//      the loop;
//   4. the kept nodes are re-indexed in their original order (a block-wide
//      ballot scan), then every kept node writes its id, new parent,
//      position id (its depth) and mask row; every kept leaf writes its
//      root-to-leaf retrieval path.
// A tree with at most M = budget + 1 nodes is kept whole.
#include "common.cuh"
#include "launch.h"

namespace tg {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kMaskWords = 8;  // kept trees have at most 256 nodes

struct PruneSmem {
  int par[kThreads];
  int depth[kThreads];
  int order[kThreads];
  int newidx[kThreads];
  uint64_t key[kThreads];
  uint32_t mask[256][kMaskWords];
  unsigned char in_k[kThreads];
  unsigned char has_kid[kThreads];
  int warp_cnt[kWarps];
};

// exclusive block-wide prefix count of `flag` (1024 threads); returns the
// thread's offset and leaves the total in *total
__device__ __forceinline__ int block_scan(bool flag, int* warp_cnt, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned b = __ballot_sync(0xffffffffu, flag);
  const int in_warp = __popc(b & ((1u << lane) - 1u));
  if (lane == 0) warp_cnt[warp] = __popc(b);
  __syncthreads();
  int before = 0, all = 0;
  for (int w = 0; w < kWarps; ++w) {
    const int c = warp_cnt[w];
    before += (w < warp) ? c : 0;
    all += c;
  }
  *total = all;
  __syncthreads();  // warp_cnt can be reused
  return before + in_warp;
}

__global__ void __launch_bounds__(kThreads, 1) global_prune_kernel(PruneArgs a) {
  __shared__ PruneSmem sm;
  const int b = blockIdx.x;
  const int v = threadIdx.x;
  pdl_launch_dependents();
  pdl_wait();
  const int off = a.node_off[b];
  const int n = a.node_off[b + 1] - off;
  const int M = a.budget + 1;
  const int Mo = a.stride;
  const int W = (Mo + 31) / 32;
  if (n < 1 || n > kThreads || off < 0 || off + n > a.n_total) {
    if (v == 0) raise_status(a.status, kStTree);
    return;
  }
  // rows outside every tree (node_off[0] > 0 or node_off[B] < n_total)
  // belong to no result; the trees themselves are still pruned
  if (v == 0 && ((b == 0 && off != 0) || (b == a.B - 1 && off + n != a.n_total)))
    raise_status(a.status, kStTree);
  // ---- tree, validation, depth
  int p = -1;
  float s = 0.f;
  if (v < n) {
    p = a.parent[off + v];
    s = a.score[off + v];
    sm.par[v] = p;
  }
  const bool bad = (v < n) && (v == 0 ? (p != -1) : (p < 0 || p >= v));
  sm.in_k[v] = 0;
  sm.has_kid[v] = 0;
  if (__syncthreads_or(bad)) {
    if (v == 0) raise_status(a.status, kStTree);
    return;
  }
  int d = 0;
  if (v < n) {
    for (int w = v; w != 0; w = sm.par[w]) ++d;
    sm.depth[v] = d;
  }
  if (n <= M) {
    if (v < n) sm.in_k[v] = 1;
  } else {
    // ---- ranking under (-s, d, id): bitonic sort of the keys (descending)
    // over the next power of two >= n; slot 0 (the root) and the padding
    // hold key 0 and sort last
    const uint64_t key = (v >= 1 && v < n)
                             ? ((uint64_t)ord_f32(s) << 20) | ((uint64_t)(1023 - d) << 10) |
                                   (uint64_t)(1023 - v)
                             : 0ull;
    int np2 = 32;
    while (np2 < n) np2 <<= 1;
    sm.key[v] = key;
    const bool parent_first = (v < 1 || v >= n || p == 0);
    __syncthreads();
    // every non-root node ranks after its parent (its score does not exceed
    // the parent's): then each ranked node's chain is the node alone
    const bool monotone =
        __syncthreads_and(parent_first || sm.key[p] > key);
    // each thread keeps its slot's key in a register: partners 32 or more
    // slots away are exchanged through shared memory, closer ones by shuffle
    uint64_t x = key;
    for (int k = 2; k <= np2; k <<= 1) {
      for (int j = k >> 1; j > 0; j >>= 1) {
        uint64_t y;
        if (j >= 32) {
          sm.key[v] = x;
          __syncthreads();
          y = sm.key[v ^ j];
          __syncthreads();
        } else {
          y = __shfl_xor_sync(0xffffffffu, x, j);
        }
        // descending runs where bit k of the slot is 0; the lower slot of a
        // pair keeps the larger key in a descending run
        const bool keep_max = ((v & k) == 0) == ((v & j) == 0);
        x = keep_max ? (x > y ? x : y) : (x < y ? x : y);
      }
    }
    if (v < n - 1) sm.order[v] = 1023 - (int)(x & 1023u);
    __syncthreads();
    if (monotone) {
      // Algorithm 3 then keeps the root and the first M - 1 ranked nodes:
      // each one's parent is the root or ranked earlier, so already kept
      if (v == 0) sm.in_k[0] = 1;
      if (v < M - 1 && v < n - 1) sm.in_k[sm.order[v]] = 1;
    } else if (v == 0) {
      // ---- greedy closure over the ranked nodes
      sm.in_k[0] = 1;
      int cnt = 1;
      int nxt = sm.order[0];
      for (int i = 0; i < n - 1 && cnt < M; ++i) {
        const int u = nxt;
        if (i + 1 < n - 1) nxt = sm.order[i + 1];
        int c = 0;
        for (int w = u; !sm.in_k[w]; w = sm.par[w]) ++c;
        if (cnt + c <= M) {
          for (int w = u; !sm.in_k[w]; w = sm.par[w]) sm.in_k[w] = 1;
          cnt += c;
        }
      }
    }
  }
  __syncthreads();

  // ---- re-index in the original order
  const bool kept = (v < n) && sm.in_k[v];
  int n_kept = 0;
  const int ni = block_scan(kept, sm.warp_cnt, &n_kept);
  if (kept) {
    sm.newidx[v] = ni;
    if (v != 0) sm.has_kid[p] = 1;
  }
  __syncthreads();
  const size_t base = (size_t)b * Mo;
  if (kept) {
    a.kept[base + ni] = v;
    a.new_parent[base + ni] = (v == 0) ? -1 : sm.newidx[p];
    a.position[base + ni] = d;
    uint32_t* row = sm.mask[ni];
    for (int j = 0; j < kMaskWords; ++j) row[j] = 0u;
    for (int w = v;; w = sm.par[w]) {
      const int k = sm.newidx[w];
      row[k >> 5] |= 1u << (k & 31);
      if (w == 0) break;
    }
  }
  if (v >= n_kept && v < Mo) {  // padding rows (disjoint from the kept rows)
    a.kept[base + v] = -1;
    a.new_parent[base + v] = -1;
    a.position[base + v] = -1;
  }
  const bool leaf = kept && !sm.has_kid[v];
  int n_leaf = 0;
  const int li = block_scan(leaf, sm.warp_cnt, &n_leaf);  // also orders the mask rows above
  // mask rows: kept rows from shared memory, the rest zero
  for (int i = v; i < Mo * W; i += kThreads) {
    const int r = i / W, w = i % W;
    a.mask[base * W + i] = (r < n_kept) ? sm.mask[r][w] : 0u;
  }
  // retrieval paths: one row per leaf, root first, -1 padded; other rows -1
  const size_t pbase = base * (size_t)a.path_cap;
  if (leaf) {
    int32_t* row = a.paths + pbase + (size_t)li * a.path_cap;
    if (d + 1 > a.path_cap) raise_status(a.status, kStIndex);
    for (int t = d + 1; t < a.path_cap; ++t) row[t] = -1;
    int t = d;
    for (int w = v;; w = sm.par[w], --t) {
      if (t < a.path_cap) row[t] = sm.newidx[w];
      if (w == 0) break;
    }
  }
  for (int i = n_leaf * a.path_cap + v; i < Mo * a.path_cap; i += kThreads) a.paths[pbase + i] = -1;
  if (v == 0) {
    a.n_kept[b] = n_kept;
    a.n_paths[b] = n_leaf;
  }
}

}  // namespace

cudaError_t launch_global_prune(const PruneArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.B, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, global_prune_kernel, a);
}

}  // namespace tg
