// accept: greedy longest-accepted-path walk at temperature 0 (verification
// step of Algorithms 1 and 2; greedy decoding setting of Appendix E).
//
// One launch.  Grid (C, n_total), clusters of C CTAs along x: each cluster
// computes the target argmax (lowest token on ties) of one node row over
// DSMEM, and its leader stores it in scratch and takes a ticket for the
// row's tree.  The leader that draws the tree's last ticket performs the
// walk for that tree with its 256 threads (one per node):
//   ok[v]   = token[v] == am[pa(v)]
//   full[v] = AND of ok over the root..v chain, depth[v] = its length
//   a*      = argmax over full nodes of (depth, -id)
// then writes the root..a* path, A = depth(a*) and the bonus token am[a*].
// The walker returns the ticket and the tree's argmax slots to zero, so the
// scratch is all zero again for the next call, whatever its shape.
// Every node's row is scanned because the bonus token needs the row of a*,
// which may be any node (a leaf included).
#include <cooperative_groups.h>

#include "launch.h"
#include "rowscan.cuh"

namespace cg = cooperative_groups;

namespace tg {
namespace {

struct AcceptSmem {
  float red_v[8];
  uint64_t recv_key[16];  // leader only: per-CTA (max, first position) keys of the row
  int minpos;
  int last;
  int par[256];
  int am[256];
  int tok[256];
  uint32_t key[8];
};

template <typename T, bool kAligned>
__global__ void __launch_bounds__(kScanThreads, 4) accept_kernel(AcceptArgs a, int row_base) {
  __shared__ AcceptSmem sm;
  cg::cluster_group cluster = cg::this_cluster();
  const int C = (int)cluster.num_blocks();
  const int crank = (int)cluster.block_rank();
  const int row = row_base + (int)blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int VW = ScanTraits<T>::kVW;
  const int V = a.V;
  pdl_launch_dependents();
  pdl_wait();
  cluster_arrive_relaxed();
  const int per = ((V + C - 1) / C + VW - 1) / VW * VW;
  const int c0 = min(V, crank * per);
  const int c1 = min(V, c0 + per);
  const T* rowp = reinterpret_cast<const T*>(a.logits) + (size_t)row * (size_t)a.ld;

  uint4 buf[kScanVecs];
  scan_load<T, kAligned>(rowp, c0, c1, buf);

  // The leader resolves the row's tree and fetches the tree's parent and
  // token arrays while the logits are in flight (any leader may turn out to
  // be the one that walks the tree).
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
  if (tid == 0) sm.minpos = 0x7FFFFFFF;
  // chunk max, then the lowest position holding it (only threads that hold it search)
  const float tmax = scan_thread_max<T>(buf);
  const float wm = warp_max_f32(tmax);
  if (lane == 0) sm.red_v[warp] = wm;
  __syncthreads();
  float cmax = sm.red_v[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) cmax = fmaxf(cmax, sm.red_v[w]);
  if (tmax == cmax && c0 + (int)tid * VW < c1) {
    const int fp = scan_first_pos<T>(buf, c0, c1, cmax);
    if (fp != 0x7FFFFFFF) atomicMin(&sm.minpos, fp);
  }
  __syncthreads();
  cluster_wait();
  if (tid == 0) {
    const int mp = sm.minpos;
    cluster.map_shared_rank(&sm, 0)->recv_key[crank] =
        (mp == 0x7FFFFFFF) ? 0ull : make_key(cmax, (uint32_t)mp);
  }
  cluster.sync();
  if (crank != 0) return;

  // leader: publish the argmax, take a ticket for the row's tree
  // a row outside its tree's own extent (node_off[0] > 0 or node_off[B] <
  // n_total) belongs to no tree: it must not draw a ticket of the tree the
  // search landed on, or that tree's walk could run before its own rows
  const bool bad_tree = (n < 1 || n > 256 || off < 0 || off + n > a.n_total || row < off ||
                         row >= off + n);
  if (tid == 0) {
    uint64_t best = 0;
    for (int c = 0; c < C; ++c) best = sm.recv_key[c] > best ? sm.recv_key[c] : best;
    // release: the argmax store below is visible to the CTA that draws the
    // last ticket; acquire: the last CTA sees every other row's argmax
    if (bad_tree) {
      sm.last = 0;  // a row in no tree stores nothing and never touches a ticket
      raise_status(a.status, kStTree);
    } else {
      a.am[row] = (int32_t)key_index(best);
      const int t = atom_add_acq_rel_gpu(&a.tickets[b], 1);
      sm.last = (t == n - 1);
      if (sm.last) a.tickets[b] = 0;  // ready for the next call (the next launch orders it)
    }
  }
  sm.par[tid] = v_par;
  sm.tok[tid] = v_tok;
  __syncthreads();
  if (!sm.last) return;

  // ---- walk of tree b (this CTA saw every row of the tree finish)
  if (tid < n) {
    sm.am[tid] = __ldcg(&a.am[off + tid]);
    a.am[off + tid] = 0;
  }
  const bool bad = (tid < n) && (tid == 0 ? (v_par != -1) : (v_par < 0 || v_par >= tid));
  if (__syncthreads_or(bad)) {
    if (tid == 0) raise_status(a.status, kStTree);
    return;
  }
  uint32_t wkey = 0;
  if (tid < n) {
    bool full = true;
    int depth = 0;
    int v = tid;
    while (v != 0) {  // parent[v] < v: at most v steps
      const int p = sm.par[v];
      full = full && (sm.tok[v] == sm.am[p]);
      v = p;
      ++depth;
    }
    wkey = full ? (((uint32_t)depth << 16) | (uint32_t)(0xFFFF - tid)) : 0u;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const uint32_t w = __shfl_xor_sync(0xffffffffu, wkey, o);
    wkey = w > wkey ? w : wkey;
  }
  if (lane == 0) sm.key[warp] = wkey;
  __syncthreads();
  uint32_t best_w = sm.key[0];
#pragma unroll
  for (int w = 1; w < 8; ++w) best_w = sm.key[w] > best_w ? sm.key[w] : best_w;
  const int A = (int)(best_w >> 16);
  const int astar = 0xFFFF - (int)(best_w & 0xFFFF);
  if (A + 1 > a.path_cap) {
    if (tid == 0) raise_status(a.status, kStIndex);
    return;
  }
  int32_t* path = a.path + (size_t)b * a.path_cap;
  if (tid == 0) {
    int v = astar;
    for (int d = A; d >= 0; --d) {
      path[d] = v;
      v = sm.par[v];
    }
    a.accept_len[b] = A;
    a.bonus[b] = sm.am[astar];
  }
  for (int d = A + 1 + tid; d < a.path_cap; d += kScanThreads) path[d] = -1;
}

template <typename T, bool kAligned>
cudaError_t launch_accept_t(const AcceptArgs& a, int C, cudaStream_t s) {
  auto kern = accept_kernel<T, kAligned>;
  if (C > 8) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
  }
  for (int r0 = 0; r0 < a.n_total; r0 += 65535) {
    const int nr = min(65535, a.n_total - r0);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C, nr, 1);
    cfg.blockDim = dim3(kScanThreads, 1, 1);
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
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, a, r0);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t s) {
  const int C = scan_cluster_size(a.V, a.is_bf16, a.n_total, device_sm_count());
  const int esz = a.is_bf16 ? 2 : 4;
  const bool aligned = ((reinterpret_cast<uintptr_t>(a.logits) & 15) == 0) &&
                       (((a.ld * esz) & 15) == 0);
  if (a.is_bf16)
    return aligned ? launch_accept_t<__nv_bfloat16, true>(a, C, s)
                   : launch_accept_t<__nv_bfloat16, false>(a, C, s);
  return aligned ? launch_accept_t<float, true>(a, C, s) : launch_accept_t<float, false>(a, C, s);
}

}  // namespace tg
