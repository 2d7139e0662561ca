// C ABI of the library (declared in include/treegraft.h): host-side argument
// validation, TMA descriptor encoding, the per-device status word, and the
// calls into the kernel launchers.  Nothing here allocates device memory.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <mutex>

#include "../../include/treegraft.h"
#include "launch.h"

namespace tg {

// One status word per device; kernels OR bits into it, the host reads and
// clears it in treegraft_last_device_status().
__device__ int g_status_word;

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_mu;
int* g_status_ptr[kMaxDevices] = {};
int g_sm_count[kMaxDevices] = {};
// bound of the waits on other CTAs (treegraft_set_wait_budget)
std::atomic<long long> g_wait_budget{kInterBlockWaitCycles};

int current_device() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
  return d;
}

int* status_ptr() {
  const int d = current_device();
  if (d < 0) return nullptr;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_status_ptr[d]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    g_status_ptr[d] = static_cast<int*>(p);
  }
  return g_status_ptr[d];
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                   const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                   const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                   CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

bool encode_bf16(CUtensorMap* m, const void* base, int rank, const cuuint64_t* dims,
                 const cuuint64_t* strides_bytes, const cuuint32_t* box) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base), dims,
            strides_bytes, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace

int device_sm_count() {
  const int d = current_device();
  if (d < 0) return 148;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!g_sm_count[d]) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, d) != cudaSuccess || n <= 0)
      n = 148;
    g_sm_count[d] = n;
  }
  return g_sm_count[d];
}

int* status_word_ptr() { return status_ptr(); }

namespace {
bool ngram_shape_ok(int B, int n_tokens, int max_n) {
  return B >= 1 && n_tokens >= B && max_n >= 1 && max_n <= TG_NGRAM_MAX_N;
}
bool ngram_shape_supported(int n_tokens) { return n_tokens <= TG_NGRAM_MAX_TOKENS; }

// index, cache and context arguments shared by draft and grow
int ngram_common(NgramArgs& a, const void* index, size_t index_bytes, int B, int n_tokens,
                 int max_n, const int32_t* cache_tok, const float* cache_lp, int m_cache,
                 const int32_t* ctx, const int32_t* ctx_len, int m) {
  if (!index || !cache_tok || !cache_lp || !ctx || !ctx_len) return TG_ERR_INVALID_ARG;
  if (!ngram_shape_ok(B, n_tokens, max_n) || m < 1 || m_cache < m) return TG_ERR_INVALID_ARG;
  if (!ngram_shape_supported(n_tokens) || m_cache > TG_MAX_TOPK) return TG_ERR_UNSUPPORTED;
  if (index_bytes < ngram_layout(B, n_tokens, max_n).total || !aligned16(index))
    return TG_ERR_INVALID_ARG;
  ngram_carve(a, const_cast<void*>(index), B, n_tokens, max_n);
  a.cache_tok = cache_tok;
  a.cache_lp = cache_lp;
  a.m_cache = m_cache;
  a.ctx = ctx;
  a.ctx_len = ctx_len;
  a.m = m;
  return TG_OK;
}
}  // namespace

}  // namespace tg

using namespace tg;

extern "C" {

size_t treegraft_tree_attn_workspace_size(int B, int max_nodes, int Hq, int Hkv, int D) {
  if (B < 1 || max_nodes < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv || (D != 64 && D != 128)) return 0;
  const int mtiles = ((Hq / Hkv) * max_nodes + 127) / 128;
  return std::max(tree_attn_split_ws_bytes(D, B, Hkv, mtiles, kAttnMaxSplits),
                  tree_attn_whole_ws_bytes(D, B, Hkv, Hq / Hkv, max_nodes));
}

int treegraft_set_wait_budget(int64_t cycles) {
  if (cycles < 0) return TG_ERR_INVALID_ARG;
  g_wait_budget.store(cycles > 0 ? (long long)cycles : kInterBlockWaitCycles);
  return TG_OK;
}

int treegraft_tree_attn(const void* q, const void* k_cache, const void* v_cache,
                        const int32_t* prefix_len, const int32_t* parent, const int32_t* node_off,
                        int B, int max_nodes, int n_total, int Hq, int Hkv, int D, int S_max,
                        float scale, void* out, float* lse_out, void* ws, size_t ws_bytes,
                        void* stream) {
  if (!q || !k_cache || !v_cache || !prefix_len || !parent || !node_off || !out)
    return TG_ERR_INVALID_ARG;
  if (B < 1 || max_nodes < 1 || max_nodes > TG_MAX_TREE_NODES || n_total < 1 || Hq < 1 ||
      Hkv < 1 || S_max < 1 || !(scale >= 0.f) || !std::isfinite(scale))
    return TG_ERR_INVALID_ARG;
  if (Hq % Hkv) return TG_ERR_INVALID_ARG;
  if ((long long)n_total > (long long)B * max_nodes || max_nodes > S_max) return TG_ERR_INVALID_ARG;
  const int G = Hq / Hkv;
  if (D != 64 && D != 128) return TG_ERR_UNSUPPORTED;
  if (G != 1 && G != 2 && G != 4 && G != 8) return TG_ERR_UNSUPPORTED;
  if ((long long)B * Hkv > 65535 || (long long)B * Hkv * S_max + 128 * 32 >= (1ll << 31))
    return TG_ERR_UNSUPPORTED;
  if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out))
    return TG_ERR_INVALID_ARG;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;

  CUtensorMap tq, tk, tv, to;
  {
    const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hq, (cuuint64_t)n_total};
    const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hq * D * 2};
    const cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(128 / G)};
    if (!encode_bf16(&tq, q, 3, dims, strides, box)) return TG_ERR_CUDA;
    if (!encode_bf16(&to, out, 3, dims, strides, box)) return TG_ERR_CUDA;  // same box as q
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)B * Hkv * S_max};
    const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    const cuuint32_t box[2] = {64, 128};
    if (!encode_bf16(&tk, k_cache, 2, dims, strides, box)) return TG_ERR_CUDA;
    if (!encode_bf16(&tv, v_cache, 2, dims, strides, box)) return TG_ERR_CUDA;
  }
  AttnArgs a;
  a.prefix_len = prefix_len;
  a.parent = parent;
  a.node_off = node_off;
  a.B = B;
  a.max_nodes = max_nodes;
  a.n_total = n_total;
  a.Hq = Hq;
  a.Hkv = Hkv;
  a.D = D;
  a.S_max = S_max;
  const float sc = scale > 0.f ? scale : 1.0f / std::sqrt((float)D);
  a.scale_log2 = sc * 1.4426950408889634f;
  a.out = out;
  a.lse_out = lse_out;
  a.status = st;
  a.split_wait_cycles = g_wait_budget.load();
  // Two kernels, one per regime: the split kernel for small problems (keys
  // of a 128-row work item split over several CTAs, partials combined
  // through the workspace), the two-tile kernel for whole units once there
  // are enough of them to fill the GPU.  Each plan estimates its launch
  // time; the cheaper one runs.
  const int nsm = device_sm_count();
  const int mtiles = (G * max_nodes + 127) / 128;
  double split_cost = 0.0;
  const SplitPlan sp = tree_attn_split_plan(D, B, Hkv, mtiles, S_max, nsm, &split_cost);
  // long units are cut into key chunks merged through the workspace when it
  // is large enough; otherwise every unit stays whole
  const bool chunks =
      ws && aligned16(ws) && ws_bytes >= tree_attn_whole_ws_bytes(D, B, Hkv, G, max_nodes);
  const WholePlan wp = tree_attn_whole_plan(D, B, Hkv, G, max_nodes, S_max, nsm, chunks);
  const cudaStream_t cs = static_cast<cudaStream_t>(stream);
  // With a wave of work items or more there is nothing to split: whole
  // units in longest-first order (ragged batches) are then the better plan.
  const bool full = (long long)B * Hkv * mtiles >= nsm;
  if (wp.cost_us < split_cost || (B > 1 && full)) {
    a.unit_rows = wp.unit_rows;
    a.rblocks = tree_attn_rblocks(G, max_nodes, wp.unit_rows);
    a.lpt = wp.lpt;
    a.ws = chunks ? ws : nullptr;
    a.slab_off = tree_attn_whole_slab_off(B, Hkv, G, max_nodes);
    a.resident = tree_attn_whole_resident(D, nsm);
    a.chunk_min = kWholeChunkMin;
    a.coop = 0;
    return launch_tree_attn(tq, tk, tv, to, a, cs) == cudaSuccess ? TG_OK : TG_ERR_CUDA;
  }
  const size_t need = tree_attn_split_ws_bytes(D, B, Hkv, mtiles, sp.splits);
  if (need > 0 && (ws == nullptr || ws_bytes < need || !aligned16(ws))) return TG_ERR_INVALID_ARG;
  a.ws = ws;
  a.coop = sp.coop;
  a.unit_rows = 128;
  a.rblocks = mtiles;
  a.lpt = 0;
  return launch_tree_attn_split(tq, tk, tv, a, sp, cs) == cudaSuccess ? TG_OK : TG_ERR_CUDA;
}


int treegraft_expand_topk(const void* logits, int dtype, int logit_rows, int V, int64_t ld,
                          int rows, const int32_t* row_idx, const float* parent_score, int k,
                          int32_t* tok, float* logprob, float* score, float* lse_out,
                          void* stream) {
  if (rows == 0) return TG_OK;
  if (!logits || !parent_score || !tok || !logprob || !score) return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (rows < 0 || V < 1 || ld < V || logit_rows < 1 || k < 1 || k > V) return TG_ERR_INVALID_ARG;
  if (!row_idx && logit_rows < rows) return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;  // elements must sit at their natural alignment
  if (k > TG_MAX_TOPK || V > (dtype == TG_BF16 ? 262144 : 131072)) return TG_ERR_UNSUPPORTED;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  TopkArgs a = {};
  a.logits = logits;
  a.is_bf16 = dtype == TG_BF16;
  a.logit_rows = logit_rows;
  a.V = V;
  a.ld = ld;
  a.rows = rows;
  a.row_idx = row_idx;
  a.parent_score = parent_score;
  a.k = k;
  a.tok = tok;
  a.logprob = logprob;
  a.score = score;
  a.lse_out = lse_out;
  a.status = st;
  return launch_expand_topk(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                               : TG_ERR_CUDA;
}

int treegraft_rescore_select(const float* weak_edge, const float* strong_lp, int V, int64_t ld,
                             const int32_t* parent, const int32_t* token, const uint8_t* visited,
                             const int32_t* node_off, int B, int max_nodes, int n_total, int N,
                             float* edge_out, float* score_out, int32_t* selected,
                             int32_t* n_selected, void* stream) {
  if (!weak_edge || !strong_lp || !parent || !token || !visited || !node_off || !edge_out ||
      !score_out || !selected || !n_selected)
    return TG_ERR_INVALID_ARG;
  if (B < 1 || V < 1 || ld < V || max_nodes < 1 || max_nodes > TG_MAX_TREE_NODES || N < 1 ||
      N > TG_MAX_TREE_NODES || n_total < B || (long long)n_total > (long long)B * max_nodes)
    return TG_ERR_INVALID_ARG;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  RescoreArgs a;
  a.weak_edge = weak_edge;
  a.strong_lp = strong_lp;
  a.V = V;
  a.ld = ld;
  a.parent = parent;
  a.token = token;
  a.visited = visited;
  a.node_off = node_off;
  a.B = B;
  a.N = N;
  a.n_total = n_total;
  a.edge_out = edge_out;
  a.score_out = score_out;
  a.selected = selected;
  a.n_selected = n_selected;
  a.status = st;
  return launch_rescore_select(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                                  : TG_ERR_CUDA;
}

size_t treegraft_accept_workspace_size(int B, int n_total) {
  if (B < 1 || n_total < 1) return 0;
  const size_t bytes = ((size_t)n_total + (size_t)B) * sizeof(int32_t);
  return (bytes + 255) & ~(size_t)255;
}

int treegraft_global_prune(const float* score, const int32_t* parent, const int32_t* node_off,
                           int B, int max_nodes, int n_total, int budget, int path_cap,
                           int32_t* kept, int32_t* n_kept, int32_t* new_parent,
                           int32_t* position, uint32_t* mask, int32_t* paths, int32_t* n_paths,
                           void* stream) {
  if (!score || !parent || !node_off || !kept || !n_kept || !new_parent || !position || !mask ||
      !paths || !n_paths)
    return TG_ERR_INVALID_ARG;
  if (B < 1 || max_nodes < 1 || n_total < 1 || (long long)n_total > (long long)B * max_nodes ||
      budget < 1 || budget + 1 > TG_MAX_TREE_NODES || path_cap < 1)
    return TG_ERR_INVALID_ARG;
  if (max_nodes > TG_MAX_PRUNE_NODES) return TG_ERR_UNSUPPORTED;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  PruneArgs a;
  a.score = score;
  a.parent = parent;
  a.node_off = node_off;
  a.B = B;
  a.n_total = n_total;
  a.budget = budget;
  a.stride = std::min(budget + 1, max_nodes);
  a.path_cap = path_cap;
  a.kept = kept;
  a.n_kept = n_kept;
  a.new_parent = new_parent;
  a.position = position;
  a.mask = mask;
  a.paths = paths;
  a.n_paths = n_paths;
  a.status = st;
  return launch_global_prune(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                                 : TG_ERR_CUDA;
}

size_t treegraft_grow_workspace_size(int B, int cap, int m) {
  if (B < 1 || cap < 1 || cap > TG_MAX_GROW_NODES || m < 1 || m > TG_MAX_TOPK) return 0;
  return grow_ws_bytes(B, cap, m);
}

int treegraft_grow_step(int mode, const void* logits, int dtype, int V, int64_t ld, int B, int cap,
                        int n, int pool_lo, int W, int m, int32_t* parent, int32_t* token,
                        float* edge, float* score, float* lse_mid, int32_t* frontier, void* ws,
                        size_t ws_bytes, void* stream) {
  if (!logits || !parent || !token || !edge || !score || !frontier || !ws) return TG_ERR_INVALID_ARG;
  if (mode != 0 && mode != 1) return TG_ERR_INVALID_ARG;
  if (mode == 1 && !lse_mid) return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (B < 1 || cap < 1 || V < 1 || ld < V || n < 1 || n > cap || pool_lo < 0 || pool_lo >= n ||
      W < 1 || m < 1 || m > V)
    return TG_ERR_INVALID_ARG;
  if ((long long)n + (long long)std::min(W, n - pool_lo) * m > (long long)cap)
    return TG_ERR_INVALID_ARG;  // the children would not fit the tree's capacity
  if (cap > TG_MAX_GROW_NODES || m > TG_MAX_TOPK || V > (dtype == TG_BF16 ? 262144 : 131072) ||
      (long long)B * cap > (1ll << 30))
    return TG_ERR_UNSUPPORTED;
  if (ws_bytes < grow_ws_bytes(B, cap, m) || !aligned16(ws)) return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;  // elements must sit at their natural alignment
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  GrowArgs a;
  a.mode = mode;
  a.logits = logits;
  a.is_bf16 = dtype == TG_BF16;
  a.V = V;
  a.ld = ld;
  a.B = B;
  a.cap = cap;
  a.n = n;
  a.pool_lo = pool_lo;
  a.W = W;
  a.m = m;
  a.parent = parent;
  a.token = token;
  a.edge = edge;
  a.score = score;
  a.lse_mid = lse_mid;
  a.frontier = frontier;
  a.status = st;
  grow_ws_carve(a, ws, B, cap, m);
  return launch_grow_step(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK : TG_ERR_CUDA;
}

int treegraft_graft_expand(const void* logits, int dtype, int logit_rows, int V, int64_t ld,
                           int B, int N, const int32_t* selected, int k, int cap, int n,
                           int32_t* parent, int32_t* token, float* edge, float* score,
                           void* stream) {
  if (!logits || !selected || !parent || !token || !edge || !score) return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (B < 1 || N < 1 || k < 1 || k > V || V < 1 || ld < V || logit_rows < 1 || n < 1 ||
      cap < 1 || (long long)n + (long long)N * k > (long long)cap)
    return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;  // elements must sit at their natural alignment
  if (k > TG_MAX_TOPK || V > (dtype == TG_BF16 ? 262144 : 131072) ||
      (long long)B * cap > (1ll << 30) || (long long)B * N > (1ll << 30))
    return TG_ERR_UNSUPPORTED;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  TopkArgs a = {};
  a.logits = logits;
  a.is_bf16 = dtype == TG_BF16;
  a.logit_rows = logit_rows;
  a.V = V;
  a.ld = ld;
  a.rows = B * N;
  a.row_idx = selected;
  a.idx_local = 1;
  a.parent_score = score;
  a.ps_gather = 1;
  a.k = k;
  a.gdiv = N;
  a.gcap = cap;
  a.app_n = n;
  a.app_parent = parent;
  a.app_token = token;
  a.app_edge = edge;
  a.app_score = score;
  a.status = st;
  return launch_expand_topk(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                               : TG_ERR_CUDA;
}

int treegraft_accept(const void* target_logits, int dtype, int V, int64_t ld, const int32_t* token,
                     const int32_t* parent, const int32_t* node_off, int B, int max_nodes,
                     int n_total, int path_cap, int32_t* path, int32_t* accept_len,
                     int32_t* bonus, void* ws, size_t ws_bytes, void* stream) {
  if (!target_logits || !token || !parent || !node_off || !path || !accept_len || !bonus || !ws)
    return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (B < 1 || V < 1 || ld < V || n_total < 1 || path_cap < 1 || max_nodes < 1 ||
      max_nodes > TG_MAX_TREE_NODES || (long long)n_total > (long long)B * max_nodes)
    return TG_ERR_INVALID_ARG;
  if (ws_bytes < treegraft_accept_workspace_size(B, n_total) || !aligned16(ws))
    return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(target_logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;  // elements must sit at their natural alignment
  if (V > (dtype == TG_BF16 ? 262144 : 131072)) return TG_ERR_UNSUPPORTED;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  AcceptArgs a;
  a.logits = target_logits;
  a.is_bf16 = dtype == TG_BF16;
  a.V = V;
  a.ld = ld;
  a.token = token;
  a.parent = parent;
  a.node_off = node_off;
  a.B = B;
  a.n_total = n_total;
  a.path_cap = path_cap;
  a.path = path;
  a.accept_len = accept_len;
  a.bonus = bonus;
  a.am = static_cast<int32_t*>(ws);
  a.tickets = static_cast<int32_t*>(ws) + n_total;
  a.status = st;
  return launch_accept(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK : TG_ERR_CUDA;
}


size_t treegraft_accept_sample_workspace_size(int B, int n_total) {
  if (B < 1 || n_total < 1) return 0;
  return sample_ws_bytes(B, n_total);
}

int treegraft_accept_sample(const void* target_logits, int dtype, int V, int64_t ld,
                            float temperature, const int32_t* token, const int32_t* parent,
                            const int32_t* node_off, int B, int max_nodes, int n_total,
                            const float* u, int path_cap, int32_t* path, int32_t* accept_len,
                            int32_t* bonus, void* ws, size_t ws_bytes, void* stream) {
  if (!target_logits || !token || !parent || !node_off || !u || !path || !accept_len || !bonus ||
      !ws)
    return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !std::isfinite(temperature)) return TG_ERR_INVALID_ARG;
  if (B < 1 || V < 1 || ld < V || n_total < 1 || path_cap < 1 || max_nodes < 1 ||
      max_nodes > TG_MAX_TREE_NODES || (long long)n_total > (long long)B * max_nodes)
    return TG_ERR_INVALID_ARG;
  if (ws_bytes < sample_ws_bytes(B, n_total) || !aligned16(ws)) return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(target_logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;  // elements must sit at their natural alignment
  if (V > (dtype == TG_BF16 ? 262144 : 131072) || B > 65535) return TG_ERR_UNSUPPORTED;
  const float scale = 1.4426950408889634f / temperature;
  if (!std::isfinite(scale)) return TG_ERR_UNSUPPORTED;  // T below what fp32 can scale
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  SampleArgs a = {};
  a.logits = target_logits;
  a.is_bf16 = dtype == TG_BF16;
  a.V = V;
  a.ld = ld;
  a.scale_log2 = scale;
  a.token = token;
  a.parent = parent;
  a.node_off = node_off;
  a.B = B;
  a.n_total = n_total;
  a.path_cap = path_cap;
  a.u = u;
  a.path = path;
  a.accept_len = accept_len;
  a.bonus = bonus;
  a.status = st;
  sample_ws_carve(a, ws, B, n_total);
  return launch_accept_sample(a, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? TG_OK
             : TG_ERR_CUDA;
}

size_t treegraft_ngram_index_bytes(int B, int n_tokens, int max_n) {
  if (!ngram_shape_ok(B, n_tokens, max_n) || !ngram_shape_supported(n_tokens)) return 0;
  return ngram_layout(B, n_tokens, max_n).total;
}

int treegraft_ngram_build(const int32_t* tokens, const int32_t* seq_off, int B, int n_tokens,
                          int max_n, void* index, size_t index_bytes, void* stream) {
  if (!tokens || !seq_off || !index) return TG_ERR_INVALID_ARG;
  if (!ngram_shape_ok(B, n_tokens, max_n)) return TG_ERR_INVALID_ARG;
  if (!ngram_shape_supported(n_tokens)) return TG_ERR_UNSUPPORTED;
  if (index_bytes < ngram_layout(B, n_tokens, max_n).total || !aligned16(index))
    return TG_ERR_INVALID_ARG;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  NgramArgs a = {};
  ngram_carve(a, index, B, n_tokens, max_n);
  a.src_tok = tokens;
  a.src_seq = seq_off;
  a.status = st;
  return launch_ngram_build(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                              : TG_ERR_CUDA;
}

int treegraft_ngram_cache(const void* logits, int dtype, int rows, int V, int64_t ld, int m_cache,
                          int32_t* cache_tok, float* cache_lp, void* stream) {
  if (rows == 0) return TG_OK;
  if (!logits || !cache_tok || !cache_lp) return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (rows < 0 || V < 1 || ld < V || m_cache < 1 || m_cache > V) return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;
  if (m_cache > TG_MAX_TOPK || V > (dtype == TG_BF16 ? 262144 : 131072)) return TG_ERR_UNSUPPORTED;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  TopkArgs a = {};
  a.logits = logits;
  a.is_bf16 = dtype == TG_BF16;
  a.logit_rows = rows;
  a.V = V;
  a.ld = ld;
  a.rows = rows;
  a.row_idx = nullptr;
  a.parent_score = nullptr;  // log-probabilities only
  a.k = m_cache;
  a.tok = cache_tok;
  a.logprob = cache_lp;
  a.score = nullptr;
  a.lse_out = nullptr;
  a.status = st;
  return launch_expand_topk(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                               : TG_ERR_CUDA;
}

int treegraft_ngram_draft(const void* index, size_t index_bytes, int B, int n_tokens, int max_n,
                          const int32_t* cache_tok, const float* cache_lp, int m_cache,
                          const int32_t* ctx, const int32_t* ctx_len, const int32_t* parent,
                          const int32_t* token, int cap, const int32_t* rows, int R,
                          const float* parent_score, int m, int32_t* tok, float* logprob,
                          float* score, int32_t* match_pos, int32_t* match_n, void* stream) {
  if (R == 0) return TG_OK;
  if (R < 0 || cap < 1 || !parent || !token || !rows || !parent_score || !tok || !logprob || !score)
    return TG_ERR_INVALID_ARG;
  if ((long long)B * cap > (1ll << 30)) return TG_ERR_UNSUPPORTED;
  NgramArgs a = {};
  const int e = ngram_common(a, index, index_bytes, B, n_tokens, max_n, cache_tok, cache_lp,
                             m_cache, ctx, ctx_len, m);
  if (e != TG_OK) return e;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  a.parent = const_cast<int32_t*>(parent);
  a.token = const_cast<int32_t*>(token);
  a.cap = cap;
  a.rows = rows;
  a.R = R;
  a.parent_score = parent_score;
  a.out_tok = tok;
  a.out_lp = logprob;
  a.out_score = score;
  a.match_pos = match_pos;
  a.match_n = match_n;
  a.status = st;
  return launch_ngram_draft(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                              : TG_ERR_CUDA;
}

int treegraft_ngram_grow_step(const void* index, size_t index_bytes, int B, int n_tokens,
                              int max_n, const int32_t* cache_tok, const float* cache_lp,
                              int m_cache, const int32_t* ctx, const int32_t* ctx_len, int cap,
                              int n, int pool_lo, int W, int m, int32_t* parent, int32_t* token,
                              float* edge, float* score, int32_t* frontier, void* stream) {
  if (!parent || !token || !edge || !score || !frontier) return TG_ERR_INVALID_ARG;
  if (cap < 1 || n < 1 || n > cap || pool_lo < 0 || pool_lo >= n || W < 1) return TG_ERR_INVALID_ARG;
  if ((long long)n + (long long)std::min(W, n - pool_lo) * m > (long long)cap)
    return TG_ERR_INVALID_ARG;  // the children would not fit the tree's capacity
  if (cap > TG_MAX_GROW_NODES || (long long)B * cap > (1ll << 30)) return TG_ERR_UNSUPPORTED;
  NgramArgs a = {};
  const int e = ngram_common(a, index, index_bytes, B, n_tokens, max_n, cache_tok, cache_lp,
                             m_cache, ctx, ctx_len, m);
  if (e != TG_OK) return e;
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  a.parent = parent;
  a.token = token;
  a.cap = cap;
  a.n = n;
  a.pool_lo = pool_lo;
  a.W = W;
  a.edge = edge;
  a.score = score;
  a.frontier = frontier;
  a.status = st;
  return launch_ngram_grow(a, static_cast<cudaStream_t>(stream)) == cudaSuccess ? TG_OK
                                                                             : TG_ERR_CUDA;
}

int treegraft_last_device_status(void* stream) {
  int* st = status_ptr();
  if (!st) return TG_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(s) != cudaSuccess) return TG_ERR_CUDA;
  int v = 0;
  if (cudaMemcpy(&v, st, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return TG_ERR_CUDA;
  if (v != 0 && cudaMemset(st, 0, sizeof(int)) != cudaSuccess) return TG_ERR_CUDA;
  return v;
}

const char* treegraft_status_string(int status) {
  switch (status) {
    case TG_OK: return "ok";
    case TG_ERR_INVALID_ARG: return "invalid argument";
    case TG_ERR_UNSUPPORTED: return "unsupported configuration";
    case TG_ERR_CUDA: return "CUDA error";
    case TG_ERR_DEVICE_TREE: return "malformed tree seen on the device";
    case TG_ERR_TIMEOUT: return "bounded device wait gave up";
    case TG_ERR_DEVICE_INDEX: return "index out of range seen on the device";
    default: return "combination of device status bits";
  }
}

}  // extern "C"
