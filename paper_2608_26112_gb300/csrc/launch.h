// Internal launchers (host side) called by the C ABI layer in api.cu.  All
// arguments are validated by the caller; these only size grids and launch.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace tg {

struct AttnArgs {
  const int32_t* prefix_len;
  const int32_t* parent;
  const int32_t* node_off;
  int B, max_nodes, n_total, Hq, Hkv, D, S_max;
  float scale_log2;  // softmax scale * log2(e)
  void* out;
  float* lse_out;
  int* status;
  // two-tile kernel (tree_attn.cu): whole units, long ones cut into key chunks
  int unit_rows;     // query rows per work unit: 256 (two tiles) or 128 (one)
  int rblocks;       // units per (tree, kv-head) at max_nodes
  int lpt;           // 1: items dealt longest first (work list built on the device)
  int resident;      // CTAs resident at once (the chunk length aims at one item each)
  int chunk_min;     // shortest key chunk, in 128-key tiles
  size_t slab_off;   // byte offset of the chunk slabs in ws (after the unit tickets)
  // split kernel (tree_attn_split.cu)
  void* ws;          // split counters + combine partial rows (tree_attn_split_ws_bytes)
  int coop;          // 1: cooperative launch, split barrier on counters in ws; 0: clusters
  long long split_wait_cycles;  // bound of the wait on the other splits of a work item
};
// two-tile kernel: one CTA per unit, every key tile
struct WholePlan {
  int unit_rows;
  int lpt;
  double cost_us;  // estimated launch time
};
cudaError_t launch_tree_attn(const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                             const CUtensorMap& tm_v, const CUtensorMap& tm_o, const AttnArgs& a,
                             cudaStream_t s);
int tree_attn_rblocks(int G, int max_nodes, int unit_rows);
WholePlan tree_attn_whole_plan(int D, int B, int Hkv, int G, int max_nodes, int S_max,
                               int num_sms, bool chunks);
// workspace of the two-tile kernel: unit tickets, then the partial-row slabs
// of the key chunks (at most kWholeMaxSlabs, twice the resident CTAs)
size_t tree_attn_whole_ws_bytes(int D, int B, int Hkv, int G, int max_nodes);
size_t tree_attn_whole_slab_off(int B, int Hkv, int G, int max_nodes);
int tree_attn_whole_resident(int D, int num_sms);
constexpr int kWholeMaxResident = 256;
constexpr int kWholeChunkMin = 8;
// split kernel: `splits` CTAs per 128-row work item, joined by a thread-block
// cluster or, with coop, by a cooperative launch whose whole grid is resident
struct SplitPlan {
  int splits;
  int coop;
};
cudaError_t launch_tree_attn_split(const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                                   const CUtensorMap& tm_v, const AttnArgs& a, SplitPlan plan,
                                   cudaStream_t s);
SplitPlan tree_attn_split_plan(int D, int B, int Hkv, int mtiles, int S_max, int num_sms,
                               double* cost_us);
size_t tree_attn_split_ws_bytes(int D, int B, int Hkv, int mtiles, int splits);
constexpr int kAttnMaxSplits = 10;
// default bound of the waits on other thread blocks: about one second at the
// GB300's maximum SM clock (the same bound as the in-block mbarrier waits)
constexpr long long kInterBlockWaitCycles = 2000000000LL;
// tmaps: q and out [D, Hq, n_total], k and v [D, B*Hkv*S_max] (innermost first)

struct TopkArgs {
  const void* logits;
  int is_bf16;
  int logit_rows, V;
  int64_t ld;
  int rows;
  const int32_t* row_idx;
  const float* parent_score;
  int k;
  int32_t* tok;
  float* logprob;
  float* score;
  float* lse_out;
  int* status;
  // Tree batches (the grow step).  Without row_idx and with gdiv > 0,
  // logical row i reads physical row (i / gdiv) * gcap + goff + i % gdiv
  // (the pool rows of each tree).  With app_token set, row i = tree i / gdiv,
  // frontier slot i % gdiv, and its children are appended to the tree
  // arrays at (i / gdiv) * gcap + app_n + (i % gdiv) * k + rank, with
  // parent = the physical row - (i / gdiv) * gcap.
  int gdiv, gcap, goff, app_n;
  int32_t* app_parent;
  int32_t* app_token;
  float* app_edge;
  float* app_score;
  int row0;  // first logical row of this launch (grids of at most 65535 rows)
  // Graft (with app_token and row_idx): row_idx holds LOCAL node ids of
  // tree i / gdiv (read at (i / gdiv) * gcap + id, id < app_n), and with
  // ps_gather the parent score is parent_score[that physical row].
  int idx_local, ps_gather;
};
cudaError_t launch_expand_topk(const TopkArgs& a, cudaStream_t s);
int scan_cluster_size(int V, int is_bf16, int rows, int num_sms);

struct RescoreArgs {
  const float* weak_edge;
  const float* strong_lp;
  int V;
  int64_t ld;
  const int32_t* parent;
  const int32_t* token;
  const uint8_t* visited;
  const int32_t* node_off;
  int B, N, n_total;
  float* edge_out;
  float* score_out;
  int32_t* selected;
  int32_t* n_selected;
  int* status;
};
cudaError_t launch_rescore_select(const RescoreArgs& a, cudaStream_t s);

struct AcceptArgs {
  const void* logits;
  int is_bf16;
  int V;
  int64_t ld;
  const int32_t* token;
  const int32_t* parent;
  const int32_t* node_off;
  int B, n_total, path_cap;
  int32_t* path;
  int32_t* accept_len;
  int32_t* bonus;
  int32_t* am;       // scratch [n_total]
  int32_t* tickets;  // scratch [B], zero between calls
  int* status;
};
cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t s);

struct SampleArgs {
  const void* logits;
  int is_bf16;
  int V;
  int64_t ld;
  float scale_log2;  // log2(e) / T
  const int32_t* token;
  const int32_t* parent;
  const int32_t* node_off;
  int B, n_total, path_cap;
  const float* u;  // [n_total, 2]
  int32_t* path;
  int32_t* accept_len;
  int32_t* bonus;
  // workspace (sample_ws_carve)
  int32_t* flag;     // [n_total] child accepted by its parent's rule
  int32_t* bcand;    // [n_total] bonus token if the walk ends at that node
  int32_t* tickets;  // [B], zero between calls
  int* status;
};
size_t sample_ws_bytes(int B, int n_total);
void sample_ws_carve(SampleArgs& a, void* ws, int B, int n_total);
cudaError_t launch_accept_sample(const SampleArgs& a, cudaStream_t s);

struct PruneArgs {
  const float* score;
  const int32_t* parent;
  const int32_t* node_off;
  int B, n_total, budget, stride, path_cap;
  int32_t* kept;
  int32_t* n_kept;
  int32_t* new_parent;
  int32_t* position;
  uint32_t* mask;
  int32_t* paths;
  int32_t* n_paths;
  int* status;
};
cudaError_t launch_global_prune(const PruneArgs& a, cudaStream_t s);

struct GrowArgs {
  int mode;  // 0 small-drafter step, 1 middle-drafter step
  const void* logits;
  int is_bf16;
  int V;
  int64_t ld;
  int B, cap, n, pool_lo, W, m;
  int32_t* parent;
  int32_t* token;
  float* edge;
  float* score;
  float* lse_mid;
  int32_t* frontier;
  // workspace (grow_ws_carve)
  int32_t* ws_row;
  float* ws_ps;
  float* ws_lse;
  int32_t* ws_tok;
  float* ws_lp;
  float* ws_sc;
  int* status;
};
size_t grow_ws_bytes(int B, int cap, int m);
void grow_ws_carve(GrowArgs& a, void* ws, int B, int cap, int m);
cudaError_t launch_grow_step(const GrowArgs& a, cudaStream_t s);

// n-gram small drafter: the index lives in one caller buffer (ngram_layout)
struct NgramLayout {
  size_t tok, seq, tab, cnt, fbk, fbp, total;  // byte offsets, 256-aligned
  int T;                                       // slots per order
};
struct NgramArgs {
  // index (ngram_carve)
  int32_t* tok;              // [n_tokens] packed prompt tokens
  int32_t* seq;              // [B + 1] sequence offsets
  int32_t* tab;              // [max_n][T] latest position per n-gram, -1 empty
  int32_t* cnt;              // [T] occurrences per order-1 slot
  unsigned long long* fbk;   // [B] (count, -token) of the most frequent token
  int32_t* fbp;              // [B] its latest position (-1: none)
  int T, B, n_tokens, max_n;
  // build
  const int32_t* src_tok;
  const int32_t* src_seq;
  // lookup
  const int32_t* cache_tok;  // [n_tokens, m_cache]
  const float* cache_lp;
  int m_cache;
  const int32_t* ctx;        // [B, max_n] committed tail, oldest first
  const int32_t* ctx_len;    // [B]
  int32_t* parent;           // [B * cap] trees
  int32_t* token;
  int cap;
  // draft
  const int32_t* rows;       // [R] b * cap + v
  int R;
  const float* parent_score;
  int m;
  int32_t* out_tok;
  float* out_lp;
  float* out_score;
  int32_t* match_pos;
  int32_t* match_n;
  // grow
  int n, pool_lo, W;
  float* edge;
  float* score;
  int32_t* frontier;
  int* status;
};
NgramLayout ngram_layout(int B, int n_tokens, int max_n);
void ngram_carve(NgramArgs& a, void* index, int B, int n_tokens, int max_n);
cudaError_t launch_ngram_build(const NgramArgs& a, cudaStream_t s);
cudaError_t launch_ngram_draft(const NgramArgs& a, cudaStream_t s);
cudaError_t launch_ngram_grow(const NgramArgs& a, cudaStream_t s);

int device_sm_count();
// device address of the per-device status word (nullptr on failure)
int* status_word_ptr();

}  // namespace tg
