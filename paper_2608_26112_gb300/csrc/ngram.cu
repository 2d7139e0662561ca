// ngram: TreeGraft's training-free small drafter (Appendix, n-gram small
// drafter): the prompt's n-gram index, the lookup with back-off, and the
// small-drafter step of Algorithm 2 that expands a frontier from it.
//
// Index (built once per prompt batch, at prefill).  Prompts are packed:
// sequence b owns token positions [seq[b], seq[b + 1]).  For every order
// n = 1..max_n there is one open-addressing hash table of T int32 slots
// (T a power of two >= 2 * n_tokens, so every table is at most half full);
// a slot holds the LATEST position p whose n-gram tok[p - n + 1 .. p] lies
// inside p's sequence.  A slot's key is implicit: the n-gram at its
// position and the sequence that position belongs to, so a probe verifies
// a hit by comparing tokens (no false matches, whatever the hash).
// Insertion is lock-free: CAS an empty slot, or atomicMax the position into
// the slot that already holds the same n-gram.  The order-1 table also
// counts occurrences per slot, from which the most frequent token of each
// prompt (ties to the lower token) and its latest position are taken: the
// back-off's last resort.
//
// Lookup for the prefix at tree node v: the query is the last max_n tokens
// of (committed context, tokens of the non-root nodes on the path root->v);
// order n probes table n with the query's last n tokens; the longest order
// with a hit wins, else the fallback position.  The children are the first
// m of the target's top-m_cache candidates cached at that position (from
// the prefill logits, by expand_topk), their cached log-probabilities the
// edge scores, score = fp32(s(v) + logprob).
//
// Hash: a running mix of the query's tokens, last token first, through the
// 32-bit finaliser of MurmurHash3 (Appleby, public domain); seeded by the
// sequence id so equal n-grams of different prompts take different chains.
#include <algorithm>

#include "common.cuh"
#include "launch.h"

namespace tg {
namespace {

constexpr int kNgramMaxN = 8;
constexpr int kPosBits = 27;  // best-hit word: order << 27 | position

__device__ __forceinline__ uint32_t fmix32(uint32_t h) {
  h ^= h >> 16;
  h *= 0x85ebca6bu;
  h ^= h >> 13;
  h *= 0xc2b2ae35u;
  h ^= h >> 16;
  return h;
}
__device__ __forceinline__ uint32_t hash_seed(int b) {
  return fmix32((uint32_t)b * 0x9E3779B9u + 0x632BE5ABu);
}
__device__ __forceinline__ uint32_t hash_step(uint32_t h, int32_t t) {
  return fmix32(h + 0x9E3779B9u * ((uint32_t)t + 1u));
}

// sequence of packed position j: the largest b < B with seq[b] <= j
__device__ __forceinline__ int seq_of(const int32_t* seq, int B, int j) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (seq[mid] <= j) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// the index's tables, counts and copies of the prompt (one launch of
// ngram_init clears them and validates seq)
__global__ void __launch_bounds__(256) ngram_init_kernel(NgramArgs a) {
  const size_t total = (size_t)a.max_n * a.T;
  const size_t span = max(total, (size_t)max(a.n_tokens, a.B + 1));
  for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < span;
       i += (size_t)gridDim.x * blockDim.x) {
    if (i < total) a.tab[i] = -1;
    if (i < (size_t)a.T) a.cnt[i] = 0;
    if (i < (size_t)a.n_tokens) a.tok[i] = a.src_tok[i];
    if (i <= (size_t)a.B) {
      const int v = a.src_seq[i];
      a.seq[i] = v;
      const bool bad = (i == 0) ? (v != 0)
                                : (v <= a.src_seq[i - 1] || (i == (size_t)a.B && v != a.n_tokens));
      if (bad) raise_status(a.status, kStIndex);
    }
    if (i < (size_t)a.B) {
      a.fbk[i] = 0ull;
      a.fbp[i] = -1;
    }
  }
}

__device__ __forceinline__ bool same_gram(const int32_t* tok, int p, int j, int n, int lo, int hi) {
  if (p < lo || p >= hi || p - n + 1 < lo) return false;
  for (int k = 0; k < n; ++k)
    if (tok[p - k] != tok[j - k]) return false;
  return true;
}

// One thread per (position j, order n): the n-gram ending at j hashed from
// its n tokens (independent loads), then inserted into table n.
__global__ void __launch_bounds__(256) ngram_insert_kernel(NgramArgs a) {
  const uint32_t mask = (uint32_t)a.T - 1u;
  const long long items = (long long)a.n_tokens * a.max_n;
  for (long long it = blockIdx.x * (long long)blockDim.x + threadIdx.x; it < items;
       it += (long long)gridDim.x * blockDim.x) {
    const int j = (int)(it / a.max_n), i = (int)(it - (long long)j * a.max_n);  // order i + 1
    const int b = seq_of(a.seq, a.B, j);
    const int lo = max(a.seq[b], 0), hi = min(a.seq[b + 1], a.n_tokens);
    if (j < lo || j >= hi || j - i < lo) continue;  // outside the prompt (or a malformed seq)
    uint32_t h = hash_seed(b);
    for (int k = 0; k <= i; ++k) h = hash_step(h, a.tok[j - k]);
    int32_t* tab = a.tab + (size_t)i * a.T;
    uint32_t slot = h & mask;
    for (int probe = 0; probe < a.T; ++probe) {  // an empty slot always exists (load <= 1/2)
      const int old = atomicCAS(tab + slot, -1, j);
      if (old == -1 || same_gram(a.tok, old, j, i + 1, lo, hi)) {
        if (old != -1) atomicMax(tab + slot, j);
        if (i == 0) atomicAdd(a.cnt + slot, 1);
        break;
      }
      slot = (slot + 1u) & mask;
    }
  }
}

// phase 0: per sequence, the max of (count, -token) over its order-1 slots;
// phase 1: the slot holding that maximum gives the fallback position
__global__ void __launch_bounds__(256) ngram_fallback_kernel(NgramArgs a, int phase) {
  for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < a.T; s += gridDim.x * blockDim.x) {
    const int p = a.tab[s];
    if (p < 0) continue;
    const int b = seq_of(a.seq, a.B, p);
    const uint32_t t = (uint32_t)a.tok[p] ^ 0x80000000u;  // signed order
    const unsigned long long key = ((unsigned long long)(uint32_t)a.cnt[s] << 32) | (0xFFFFFFFFu - t);
    if (phase == 0) atomicMax(a.fbk + b, key);
    else if (a.fbk[b] == key) a.fbp[b] = p;
  }
}

// Position of the latest occurrence, inside sequence [lo, hi), of the n
// tokens q[0..n) (q[0] the last token of the n-gram), or -1.
__device__ __forceinline__ int ngram_probe(const NgramArgs& a, int lo, int hi,
                                           const int32_t (&q)[kNgramMaxN], int n, uint32_t h) {
  const int32_t* tab = a.tab + (size_t)(n - 1) * a.T;
  const uint32_t mask = (uint32_t)a.T - 1u;
  uint32_t slot = h & mask;
  for (int it = 0; it < a.T; ++it) {
    const int p = __ldg(tab + slot);
    if (p < 0) return -1;
    if (p >= lo && p < hi && p - n + 1 >= lo) {
      bool eq = true;
#pragma unroll
      for (int k = 0; k < kNgramMaxN; ++k)
        if (k < n) eq &= (__ldg(a.tok + p - k) == q[k]);
      if (eq) return p;
    }
    slot = (slot + 1u) & mask;
  }
  return -1;
}

// Order-n probe for the prefix at node v of tree b: q[k] is the k-th token
// from the end of (context, path tokens).  tree(w, x, pa) reads node w's
// token and parent (from shared or global memory; a parent that does not
// precede its child is the caller's to catch).  Returns the hit word
// (n << 27 | position) or -1 (query shorter than n, or no occurrence).
template <typename TreeRead>
__device__ __forceinline__ int ngram_order_hit(const NgramArgs& a, int b, int v, int n,
                                               const int32_t* ctxp, int clen,
                                               TreeRead&& tree) {
  int32_t q[kNgramMaxN];
  int w = v, ci = clen - 1;
  bool full = true;
  uint32_t h = hash_seed(b);
#pragma unroll
  for (int k = 0; k < kNgramMaxN; ++k) {
    if (k < n) {
      int32_t x = 0;
      if (w != 0) {
        int pa;
        tree(w, x, pa);
        w = pa;
      } else if (ci >= 0) {
        x = ctxp[ci];
        --ci;
      } else {
        full = false;
      }
      q[k] = x;
      h = hash_step(h, x);
    }
  }
  if (!full) return -1;
  const int lo = __ldg(a.seq + b), hi = __ldg(a.seq + b + 1);
  const int p = ngram_probe(a, lo, hi, q, n, h);
  return p < 0 ? -1 : ((n << kPosBits) | p);
}

__device__ __forceinline__ int ctx_len_of(const NgramArgs& a, int b) {
  const int c = __ldg(a.ctx_len + b);
  if (c < 0 || c > a.max_n) {
    raise_status(a.status, kStIndex);
    return max(0, min(c, a.max_n));
  }
  return c;
}

// Lookup for arbitrary tree nodes: one warp per row, lane j probes order j+1.
__global__ void __launch_bounds__(256) ngram_draft_kernel(NgramArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (r >= a.R) return;
  const int node = __ldg(a.rows + r);
  if (node < 0 || node >= a.B * a.cap) {
    if (lane == 0) raise_status(a.status, kStIndex);
    return;
  }
  const int b = node / a.cap, v = node - b * a.cap;
  const size_t base = (size_t)b * a.cap;
  const int clen = ctx_len_of(a, b);
  bool bad = false;
  int hit = -1;
  if (lane < a.max_n) {
    hit = ngram_order_hit(a, b, v, lane + 1, a.ctx + (size_t)b * a.max_n, clen,
                          [&](int w, int32_t& x, int& pa) {
      x = __ldg(a.token + base + w);
      pa = __ldg(a.parent + base + w);
      if (pa < 0 || pa >= w) {  // parents come before children
        bad = true;
        pa = 0;
      }
    });
  }
  if (__any_sync(0xffffffffu, bad)) {
    if (lane == 0) raise_status(a.status, kStTree);
    return;
  }
  const int best = __reduce_max_sync(0xffffffffu, hit);
  int p, n;
  if (best >= 0) {
    p = best & ((1 << kPosBits) - 1);
    n = best >> kPosBits;
  } else {
    p = __ldg(a.fbp + b);
    n = 0;
  }
  if (p < 0) {  // no fallback: the prompt index is malformed
    if (lane == 0) raise_status(a.status, kStIndex);
    return;
  }
  const float ps = __ldg(a.parent_score + r);
  if (lane < a.m) {
    const size_t src = (size_t)p * a.m_cache + lane;
    const size_t o = (size_t)r * a.m + lane;
    const float lp = __ldg(a.cache_lp + src);
    a.out_tok[o] = __ldg(a.cache_tok + src);
    a.out_lp[o] = lp;
    a.out_score[o] = __fadd_rn(ps, lp);
  }
  if (lane == 0) {
    if (a.match_pos) a.match_pos[r] = p - __ldg(a.seq + b);
    if (a.match_n) a.match_n[r] = n;
  }
}

// One small-drafter step of Algorithm 2 with the n-gram drafter, one CTA per
// tree: F = Top_W of the pool [pool_lo, n) by (s desc, id asc), the lookup
// for every frontier node (all orders at once), and the children appended
// at n, n + 1, ... in frontier order, then cached-candidate rank.
constexpr int kGrowThreads = 1024;

__global__ void __launch_bounds__(kGrowThreads) ngram_grow_kernel(NgramArgs a) {
  __shared__ int par_s[kGrowThreads];
  __shared__ int tok_s[kGrowThreads];
  __shared__ float score_s[kGrowThreads];
  __shared__ uint64_t key_s[kGrowThreads];
  __shared__ int front_s[kGrowThreads];
  __shared__ int best_s[kGrowThreads];
  __shared__ int32_t ctx_s[kNgramMaxN];
  const int b = blockIdx.x;
  const int tid = threadIdx.x, nth = blockDim.x;
  const int n = a.n, lo = a.pool_lo, nf = min(a.W, n - lo);
  const size_t base = (size_t)b * a.cap;
  pdl_launch_dependents();
  pdl_wait();
  // the committed context and the fallback position load with the tree
  if (tid < a.max_n) ctx_s[tid] = __ldg(a.ctx + (size_t)b * a.max_n + tid);
  const int fb = __ldg(a.fbp + b);
  int bad = 0;
  for (int v = tid; v < n; v += nth) {
    const int p = a.parent[base + v];
    bad |= (v == 0) ? (p != -1) : (p < 0 || p >= v);
    par_s[v] = p;
    tok_s[v] = a.token[base + v];
    score_s[v] = a.score[base + v];
  }
  if (__syncthreads_or(bad)) {
    if (tid == 0) raise_status(a.status, kStTree);
    return;
  }
  for (int v = lo + tid; v < n; v += nth) key_s[v] = make_key(score_s[v], (uint32_t)v);
  for (int i = tid; i < nf; i += nth) best_s[i] = -1;
  const int clen = ctx_len_of(a, b);
  __syncthreads();
  for (int v = lo + tid; v < n; v += nth) {
    const uint64_t mine = key_s[v];
    int rank = 0;
    for (int w = lo; w < n; ++w) rank += (key_s[w] > mine) ? 1 : 0;
    if (rank < nf) {
      front_s[rank] = v;
      a.frontier[(size_t)b * a.W + rank] = v;
    }
  }
  for (int r = nf + tid; r < a.W; r += nth) a.frontier[(size_t)b * a.W + r] = -1;
  __syncthreads();
  for (int item = tid; item < nf * a.max_n; item += nth) {
    const int i = item / a.max_n, ord = item - i * a.max_n + 1;
    const int hit = ngram_order_hit(a, b, front_s[i], ord, ctx_s, clen, [&](int w, int32_t& x, int& pa) {
      x = tok_s[w];
      pa = par_s[w];
    });
    if (hit >= 0) atomicMax(&best_s[i], hit);
  }
  __syncthreads();
  const int m = a.m;
  for (int item = tid; item < nf * m; item += nth) {
    const int i = item / m, c = item - i * m;
    const int f = front_s[i], best = best_s[i];
    const int p = best >= 0 ? (best & ((1 << kPosBits) - 1)) : fb;
    const size_t u = base + n + item;
    a.parent[u] = f;
    if (p < 0) {  // no fallback: the prompt index is malformed
      if (c == 0) raise_status(a.status, kStIndex);
      a.token[u] = -1;
      a.edge[u] = __int_as_float(0xff800000);
      a.score[u] = __int_as_float(0xff800000);
      continue;
    }
    const size_t src = (size_t)p * a.m_cache + c;
    const float lp = __ldg(a.cache_lp + src);
    a.token[u] = __ldg(a.cache_tok + src);
    a.edge[u] = lp;
    a.score[u] = __fadd_rn(score_s[f], lp);
  }
}

cudaError_t launch_pdl1(const void* fn, dim3 grid, dim3 block, const NgramArgs& a, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {const_cast<NgramArgs*>(&a)};
  return cudaLaunchKernelExC(&cfg, fn, args);
}

unsigned grid_for(size_t work) {
  const size_t g = (work + 255) / 256;
  const size_t cap = (size_t)device_sm_count() * 8;
  return (unsigned)std::max<size_t>(1, std::min(g, cap));
}

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

NgramLayout ngram_layout(int B, int n_tokens, int max_n) {
  NgramLayout L;
  int T = 64;
  while (T < 2 * n_tokens) T *= 2;
  L.T = T;
  size_t o = 0;
  L.tok = o; o += align256((size_t)n_tokens * 4);
  L.seq = o; o += align256((size_t)(B + 1) * 4);
  L.tab = o; o += align256((size_t)max_n * T * 4);
  L.cnt = o; o += align256((size_t)T * 4);
  L.fbk = o; o += align256((size_t)B * 8);
  L.fbp = o; o += align256((size_t)B * 4);
  L.total = o;
  return L;
}

void ngram_carve(NgramArgs& a, void* index, int B, int n_tokens, int max_n) {
  const NgramLayout L = ngram_layout(B, n_tokens, max_n);
  char* p = static_cast<char*>(index);
  a.tok = reinterpret_cast<int32_t*>(p + L.tok);
  a.seq = reinterpret_cast<int32_t*>(p + L.seq);
  a.tab = reinterpret_cast<int32_t*>(p + L.tab);
  a.cnt = reinterpret_cast<int32_t*>(p + L.cnt);
  a.fbk = reinterpret_cast<unsigned long long*>(p + L.fbk);
  a.fbp = reinterpret_cast<int32_t*>(p + L.fbp);
  a.T = L.T;
  a.B = B;
  a.n_tokens = n_tokens;
  a.max_n = max_n;
}

cudaError_t launch_ngram_build(const NgramArgs& a, cudaStream_t s) {
  const size_t span = std::max((size_t)a.max_n * a.T, (size_t)std::max(a.n_tokens, a.B + 1));
  ngram_init_kernel<<<grid_for(span), 256, 0, s>>>(a);
  ngram_insert_kernel<<<grid_for((size_t)a.n_tokens * a.max_n), 256, 0, s>>>(a);
  ngram_fallback_kernel<<<grid_for(a.T), 256, 0, s>>>(a, 0);
  ngram_fallback_kernel<<<grid_for(a.T), 256, 0, s>>>(a, 1);
  return cudaGetLastError();
}

cudaError_t launch_ngram_draft(const NgramArgs& a, cudaStream_t s) {
  const unsigned blocks = (unsigned)(((size_t)a.R * 32 + 255) / 256);
  return launch_pdl1(reinterpret_cast<const void*>(ngram_draft_kernel), dim3(blocks), dim3(256), a,
                     s);
}

cudaError_t launch_ngram_grow(const NgramArgs& a, cudaStream_t s) {
  const int nf = std::min(a.W, a.n - a.pool_lo);
  const int work = std::max(a.n, std::max(nf * a.max_n, nf * a.m));
  const unsigned threads = (unsigned)std::min(kGrowThreads, std::max(32, (work + 31) / 32 * 32));
  return launch_pdl1(reinterpret_cast<const void*>(ngram_grow_kernel), dim3(a.B), dim3(threads), a,
                     s);
}

}  // namespace tg
