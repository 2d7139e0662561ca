// tree_attn: ancestor-masked GQA tree attention on the 5th-generation tensor
// cores (Sec. 3.1 tree attention; Algorithm 3 tree mask).
//
// Work unit = (tree b, kv-head h, row block rb).  The query rows of one
// kv-head are the G * n pairs (node u, q-head h*G + g), row index u*G + g;
// a row block is 256 consecutive rows, held as two 128-row query tiles
// (M = 128 each, one 3-D TMA box {64, G, 128/G} of q per tile).  Both tiles
// read every K/V tile once: the key axis (prefix [0, P) followed by the tree
// slots [P, P+n)) is cut into 128-key tiles streamed through a two-stage K
// ring and a two-stage V ring.
//
// Warp roles (320 threads, one CTA per SM):
//   warp 0      TMA producer: Q tiles once, K and V tiles into their rings;
//   warp 1      TMEM owner (512 columns: S0, S1, O0, O1) and MMA issuer:
//               S_t = Q_t K^T (M=128, N=128, K=D) and O_t += P_t V (M=128,
//               N=D, K=128, P read from TMEM), bf16 in, fp32 accumulate,
//               completion signalled by tcgen05.commit on mbarriers.  Pipe
//               order per key tile i: PV0(i) S0(i+1) PV1(i) S1(i+1), so the
//               tensor pipe runs one tile's products while the other tile's
//               softmax runs (a two-tile ping-pong).  The whole warp runs the
//               issue loop and one lane issues;
//   warps 2..5  softmax of query tile 0, warps 6..9 of query tile 1: one
//               thread per row (TMEM lane = row), so a row's max and sum
//               never leave the thread.  A thread reads its 128 S values
//               with tcgen05.ld, masks tree keys with the node's ancestor
//               bitmask (built in shared memory from parent[], Algorithm 3),
//               keeps a base-2 online max / sum, writes P as bf16 over the
//               S columns it came from (tcgen05.st), and rescales its O row
//               in TMEM only when the row max grows by more than 8 (base 2)
//               past the reference its P values were taken against.
//
// One CTA computes a whole unit (every key tile) and writes its output rows
// straight from TMEM.  The host sends launches here when there are enough
// units to fill the GPU (large or batched verification: the Llama-3-70B
// shape, serving batches); small problems whose keys must be split over
// several CTAs go to tree_attn_split.cu.  For batches of several trees the
// units are dealt in longest-tree-first order (a ranking every CTA computes
// from prefix_len and node_off), so ragged batches end together.
// Every mbarrier wait is bounded.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "launch.h"

namespace tg {
namespace {

constexpr int kBM = 128;              // query rows per tile (TMEM lanes)
constexpr int kQT = 2;                // query tiles per unit, sharing every K/V tile
constexpr int kRows = kBM * kQT;      // query rows of one unit
constexpr int kBN = 128;              // keys per K/V tile
constexpr int kStages = 2;            // K and V ring depth
constexpr int kGroup = 128;           // softmax threads per query tile (one per row)
constexpr int kThreads = 64 + kQT * kGroup;
constexpr int kAncWords = 9;          // 256 tree slots + one zero word
constexpr int kAncRows = 256 + 1;     // one row per node of a unit, then a zero row
constexpr int kRegion = 128 * 128;    // 128 rows x 128 bytes: one swizzled operand region
constexpr int kLptMaxTrees = 512;     // longest-first ranking only up to this many trees
constexpr float kLn2 = 0.6931471805599453f;

// K and V have their own rings: a K stage is free once both S products of
// its tile are done, a V stage once both PV products are.  S_FULL, P_FULL
// and O_DONE exist once per query tile.
enum { BAR_K_FULL = 0, BAR_V_FULL = 2, BAR_K_EMPTY = 4, BAR_V_EMPTY = 6, BAR_Q_FULL = 8,
       BAR_S_FULL = 9, BAR_P_FULL = 11, BAR_O_DONE = 13, kNumBars = 15 };

constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

template <int D>
struct Layout {
  static constexpr int kQBytes = kBM * D * 2;  // one query tile
  static constexpr int kKVBytes = kBN * D * 2;
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQT * kQBytes;
  static constexpr int kOffV = kOffK + kStages * kKVBytes;
  static constexpr int kTileEnd = kOffV + kStages * kKVBytes;
  // ancestor bitmasks of the unit's nodes; before the unit is known the
  // same bytes hold the longest-first ranking scratch (3 ints per tree)
  static constexpr int kOffAnc = kTileEnd;
  static constexpr int kOffPar = align_up(kOffAnc + kAncRows * kAncWords * 4, 16);
  static constexpr int kOffBar = align_up(kOffPar + 256 * 4, 16);
  static constexpr int kOffMisc = align_up(kOffBar + kNumBars * 8, 16);  // tmem addr, flags, item
  static constexpr int kBytes = kOffMisc + 80;
  static constexpr int kAlloc = kBytes + 1024;  // 1024-byte alignment slack
  static_assert(kAlloc <= 227 * 1024, "shared memory budget");
  static_assert(kOffQ % 1024 == 0 && kOffK % 1024 == 0 && kOffV % 1024 == 0,
                "128-byte-swizzled operand tiles need 1024-byte alignment");
  static_assert(kOffBar % 8 == 0 && kOffMisc % 16 == 0, "mbarrier / scalar alignment");
  static_assert(kAncRows * kAncWords * 4 >= 4 * kLptMaxTrees * 4, "ranking scratch");
  // One chunk's partial rows in the workspace: O / l as bf16 in [D / 8][kRows]
  // groups of 8 (a warp's 32 rows are 512 contiguous bytes), then m[kRows]
  // (base 2) and l[kRows] (fp32).
  static constexpr int kSlabBytes = kRows * (2 * D + 8);
  static constexpr int kSlabM = kRows * D * 2;
  static constexpr int kSlabL = kSlabM + kRows * 4;
  // chunks of one unit: the merge keeps two floats per (chunk, row) over the
  // tile buffers
  static constexpr int kMaxChunks = kTileEnd / (kRows * 8);
};

// 32 mask bits of one node for tree slots [b0, b0 + 32): slot < 0 is the
// committed prefix (always visible), slots >= 256 are beyond any tree.
__device__ __forceinline__ uint32_t mask_word(const uint32_t* anc, int b0) {
  if (b0 <= -32) return 0xFFFFFFFFu;
  if (b0 < 0) {
    const int k = -b0;
    return (anc[0] << k) | ((1u << k) - 1u);
  }
  const int w = b0 >> 5, sh = b0 & 31;
  if (w >= kAncWords) return 0u;
  const uint32_t lo = anc[w];
  const uint32_t hi = (w + 1 < kAncWords) ? anc[w + 1] : 0u;
  return sh ? ((lo >> sh) | (hi << (32 - sh))) : lo;
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

// Paired fp32 arithmetic of sm_100-class SMs: one instruction for two
// independent round-to-nearest operations (the same results as two scalar
// ones), and the three-input max.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;"
      : "=l"(d)
      : "l"(*reinterpret_cast<const uint64_t*>(&a)), "l"(*reinterpret_cast<const uint64_t*>(&b)),
        "l"(*reinterpret_cast<const uint64_t*>(&c)));
  return *reinterpret_cast<float2*>(&d);
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;"
      : "=l"(d)
      : "l"(*reinterpret_cast<const uint64_t*>(&a)), "l"(*reinterpret_cast<const uint64_t*>(&b)));
  return *reinterpret_cast<float2*>(&d);
}
__device__ __forceinline__ float max3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// max of 128 values as four independent chains of three-input maxima
__device__ __forceinline__ float max128(const float (&s)[128]) {
  float ma = s[0], mb = s[2], mc = s[4], md = s[6];
  ma = fmaxf(ma, s[1]);
  mb = fmaxf(mb, s[3]);
  mc = fmaxf(mc, s[5]);
  md = fmaxf(md, s[7]);
#pragma unroll
  for (int c = 8; c < 128; c += 8) {
    ma = max3(ma, s[c], s[c + 1]);
    mb = max3(mb, s[c + 2], s[c + 3]);
    mc = max3(mc, s[c + 4], s[c + 5]);
    md = max3(md, s[c + 6], s[c + 7]);
  }
  return max3(ma, mb, fmaxf(mc, md));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// named barrier among the 128 softmax threads of query tile g (ids 1, 2;
// id 0 is __syncthreads)
__device__ __forceinline__ void group_bar(int g) {
  asm volatile("bar.sync %0, %1;" ::"r"(1 + g), "n"(kGroup) : "memory");
}

// The work item this CTA computes in a longest-first launch.  Every CTA
// derives the same list from prefix_len and node_off: the total work W (key
// tiles summed over units), a chunk length L = max(chunk_min, ceil(1.25 W /
// resident CTAs)), and for each tree nch = min(max_chunks, ceil(tiles / L))
// key chunks per unit (a unit whose keys are split this way has its chunks
// merged by the last one to finish).  Trees are ranked by chunk length (desc, tree id asc),
// items of a tree by (kv-head, row block, chunk); the slot-th item of that
// order is this CTA's.  All threads take part; the result goes to misc:
// [0] b (-1 past the last item), [1] h, [2] rb, [3] chunk, [6] chunks of the
// unit, [7] partial-row slab of the item (-1 for a whole unit).  Invalid
// tree extents count as one item of length 0 (its CTA raises the status).
__device__ void lpt_item(const AttnArgs& a, int G, long long slot, int max_chunks, int* scratch,
                         int* misc) {
  const int B = a.B;
  int* tiles = scratch;
  int* units = scratch + B;
  int* order = scratch + 2 * B;
  int* nch = scratch + 3 * B;
  // W fits an int with room for 5 W: a batch's units hold at most 8 row
  // blocks per kv-head, so W <= 8 B Hkv S_max / 128, and the K/V cache of
  // B Hkv S_max rows of 256 bytes or more must fit in device memory
  int* wsum = misc + 8;
  if (threadIdx.x == 0) *wsum = 0;
  __syncthreads();
  int w = 0;
  for (int t = threadIdx.x; t < B; t += kThreads) {
    const int off = a.node_off[t];
    const int n = a.node_off[t + 1] - off;
    const int P = a.prefix_len[t];
    const bool ok = n >= 1 && n <= 256 && P >= 0 && P + n <= a.S_max && off >= 0 &&
                    off + n <= a.n_total;
    tiles[t] = ok ? (P + n + kBN - 1) / kBN : 0;
    units[t] = ok ? a.Hkv * ((G * n + a.unit_rows - 1) / a.unit_rows) : 1;
    w += tiles[t] * units[t];
  }
  if (w) atomicAdd(wsum, w);
  __syncthreads();
  // chunk length: a quarter above the balanced share W / resident, so that
  // units near the share stay whole (cutting them only adds merges and a
  // second wave) while the long ones are cut
  const int chunk =
      a.ws ? max(a.chunk_min, (5 * *wsum + 4 * a.resident - 1) / (4 * a.resident)) : (1 << 30);
  // nch per tree, and each tree's chunk length in place of its tile count
  // (the ranking below compares lengths only)
  for (int t = threadIdx.x; t < B; t += kThreads) {
    const int nc = tiles[t] > 0 ? min(max_chunks, (tiles[t] + chunk - 1) / chunk) : 1;
    nch[t] = nc;
    tiles[t] = (tiles[t] + nc - 1) / nc;
  }
  __syncthreads();
  for (int t = threadIdx.x; t < B; t += kThreads) {
    const int mine = tiles[t];
    int rank = 0;
    for (int j = 0; j < B; ++j) {
      const int o = tiles[j];
      rank += (o > mine || (o == mine && j < t)) ? 1 : 0;
    }
    order[rank] = t;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    // inclusive scans of items and of split-unit items in rank order, 32
    // ranks at a time
    const int lane = threadIdx.x;
    long long carry = 0, carry_s = 0;
    int found_b = -1, found_li = 0;
    long long found_slab = 0;
    for (int r0 = 0; r0 < B && found_b < 0; r0 += 32) {
      const int r = r0 + lane;
      const int tb = r < B ? order[r] : 0;
      const long long items = r < B ? (long long)units[tb] * nch[tb] : 0;
      const long long sitems = (r < B && nch[tb] > 1) ? items : 0;
      long long x = items, xs = sitems;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, x, o);
        const long long ys = __shfl_up_sync(0xffffffffu, xs, o);
        if (lane >= o) {
          x += y;
          xs += ys;
        }
      }
      const long long hi = carry + x;  // end of this rank's items
      const long long lo = hi - items;
      const long long slo = carry_s + xs - sitems;  // first slab of this rank's items
      const bool here = r < B && slot >= lo && slot < hi;
      const unsigned m = __ballot_sync(0xffffffffu, here);
      if (m) {
        const int src = __ffs(m) - 1;
        found_b = __shfl_sync(0xffffffffu, tb, src);
        found_li = __shfl_sync(0xffffffffu, (int)(slot - lo), src);
        found_slab = __shfl_sync(0xffffffffu, slo, src);
      }
      carry = __shfl_sync(0xffffffffu, hi, 31);
      carry_s = __shfl_sync(0xffffffffu, carry_s + xs, 31);
    }
    if (lane == 0) {
      int h = 0, rb = 0, c = 0, nc = 1, slab = -1;
      if (found_b >= 0) {
        const int off = a.node_off[found_b];
        const int n = a.node_off[found_b + 1] - off;
        const bool ok = n >= 1 && n <= 256;
        const int rbs = max(1, (G * n + a.unit_rows - 1) / a.unit_rows);
        nc = nch[found_b];
        const int lu = found_li / nc;
        c = found_li % nc;
        h = ok ? lu / rbs : 0;
        rb = ok ? lu % rbs : 0;
        if (nc > 1) slab = (int)(found_slab + found_li);
      }
      misc[0] = found_b;
      misc[1] = h;
      misc[2] = rb;
      misc[3] = c;
      misc[6] = nc;
      misc[7] = slab;
    }
  }
  __syncthreads();
}

// Merge the partial rows of a unit whose keys were split into nc chunks
// (Sec. 3.1 attention as a softmax over the union of the chunks' keys).
// Chunk s holds O_s / l_s (bf16), its max m_s (base 2) and sum l_s: with
// w_s = 2^(m_s - M) l_s, M = max_s m_s, the row is o = sum_s w_s (O_s / l_s)
// / sum_s w_s and lse = ln 2 (M + log2 sum_s w_s).  One thread per row: it
// turns the chunks' (m_s, l_s) into normalised weights, kept in its own
// column of `wgt` (2 nc x kRows floats over the CTA's idle tile buffers, so
// no barrier is needed), then accumulates its D / 8 column groups, kU groups
// of kS chunks with their loads in flight together.  Slab reads are
// coalesced across the warp's rows; no per-item index arithmetic.  Kept out
// of line: inlined, its registers made the kernel spill.
template <int D>
__device__ __noinline__ void merge_chunks(const char* __restrict__ slabs, int nc, int rows, int rb,
                                          int G, int n, int off, int h, float* __restrict__ wgt,
                                          const AttnArgs& a) {
  using L = Layout<D>;
  const float NEG_INF = __int_as_float(0xff800000);
  constexpr int CG = D / 8;
  constexpr int kU = 8;   // column groups per pass
  constexpr int kS = 2;   // chunks per pass
  constexpr int kSB = 8;  // chunks whose (m, l) are loaded at once
  static_assert(CG % kU == 0, "column groups per pass");
  const int ur = threadIdx.x;
  if (ur >= rows) return;
  const int rg = rb * a.unit_rows + ur;
  const int uu = rg / G, g = rg % G;
  if (uu >= n) return;
  float M = NEG_INF;
  for (int s0 = 0; s0 < nc; s0 += kSB) {
    float mv[kSB], lv[kSB];
#pragma unroll
    for (int j = 0; j < kSB; ++j) {
      const char* src = slabs + (size_t)min(s0 + j, nc - 1) * L::kSlabBytes;
      mv[j] = __ldcg(reinterpret_cast<const float*>(src + L::kSlabM) + ur);
      lv[j] = __ldcg(reinterpret_cast<const float*>(src + L::kSlabL) + ur);
    }
#pragma unroll
    for (int j = 0; j < kSB; ++j) {
      if (s0 + j < nc) {
        wgt[(s0 + j) * kRows + ur] = mv[j];  // m and l parked, weighted below
        wgt[(nc + s0 + j) * kRows + ur] = lv[j];
        M = fmaxf(M, mv[j]);
      }
    }
  }
  float Ls = 0.f;
  for (int s = 0; s < nc; ++s) {
    const float m = wgt[s * kRows + ur];
    const float w = (m == NEG_INF) ? 0.f : ex2(m - M) * wgt[(nc + s) * kRows + ur];
    wgt[s * kRows + ur] = w;
    Ls += w;
  }
  const float inv = (Ls > 0.f) ? 1.f / Ls : 0.f;
  const size_t orow = (size_t)(off + uu) * a.Hq + (size_t)(h * G + g);
  if (a.lse_out) a.lse_out[orow] = (M == NEG_INF || !(Ls > 0.f)) ? NEG_INF : (M + log2f(Ls)) * kLn2;
  uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.out) + orow * D);
  for (int c0 = 0; c0 < CG; c0 += kU) {
    float acc[kU][8];
#pragma unroll
    for (int u = 0; u < kU; ++u)
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[u][q] = 0.f;
    for (int s0 = 0; s0 < nc; s0 += kS) {
      uint4 ov[kS][kU];
#pragma unroll
      for (int e = 0; e < kS; ++e) {
        const uint4* o = reinterpret_cast<const uint4*>(
                             slabs + (size_t)min(s0 + e, nc - 1) * L::kSlabBytes) +
                         (size_t)c0 * kRows + ur;
#pragma unroll
        for (int u = 0; u < kU; ++u) ov[e][u] = __ldcg(o + u * kRows);
      }
#pragma unroll
      for (int e = 0; e < kS; ++e) {
        if (s0 + e >= nc) break;
        const float w = wgt[(s0 + e) * kRows + ur] * inv;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
          const uint32_t wd[4] = {ov[e][u].x, ov[e][u].y, ov[e][u].z, ov[e][u].w};
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            acc[u][2 * q] = fmaf(w, __uint_as_float(wd[q] << 16), acc[u][2 * q]);
            acc[u][2 * q + 1] = fmaf(w, __uint_as_float(wd[q] & 0xFFFF0000u), acc[u][2 * q + 1]);
          }
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u)
      dst[c0 + u] = make_uint4(pack_bf16(acc[u][0], acc[u][1]), pack_bf16(acc[u][2], acc[u][3]),
                               pack_bf16(acc[u][4], acc[u][5]), pack_bf16(acc[u][6], acc[u][7]));
  }
}

template <int D>
__global__ void __maxnreg__(168)
    tree_attn_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v,
                     const __grid_constant__ CUtensorMap tm_o, const AttnArgs a) {
  using L = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.Hq / a.Hkv;
  // x = unit: (b, h, rb) with rb fastest, or with lpt the slot in
  // longest-first order.  The key tiles of a unit all belong to this CTA.

  int* par_s = reinterpret_cast<int*>(smem + L::kOffPar);
  uint32_t* anc_s = reinterpret_cast<uint32_t*>(smem + L::kOffAnc);
  int* misc = reinterpret_cast<int*>(smem + L::kOffMisc);  // [0..2] unit, [4] tmem, [5] bad
  const uint32_t bar0 = smem_u32(smem + L::kOffBar);
  auto bar = [&](int i) -> uint32_t { return bar0 + 8u * (uint32_t)i; };
  const uint32_t q_base = smem_u32(smem + L::kOffQ);
  const uint32_t k_base = smem_u32(smem + L::kOffK);
  const uint32_t v_base = smem_u32(smem + L::kOffV);
  const float NEG_INF = __int_as_float(0xff800000);

  // the next kernel on the stream may be dispatched now; this one's global
  // reads wait for the previous kernel (a no-op without programmatic
  // dependent launch)
  pdl_launch_dependents();
  pdl_wait();

  int b = 0, h = 0, rb = 0;
  int t0 = 0, t1 = 0;  // key tiles [t0, t1) of this CTA's share of the unit
  if (!a.lpt) {
    const int ui = blockIdx.x;
    b = ui / (a.Hkv * a.rblocks);
    h = (ui / a.rblocks) % a.Hkv;
    rb = ui % a.rblocks;
  }
  // ---- barriers; in unit order the first K/V copies (and tree 0's Q
  //      tiles, which start at node 0) go out before any global read returns
  const int kv_rows = a.B * a.Hkv * a.S_max;
  auto kv_row0 = [&]() { return (b * a.Hkv + h) * a.S_max; };
  auto load_k = [&](int it) {  // it-th key tile of the unit
    const int st = it & 1;
    mbar_arrive_expect_tx(bar(BAR_K_FULL + st), L::kKVBytes);
    const int y = kv_row0() + (t0 + it) * kBN;
#pragma unroll
    for (int c = 0; c < D / 64; ++c)
      tma_load_2d(k_base + st * L::kKVBytes + c * kRegion, &tm_k, c * 64, y, bar(BAR_K_FULL + st));
  };
  auto load_v = [&](int it) {
    const int st = it & 1;
    mbar_arrive_expect_tx(bar(BAR_V_FULL + st), L::kKVBytes);
    const int y = kv_row0() + (t0 + it) * kBN;
#pragma unroll
    for (int c = 0; c < D / 64; ++c)
      tma_load_2d(v_base + st * L::kKVBytes + c * kRegion, &tm_v, c * 64, y, bar(BAR_V_FULL + st));
  };
  // Q tiles t (mask bit t): rows rb*256 + t*128 .. of the unit, from node
  // off + (rb*256 + t*128) / G; one arrive covers every tile issued
  auto load_q = [&](int off, int tmask) {
    int nq = 0;
    for (int t = 0; t < kQT; ++t) nq += (tmask >> t) & 1;
    mbar_arrive_expect_tx(bar(BAR_Q_FULL), nq * L::kQBytes);
    for (int t = 0; t < kQT; ++t) {
      if (!((tmask >> t) & 1)) continue;
      const int node0 = off + (rb * a.unit_rows + t * kBM) / G;
#pragma unroll
      for (int c = 0; c < D / 64; ++c)
        tma_load_3d(q_base + t * L::kQBytes + c * kRegion, &tm_q, c * 64, h * G, node0,
                    bar(BAR_Q_FULL));
    }
  };
  // Early copies are issued only for boxes that start inside the tensors,
  // and every issued copy is awaited before the buffers are reused or the
  // CTA exits.
  bool kv_early[kStages];
  int q_early = 0;  // tile mask
#pragma unroll
  for (int s = 0; s < kStages; ++s)
    kv_early[s] = !a.lpt && kv_row0() + s * kBN < kv_rows;
  if (!a.lpt && b == 0)
    for (int t = 0; t < kQT; ++t)
      if (t * kBM < a.unit_rows && (rb * a.unit_rows + t * kBM) / G < a.n_total) q_early |= 1 << t;
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(BAR_K_FULL + s), 1);
      mbar_init(bar(BAR_V_FULL + s), 1);
      mbar_init(bar(BAR_K_EMPTY + s), 1);
      mbar_init(bar(BAR_V_EMPTY + s), 1);
    }
    mbar_init(bar(BAR_Q_FULL), 1);
    for (int t = 0; t < kQT; ++t) {
      mbar_init(bar(BAR_S_FULL + t), 1);
      mbar_init(bar(BAR_P_FULL + t), kGroup);
      mbar_init(bar(BAR_O_DONE + t), 1);
    }
    fence_mbar_init();
    misc[5] = 0;
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
    tma_prefetch_desc(&tm_q);
    if (q_early) load_q(0, q_early);
#pragma unroll
    for (int s = 0; s < kStages; ++s)
      if (kv_early[s]) {  // used when the unit has that many tiles
        load_k(s);
        load_v(s);
      }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(misc + 4), 512);  // S0 [0,128) S1 [128,256) O0 [256,256+D) O1 after
    tmem_relinquish();
  }
  int chunk = 0, nch = 1, slab = -1;  // key chunk of the unit, chunks, partial-row slab
  if (a.lpt) {
    long long slot = blockIdx.x;
    if (a.B <= kLptMaxTrees) {
      lpt_item(a, G, slot, L::kMaxChunks, reinterpret_cast<int*>(anc_s), misc);
      b = misc[0];
      h = misc[1];
      rb = misc[2];
      chunk = misc[3];
      nch = misc[6];
      slab = misc[7];
    } else {  // tree-major order, whole units
      b = (int)(slot / ((long long)a.Hkv * a.rblocks));
      h = (int)((slot / a.rblocks) % a.Hkv);
      rb = (int)(slot % a.rblocks);
      if (b >= a.B) b = -1;
    }
  }

  // ---- the unit's tree and shape checks (uniform over the CTA)
  const bool no_unit = b < 0;
  int off = 0, n = 0, P = 0;
  if (!no_unit) {
    off = a.node_off[b];
    n = a.node_off[b + 1] - off;
    P = a.prefix_len[b];
  }
  const bool bad_shape = !no_unit && (n < 1 || n > 256 || P < 0 || P + n > a.S_max || off < 0 ||
                                      off + n > a.n_total || (b == 0 && off != 0) ||
                                      (b == a.B - 1 && off + n != a.n_total));
  const int rows = no_unit || bad_shape ? 0 : min(a.unit_rows, G * n - rb * a.unit_rows);
  const bool skip = rows <= 0;
  const bool two = rows > kBM;  // query tile 1 holds rows
  const int Lk = P + n;
  const int T = (Lk + kBN - 1) / kBN;
  // key tiles [t0, t1) of this chunk of the unit (all of them when nch = 1)
  t0 = (int)((long long)chunk * T / nch);
  t1 = (int)((long long)(chunk + 1) * T / nch);
  const int nt = skip ? 0 : t1 - t0;
  if (tid == 0 && !q_early && nt > 0) load_q(off, two ? 3 : 1);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = (uint32_t)misc[4];
  if (skip) {
    // nothing to compute: let the early copies land, leave
    if (tid == 0) {
      bool ok = true;
      for (int s = 0; s < kStages; ++s)
        if (kv_early[s]) {
          ok = mbar_wait(bar(BAR_K_FULL + s), 0) && ok;
          ok = mbar_wait(bar(BAR_V_FULL + s), 0) && ok;
        }
      if (q_early) ok = mbar_wait(bar(BAR_Q_FULL), 0) && ok;
      if (!ok) raise_status(a.status, kStTimeout);
      if (bad_shape && rb == 0 && h == 0) raise_status(a.status, kStTree);
    }
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 512);
    return;
  }

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane < 2) {
      // lane 0 issues K tiles, lane 1 V tiles; a stage past the first two is
      // refilled once its products are done
      const int empty = lane == 0 ? BAR_K_EMPTY : BAR_V_EMPTY;
      for (int it = 0; it < nt; ++it) {
        if (it < kStages) {
          if (!kv_early[it]) {
            if (lane == 0) load_k(it); else load_v(it);
          }
          continue;
        }
        const int st = it & 1;
        if (!mbar_wait(bar(empty + st), ((it >> 1) - 1) & 1)) {
          raise_status(a.status, kStTimeout);
          break;
        }
        if (lane == 0) load_k(it); else load_v(it);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    // the whole warp runs this loop; one elected lane issues (see tc_mma_f16)
    if (nt > 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(kBM, kBN, false);
      constexpr uint32_t kIdO = idesc_bf16_f32(kBM, D, true);
      // Operand descriptors as base + offset / 16: the start-address field
      // (bits 0-13, 16-byte units) of a base descriptor plus the byte offset
      // of the operand, exact while the address stays below 256 KB.
      const uint64_t dq0 = smem_desc_sw128(q_base, 16, 1024);
      const uint64_t dk0 = smem_desc_sw128(k_base, 16, 1024);
      const uint64_t dv0 = smem_desc_sw128(v_base, kRegion, 1024);
      auto issue_s = [&](int t, int st) {  // S_t = Q_t K(stage st)^T into TMEM columns t*128
        const uint64_t dq = dq0 + (uint64_t)((t * L::kQBytes) >> 4);
        const uint64_t dk = dk0 + (uint64_t)((st * L::kKVBytes) >> 4);
        const uint32_t ts = tmem + (uint32_t)(t * 128);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t o = (uint32_t)((kk >> 2) * kRegion + (kk & 3) * 32) >> 4;
          tc_mma_f16(ts, dq + o, dk + o, kIdS, kk > 0 ? 1u : 0u);
        }
        tc_commit(bar(BAR_S_FULL + t));
      };
      auto issue_pv = [&](int t, int st, bool acc) {  // O_t += P_t V(stage st)
        const uint64_t dv = dv0 + (uint64_t)((st * L::kKVBytes) >> 4);
        const uint32_t pa = tmem + (uint32_t)(t * 128);
        const uint32_t to = tmem + 256u + (uint32_t)(t * D);
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk)  // 16 keys per MMA = 8 TMEM columns of P
          tc_mma_f16_ts(to, pa + (uint32_t)(kk * 8), dv + (uint64_t)((kk * 16 * 128) >> 4), kIdO,
                        (kk > 0 || acc) ? 1u : 0u);
        tc_commit(bar(BAR_O_DONE + t));
      };
      bool ok = mbar_wait_warp(bar(BAR_Q_FULL), 0) && mbar_wait_warp(bar(BAR_K_FULL), 0);
      if (ok) {
        tc_fence_after();
        issue_s(0, 0);
        if (two) issue_s(1, 0);
        tc_commit(bar(BAR_K_EMPTY));
      }
      // Pipe order PV0(i) S0(i+1) PV1(i) S1(i+1): tile 0's next S product is
      // queued as soon as its PV product frees the TMEM columns, while tile 1
      // still runs its softmax, so the two softmaxes alternate with the pipe.
      for (int it = 0; ok && it < nt; ++it) {
        const int st = it & 1, ph = it & 1;
        const bool nxt = it + 1 < nt;
        const int st2 = (it + 1) & 1;
        ok = mbar_wait_warp(bar(BAR_P_FULL), ph) && mbar_wait_warp(bar(BAR_V_FULL + st), (it >> 1) & 1);
        if (!ok) break;
        tc_fence_after();
        issue_pv(0, st, it > 0);
        if (!two) tc_commit(bar(BAR_V_EMPTY + st));
        if (nxt) {
          // S_t(it+1) overwrites the TMEM columns PV_t(it) reads P_t(it) from:
          // it waits for that product (products with different accumulators
          // are not ordered)
          ok = mbar_wait_warp(bar(BAR_K_FULL + st2), ((it + 1) >> 1) & 1) && mbar_wait_warp(bar(BAR_O_DONE), ph);
          if (!ok) break;
          tc_fence_after();
          issue_s(0, st2);
          if (!two) tc_commit(bar(BAR_K_EMPTY + st2));
        }
        if (two) {
          if (!(ok = mbar_wait_warp(bar(BAR_P_FULL + 1), ph))) break;
          tc_fence_after();
          issue_pv(1, st, it > 0);
          tc_commit(bar(BAR_V_EMPTY + st));
          if (nxt) {
            if (!(ok = mbar_wait_warp(bar(BAR_O_DONE + 1), ph))) break;
            tc_fence_after();
            issue_s(1, st2);
            tc_commit(bar(BAR_K_EMPTY + st2));
          }
        }
      }
      if (!ok && lane == 0) raise_status(a.status, kStTimeout);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ softmax warps
    const int g = (warp - 2) >> 2;        // query tile of this warp
    const int q4 = warp & 3;              // TMEM lane quarter of this warp
    const int r = q4 * 32 + lane;         // tile row = TMEM lane
    const int gt = g * kGroup + r;        // thread index within the softmax warps
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const float sl2 = a.scale_log2;       // softmax scale * log2(e): scores in base 2
    const int ur = g * kBM + r;           // row of the unit
    const int u_lo = rb * a.unit_rows / G;      // first node of the unit
    const int u = (rb * a.unit_rows + ur) / G;  // this row's node
    const bool row_live = g == 0 || two;  // this tile has rows
    // parent array and its validation, while the first copies are in flight
    int bad = 0;
    for (int v = gt; v < n; v += kQT * kGroup) {
      const int p = a.parent[off + v];
      par_s[v] = p;
      bad |= (v == 0) ? (p != -1) : (p < 0 || p >= v);
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(misc + 5, 1);
    // both groups meet once: parent array and validity are shared
    asm volatile("bar.sync 3, %0;" ::"n"(kQT * kGroup) : "memory");
    const bool tree_ok = misc[5] == 0;
    if (!tree_ok && gt == 0 && rb == 0 && h == 0) raise_status(a.status, kStTree);
    const uint32_t* anc = anc_s + (u < n ? (u - u_lo) : (kAncRows - 1)) * kAncWords;
    // The tree's own keys sit in the unit's last tiles: if this chunk reaches
    // them, each group builds its nodes' ancestor bitmasks now, before any
    // bounded wait, so every warp of the group meets the group barriers
    // (walk parent pointers to the root, Algorithm 3; a malformed tree keeps
    // every tree slot masked, its outputs undefined).
    if (nt > 0 && row_live && t1 * kBN > P) {
      const int n_lo = (g * kBM) / G, n_hi = min((g + 1) * kBM / G, n - u_lo);
      for (int i = n_lo * kAncWords + r; i < n_hi * kAncWords; i += kGroup) anc_s[i] = 0u;
      if (g == 0 && r < kAncWords) anc_s[(kAncRows - 1) * kAncWords + r] = 0u;
      group_bar(g);
      if (tree_ok)
        for (int t = n_lo + r; t < n_hi; t += kGroup) {
          uint32_t* w = anc_s + t * kAncWords;
          for (int v = u_lo + t; v >= 0; v = par_s[v]) w[v >> 5] |= 1u << (v & 31);
        }
      group_bar(g);
    }

    float m_run = NEG_INF, l_run = 0.f;  // m_run in raw score units
    bool ok = true;
    for (int it = 0; it < nt && row_live; ++it) {
      const int st = it & 1, ph = it & 1;
      const int key0 = (t0 + it) * kBN;  // first key of the tile
      ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_S_FULL + g), ph));
      if (!ok) break;
      tc_fence_after();
      float s[128];
      const uint32_t ts = tmem + (uint32_t)(g * 128) + lane_off;
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32f(ts + c * 32, *reinterpret_cast<float(*)[32]>(&s[32 * c]));
      tc_wait_ld();
      if (key0 + kBN > P) {
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          const uint32_t mw = mask_word(anc, key0 + 32 * c - P);
#pragma unroll
          for (int j = 0; j < 32; ++j) s[32 * c + j] = ((mw >> j) & 1u) ? s[32 * c + j] : NEG_INF;
        }
      }
      // The reference max only moves when the row max grows by more than 8
      // (base 2): P = 2^(s - m_ref) stays below 2^8, exact enough in bf16
      // and far from fp32 overflow, and most tiles skip the rescale of O.
      const float m_max = fmaxf(m_run, max128(s));
      const float m_new = (m_run == NEG_INF || (m_max - m_run) * sl2 > 8.f) ? m_max : m_run;
      const float m_use = (m_new == NEG_INF) ? 0.f : m_new;
      const float nb = -m_use * sl2;
      const float corr = ex2(fmaf(m_run, sl2, nb));
      const float2 sl2v = make_float2(sl2, sl2), nbv = make_float2(nb, nb);
      // P = 2^(s sl2 - m sl2) in four chunks of 32 columns; each chunk's bf16
      // pairs go to TMEM (16 columns) while the next chunk is computed, so
      // only the last store's latency is exposed.  Row sum in eight
      // independent chains (four paired accumulators).
      float2 racc[4];
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t pw[16];
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          const int col = 32 * c + j;
          const float2 x = fma2(make_float2(s[col], s[col + 1]), sl2v, nbv);
          const float2 e = make_float2(ex2(x.x), ex2(x.y));
          const int ra = (j >> 1) & 3;
          racc[ra] = (c == 0 && j < 8) ? e : add2(racc[ra], e);
          pw[j >> 1] = pack_bf16(e.x, e.y);
        }
        tmem_st16(ts + (uint32_t)(16 * c), pw);
      }
      const float2 rsum = add2(add2(racc[0], racc[1]), add2(racc[2], racc[3]));
      l_run = l_run * corr + (rsum.x + rsum.y);
      if (it > 0 && __any_sync(0xffffffffu, m_new != m_run)) {
        // PV(it-1) must finish before O is rescaled; PV(it) waits for P below
        ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_O_DONE + g), (it - 1) & 1));
        if (!ok) break;
        tc_fence_after();
        const uint32_t to = tmem + 256u + (uint32_t)(g * D) + lane_off;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(to + c * 32, o);
          tc_wait_ld();
#pragma unroll
          for (int q = 0; q < 32; ++q) o[q] = __float_as_uint(__uint_as_float(o[q]) * corr);
          tmem_st32(to + c * 32, o);
        }
      }
      if (g == 0 && key0 + kBN > Lk) {
        // last tile of the sequence: V rows past the end may hold anything;
        // zero them so that 0-weight rows contribute exactly 0 (both PV
        // products of the tile are issued after this group's P arrives)
        ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_V_FULL + st), (it >> 1) & 1));
        if (!ok) break;
        if (key0 + r >= Lk) {
#pragma unroll
          for (int c = 0; c < D / 64; ++c)
#pragma unroll
            for (int q = 0; q < 8; ++q)
              st_shared_v4(v_base + st * L::kKVBytes + c * kRegion + r * 128 + q * 16,
                           make_uint4(0u, 0u, 0u, 0u));
        }
        fence_proxy_async_smem();  // the zeroed rows (generic stores) for the PV products
      }
      tc_wait_st();
      tc_fence_before();
      mbar_arrive(bar(BAR_P_FULL + g));
      m_run = m_new;
    }
    if (ok && nt > 0 && row_live) {
      ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_O_DONE + g), (nt - 1) & 1));
      if (ok) tc_fence_after();
    }
    ok = __all_sync(0xffffffffu, ok);
    if (!ok && lane == 0) raise_status(a.status, kStTimeout);
    // ---- epilogue.  With one query tile, both groups write it: group 0
    // hands its row statistics over through shared memory (the mask bytes
    // are free now) and each group takes half of the O columns.  With two
    // tiles each group writes its own tile.
    bool have = ok && nt > 0 && row_live;  // this warp's O rows are in TMEM
    float m_out = m_run, l_out = l_run;
    int tile = g, c_lo = 0, c_hi = D / 32;
    if (!two) {
      float* rs = reinterpret_cast<float*>(anc_s);
      if (g == 0) {
        rs[r] = m_run;
        rs[kBM + r] = l_run;
        rs[2 * kBM + r] = have ? 1.f : 0.f;
      }
      asm volatile("bar.sync 3, %0;" ::"n"(kQT * kGroup) : "memory");
      if (g == 1) {
        m_out = rs[r];
        l_out = rs[kBM + r];
        have = rs[2 * kBM + r] != 0.f;  // uniform over the warp: group 0's warp of these lanes
        // observe tile 0's last PV product itself (complete: group 0 saw it)
        if (have) have = __all_sync(0xffffffffu, mbar_wait(bar(BAR_O_DONE), (nt - 1) & 1));
        if (have) tc_fence_after();
      }
      tile = 0;
      c_lo = g * (D / 64);
      c_hi = c_lo + D / 64;
    }
    const int urw = tile * kBM + r;                   // unit row written
    const int rg = rb * a.unit_rows + urw;
    const int uw = rg / G, gq = rg % G;
    const bool store = (tile == 0 || two) && urw < rows && uw < n;
    const bool live = have && m_out != NEG_INF;
    const uint32_t to = tmem + 256u + (uint32_t)(tile * D) + lane_off;
    const float inv = (live && l_out > 0.f) ? 1.f / l_out : 0.f;
    // ---- output.  A whole unit normalises its rows and writes them; a
    // tile whose 128 rows all lie in the tree (head size 128, so each group
    // owns whole 64-column regions) is staged in the consumed stage-0 K / V
    // buffers in the TMA box layout (128-byte swizzle) and written by bulk
    // tensor stores, one per region: coalesced, asynchronous; other tiles
    // are stored row by row.  A chunk of a split unit writes its partial rows
    // (O / l in bf16, m base 2, l) to its workspace slab instead.
    const size_t orow = (size_t)(off + uw) * a.Hq + (size_t)(h * G + gq);
    float o[D];  // this thread's O columns [32 c_lo, 32 c_hi), loaded together
    const int n32 = c_hi - c_lo;
#pragma unroll
    for (int cc = 0; cc < D / 32; ++cc)
      if (have && cc < n32)
        tmem_ld32f(to + (c_lo + cc) * 32, *reinterpret_cast<float(*)[32]>(&o[32 * cc]));
    if (have) tc_wait_ld();
    const int tile_row0 = rb * a.unit_rows + tile * kBM;  // first query row of the tile
    const bool full_tile = nch == 1 && D == 128 && tile_row0 + kBM <= G * n && (tile == 0 || two);
    if (nch > 1) {
      char* sl = static_cast<char*>(a.ws) + a.slab_off + (size_t)slab * L::kSlabBytes;
      uint4* sl8 = reinterpret_cast<uint4*>(sl);  // [D / 8][kRows] groups of 8 bf16
      if (store) {
#pragma unroll
        for (int cc = 0; cc < D / 32; ++cc) {
          if (cc >= n32) break;
          const int c = c_lo + cc;
          const float* oc = &o[32 * cc];
#pragma unroll
          for (int q = 0; q < 4; ++q)
            __stcg(sl8 + (c * 4 + q) * kRows + urw,
                   live ? make_uint4(pack_bf16(oc[8 * q + 0] * inv, oc[8 * q + 1] * inv),
                                     pack_bf16(oc[8 * q + 2] * inv, oc[8 * q + 3] * inv),
                                     pack_bf16(oc[8 * q + 4] * inv, oc[8 * q + 5] * inv),
                                     pack_bf16(oc[8 * q + 6] * inv, oc[8 * q + 7] * inv))
                        : make_uint4(0u, 0u, 0u, 0u));
        }
        if (c_lo == 0) {
          __stcg(reinterpret_cast<float*>(sl + L::kSlabM) + urw, live ? m_out * sl2 : NEG_INF);
          __stcg(reinterpret_cast<float*>(sl + L::kSlabL) + urw, live ? l_out : 0.f);
        }
      }
      __threadfence();  // this thread's partial rows reach L2 before the unit's ticket
    } else if (full_tile) {
      // group g stages into its own buffer: tile 1's group uses V stage 0,
      // the other (and, with one tile, both groups' regions) K stage 0
      const uint32_t stage = (two ? (g == 0 ? k_base : v_base) : k_base);
#pragma unroll
      for (int cc = 0; cc < D / 32; ++cc) {
        if (cc >= n32) break;
        const int c = c_lo + cc;                  // 32-column chunk
        const uint32_t region = stage + (uint32_t)((c >> 1) * kRegion) + (uint32_t)r * 128u;
        const float* oc = &o[32 * cc];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int j = (c & 1) * 4 + q;          // 16-byte chunk within the 128-byte row
          const uint4 v4 = make_uint4(pack_bf16(oc[8 * q + 0] * inv, oc[8 * q + 1] * inv),
                                      pack_bf16(oc[8 * q + 2] * inv, oc[8 * q + 3] * inv),
                                      pack_bf16(oc[8 * q + 4] * inv, oc[8 * q + 5] * inv),
                                      pack_bf16(oc[8 * q + 6] * inv, oc[8 * q + 7] * inv));
          st_shared_v4(region + (uint32_t)(((j ^ (r & 7)) << 4)), live ? v4 : make_uint4(0u, 0u, 0u, 0u));
        }
      }
      fence_proxy_async_smem();  // generic stores -> bulk copy engine
      group_bar(g);
      if (r == 0) {
        const int node0 = off + tile_row0 / G;
        for (int c2 = c_lo / 2; c2 < (c_hi + 1) / 2; ++c2)
          tma_store_3d(&tm_o, stage + (uint32_t)(c2 * kRegion), c2 * 64, h * G, node0);
        bulk_commit();
        bulk_wait_read0();  // the staging buffer is read before the CTA moves on
      }
    } else if (store) {
#pragma unroll
      for (int cc = 0; cc < D / 32; ++cc) {
        if (cc >= n32) break;
        const int c = c_lo + cc;
        const float* oc = &o[32 * cc];
        uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.out) + orow * D + c * 32);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          dst[q] = live ? make_uint4(pack_bf16(oc[8 * q + 0] * inv, oc[8 * q + 1] * inv),
                                     pack_bf16(oc[8 * q + 2] * inv, oc[8 * q + 3] * inv),
                                     pack_bf16(oc[8 * q + 4] * inv, oc[8 * q + 5] * inv),
                                     pack_bf16(oc[8 * q + 6] * inv, oc[8 * q + 7] * inv))
                        : make_uint4(0u, 0u, 0u, 0u);
      }
    }
    if (nch == 1 && store && c_lo == 0 && a.lse_out)
      a.lse_out[orow] = live ? (m_out * sl2 + log2f(l_out)) * kLn2 : NEG_INF;
  }
  if (tid == 0) {
    // speculative K/V and Q copies this CTA did not consume land in buffers
    // that are released at exit: wait for them first
    bool ok = true;
    for (int it = nt; it < kStages; ++it)
      if (kv_early[it] && !(mbar_wait(bar(BAR_K_FULL + it), 0) && mbar_wait(bar(BAR_V_FULL + it), 0)))
        ok = false;
    if (nt == 0 && q_early && !mbar_wait(bar(BAR_Q_FULL), 0)) ok = false;
    if (!ok) raise_status(a.status, kStTimeout);
  }
  tc_fence_before();
  __syncthreads();  // every TMEM read and partial store of the CTA is done
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if (nch == 1) return;
  // ---- a chunk of a split unit: the last of its nch chunks to finish
  // merges them (no chunk ever waits for another).  Thread 0 publishes this
  // CTA's partial rows (fence after the block barrier, then a ticket); the
  // one that draws the unit's last ticket reads every chunk's rows.
  int* misc_last = misc + 10;
  if (tid == 0) {
    int* ticket = static_cast<int*>(a.ws) + ((size_t)(b * a.Hkv + h) * a.rblocks + rb);
    __threadfence();
    const int t = atomicAdd(ticket, 1);
    const bool last = t == nch - 1;
    if (last) {
      __threadfence();
      atomicExch(ticket, 0);  // ready for the next launch
    }
    *misc_last = last ? 1 : 0;
  }
  __syncthreads();
  if (*misc_last == 0) return;
  const char* slabs = static_cast<const char*>(a.ws) + a.slab_off +
                      (size_t)(slab - chunk) * L::kSlabBytes;
  // the chunks' row weights go over the Q / K / V tiles, idle now (a split
  // unit never stages its output there); lpt_item keeps nch within them
  merge_chunks<D>(slabs, nch, rows, rb, G, n, off, h, reinterpret_cast<float*>(smem + L::kOffQ), a);
}

template <int D>
cudaError_t launch_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                     const CUtensorMap& to, const AttnArgs& a, cudaStream_t s) {
  using L = Layout<D>;
  auto kern = tree_attn_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc);
  if (e != cudaSuccess) return e;
  // with key chunks (a workspace is given) a unit may become several items:
  // at most `resident` more than the units in all
  const long long units = (long long)a.B * a.Hkv * a.rblocks;
  const long long items = units + ((a.lpt && a.ws) ? a.resident : 0);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)items, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kAlloc;
  cfg.stream = s;
  // programmatic dependent launch: this launch is dispatched while the
  // previous kernel on the stream finishes (its reads wait in the kernel)
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, tq, tk, tv, to, a);
}

// CTAs of this kernel resident on one SM
template <int D>
int blocks_per_sm_d() {
  using L = Layout<D>;
  auto kern = tree_attn_kernel<D>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc) !=
      cudaSuccess)
    return 0;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, kThreads, L::kAlloc) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

}  // namespace

int tree_attn_rblocks(int G, int max_nodes, int unit_rows) {
  return (G * max_nodes + unit_rows - 1) / unit_rows;
}

// Whole-unit plan for this kernel: units of 256 rows (two query tiles
// sharing each K/V tile) or of 128 rows, and the estimated launch time
// (microseconds, fitted to measured launches).  A 128-key tile costs about
// the same with one query tile as with two (the chain S -> softmax -> PV of
// a tile sets the pace, and two tiles overlap theirs), so 256-row units do
// twice the work per CTA.  Without key chunks: waves of resident CTAs, each
// a fixed part plus one part per key tile of its unit.  With key chunks (a
// batch with a large enough workspace), the longest-first list spreads the
// tiles over the resident CTAs: the longer of the average share and the
// longest item, a fixed part per item of a CTA, and a merge when units are
// cut.  Occupancy is cached per device and head size.
WholePlan tree_attn_whole_plan(int D, int B, int Hkv, int G, int max_nodes, int S_max,
                               int num_sms, bool chunks) {
  const long long resident = tree_attn_whole_resident(D, num_sms);
  const int tiles = (S_max + kBN - 1) / kBN;
  const double kFixed = 5.0, kMerge = 2.0;
  const int lpt = B > 1 ? 1 : 0;
  WholePlan best{kRows, lpt, 1e30};
  for (int ur = kRows; ur >= kBM; ur -= kBM) {
    const long long units = (long long)B * Hkv * tree_attn_rblocks(G, max_nodes, ur);
    const int rows = std::min(ur, G * max_nodes);
    const double per_tile = rows > kBM ? 1.9 : 1.85;
    double cost = (double)((units + resident - 1) / resident) * (kFixed + per_tile * tiles);
    if (lpt && chunks) {
      // average tiles per CTA, the longest item (a chunk or a whole unit),
      // the items each CTA runs
      const double avg = (double)units * tiles / (double)resident;
      const double len = std::min((double)tiles, std::max((double)kWholeChunkMin, std::ceil(1.25 * avg)));
      const double nch = std::ceil((double)tiles / len);
      const double per_cta = std::ceil((double)units * nch / (double)resident);
      cost = std::min(cost, per_cta * kFixed + (nch > 1 ? kMerge : 0.0) + per_tile * std::max(len, avg));
    }
    if (cost < best.cost_us - 1e-9) best = WholePlan{ur, lpt, cost};
  }
  return best;
}

int tree_attn_whole_resident(int D, int num_sms) {
  static int bps_cache[64][2] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  const int di = D == 64 ? 0 : 1;
  int& bps = bps_cache[dev][di];
  if (bps == 0) bps = di ? blocks_per_sm_d<128>() : blocks_per_sm_d<64>();
  return std::min((bps > 0 ? bps : 1) * num_sms, kWholeMaxResident);
}

// the tickets cover every unit id (b, h, rb) at the smaller unit size
size_t tree_attn_whole_slab_off(int B, int Hkv, int G, int max_nodes) {
  const long long units = (long long)B * Hkv * tree_attn_rblocks(G, max_nodes, kBM);
  return (size_t)((units * 4 + 255) / 256 * 256);
}

size_t tree_attn_whole_ws_bytes(int D, int B, int Hkv, int G, int max_nodes) {
  const size_t slab = D == 64 ? (size_t)Layout<64>::kSlabBytes : (size_t)Layout<128>::kSlabBytes;
  return tree_attn_whole_slab_off(B, Hkv, G, max_nodes) + (size_t)2 * kWholeMaxResident * slab;
}

cudaError_t launch_tree_attn(const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                             const CUtensorMap& tm_v, const CUtensorMap& tm_o, const AttnArgs& a,
                             cudaStream_t s) {
  if (a.D == 64) return launch_d<64>(tm_q, tm_k, tm_v, tm_o, a, s);
  return launch_d<128>(tm_q, tm_k, tm_v, tm_o, a, s);
}

}  // namespace tg
