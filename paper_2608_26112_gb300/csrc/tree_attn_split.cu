// tree_attn_split: ancestor-masked GQA tree attention for small problems,
// the keys of each work item split over several thread blocks (Sec. 3.1
// tree attention; Algorithm 3 tree mask).  The host plan sends a launch here
// when the query rows are too few to keep the GPU busy with whole work items
// (verification of one or a few draft trees); larger batches go to the
// two-tile kernel in tree_attn.cu.
//
// Work item = (tree b, kv-head h, 128-row query tile, KV split).  The
// query rows of one kv-head are the G * n pairs (node u, q-head h*G + g),
// row index u*G + g, so the tile is a dense 128 x D bf16 operand: a single
// 3-D TMA box {64, G, 128/G} of q gathers it.  The key axis (prefix
// [0, P) followed by the tree slots [P, P+n)) is cut into 128-key tiles;
// the S_kv CTAs of a thread-block cluster take the tiles round-robin (split
// s: tiles s, s + S_kv, ...), so each CTA can start its first K/V copies
// before it has read anything from global memory.
//
// Warp roles (320 threads, one CTA per SM):
//   warp 0      TMA producer: K and V tiles into a 2-stage ring, Q once;
//   warp 1      TMEM owner and MMA issuer (the whole warp runs the issue loop,
//               one lane issues): S = Q K^T (M=128, N=128, K=D) into
//               one of two TMEM buffers and O += P V (M=128, N=D, K=128) with
//               P read from TMEM, bf16 in, fp32 accumulate, completion
//               signalled by tcgen05.commit on mbarriers.  Pipe order S(0)
//               S(1) PV(0) S(2) PV(1) ...: S(i+1) runs while the softmax of
//               tile i runs; S(i+2) reuses the buffer of P(i) once PV(i) is
//               done;
//   warps 2..9  softmax: two threads per query row (TMEM lane = row), each
//               owning half of the 128 key columns and half of O's columns.
//               They read S with tcgen05.ld, apply the ancestor mask from a
//               per-node bitmask in shared memory, exchange the row max
//               through shared memory, keep a base-2 online max / sum, write
//               P as bf16 over the S buffer it came from (tcgen05.st), and
//               rescale O in TMEM only when the row max grows by more than 8
//               (base 2) past the reference the tile's P was taken against.
//               P(i+1) goes to the other TMEM buffer than P(i), so the
//               softmax never waits for PV(i) unless O has to be rescaled.
// Split combine: each CTA stages its partial rows (O, max, sum) in shared
// memory, copies them with coalesced stores into the caller's workspace (L2
// resident), and after one cluster barrier reduces the S_kv partials of the
// rows it owns, read back from L2.  With a single split the rows are
// normalised and written straight from TMEM.  Every mbarrier wait is bounded.
#include <cooperative_groups.h>

#include "common.cuh"
#include "launch.h"

namespace cg = cooperative_groups;

namespace tg {
namespace {

constexpr int kBM = 128;      // query rows per tile (TMEM lanes)
constexpr int kBN = 128;      // keys per KV tile
constexpr int kStages = 2;    // K and V ring depth
constexpr int kSoftmaxThreads = 256;
constexpr int kThreads = 64 + kSoftmaxThreads;
constexpr int kAncWords = 9;  // 256 tree slots + one zero word
constexpr int kRegion = 128 * 128;  // 128 rows x 128 bytes: one swizzled operand region
constexpr int kClusterMaxSplits = 8;  // portable cluster size
constexpr float kLn2 = 0.6931471805599453f;

// K and V have their own rings: a K stage is free once its S = Q K^T
// product is done, a V stage once its PV product is, so the next K tile is
// requested well before the current PV finishes.
// PV(j) commits to BAR_O_DONE + (j & 1) (phase j >> 1): with two barriers a
// waiter that observes PV(j) before P(j + 2) can be produced never finds a
// barrier two phases ahead, so the softmax may skip waits on PV products.
enum { BAR_K_FULL = 0, BAR_V_FULL = 2, BAR_K_EMPTY = 4, BAR_V_EMPTY = 6, BAR_Q_FULL = 8,
       BAR_S_FULL = 9 /* 2 buffers */, BAR_P_FULL = 11, BAR_O_DONE = 12 /* 2 */, kNumBars = 14 };

constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

template <int D>
struct Layout {
  static constexpr int kQBytes = kBM * D * 2;
  static constexpr int kKVBytes = kBN * D * 2;
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQBytes;
  static constexpr int kOffV = kOffK + kStages * kKVBytes;
  static constexpr int kTileEnd = kOffV + kStages * kKVBytes;
  static constexpr int kOffAnc = kTileEnd;                            // (kBM + 1) rows
  static constexpr int kOffPar = align_up(kOffAnc + (kBM + 1) * kAncWords * 4, 16);
  static constexpr int kOffRedMax = align_up(kOffPar + 256 * 4, 16); // [2 parity][2 half][kBM]
  static constexpr int kOffRedL = align_up(kOffRedMax + 4 * kBM * 4, 16);  // [2 half][kBM]
  static constexpr int kOffBar = align_up(kOffRedL + 2 * kBM * 4, 16);     // mbarriers
  static constexpr int kOffMisc = align_up(kOffBar + kNumBars * 8, 16);    // tmem addr, flag
  static constexpr int kBytes = kOffMisc + 16;
  static constexpr int kAlloc = kBytes + 1024;                       // 1024-byte alignment slack
  // One CTA's partial rows in the workspace, laid out so that a warp (32
  // consecutive rows) writes and reads 512 contiguous bytes: O as
  // [D / 4][kBM] float4 (column group major), then m[kBM] (base 2) and
  // l[kBM], then kBM * 2 spare floats.
  static constexpr int kSlabBytes = kBM * (2 * D + 8);
  static constexpr int kSlabM = kBM * D * 2;  // byte offset of m[] (fp32)
  static constexpr int kSlabL = kSlabM + kBM * 4;  // byte offset of l[] (fp32)
  static_assert(kAlloc <= 227 * 1024, "shared memory budget");
  static_assert(kOffQ % 1024 == 0 && kOffK % 1024 == 0 && kOffV % 1024 == 0,
                "128-byte-swizzled operand tiles need 1024-byte alignment");
  static_assert(kOffBar % 8 == 0 && kOffMisc % 16 == 0, "mbarrier / scalar alignment");
  static_assert(kSlabBytes % 16 == 0 && kSlabM % 16 == 0, "16-byte slab groups");
};

__device__ __forceinline__ uint32_t ld_shared_u32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}
// 32 mask bits of one node for tree slots [b0, b0 + 32): slot < 0 is the
// committed prefix (always visible), slots >= 256 are beyond any tree.  The
// node's bitmask row is at shared-memory address `row`: one register, where
// a generic pointer takes two and the softmax loop, at the register cap,
// would spill one and reload it from local memory on the tree's tile.
__device__ __forceinline__ uint32_t mask_word(uint32_t row, int b0) {
  if (b0 <= -32) return 0xFFFFFFFFu;
  if (b0 < 0) {
    const int k = -b0;
    return (ld_shared_u32(row) << k) | ((1u << k) - 1u);
  }
  const int w = b0 >> 5, sh = b0 & 31;
  if (w >= kAncWords) return 0u;
  const uint32_t lo = ld_shared_u32(row + 4 * w);
  const uint32_t hi = (w + 1 < kAncWords) ? ld_shared_u32(row + 4 * (w + 1)) : 0u;
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
// max of 64 values as four independent chains of three-input maxima
__device__ __forceinline__ float max64(const float (&s)[64]) {
  float ma = s[0], mb = s[2], mc = s[4], md = s[6];
  ma = fmaxf(ma, s[1]);
  mb = fmaxf(mb, s[3]);
  mc = fmaxf(mc, s[5]);
  md = fmaxf(md, s[7]);
#pragma unroll
  for (int c = 8; c < 64; c += 8) {
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

// barrier among the 256 softmax threads only (id 1; id 0 is __syncthreads)
__device__ __forceinline__ void softmax_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(kSoftmaxThreads) : "memory");
}

// Workspace: two int counters per work item (the cooperative split
// barrier), padded to 256 bytes, then the partial-row slabs.
__host__ __device__ constexpr size_t attn_counter_bytes(long long units) {
  return (size_t)((units * 8 + 255) / 256 * 256);
}
__device__ __forceinline__ float* attn_slabs(void* ws, long long units) {
  return reinterpret_cast<float*>(static_cast<char*>(ws) + attn_counter_bytes(units));
}
__device__ __forceinline__ void red_add_release_gpu(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ int ld_acquire_gpu(const int* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Columns one combine item covers with S splits: wide enough that a single
// pass of the CTA's threads covers the rows it owns (ceil(128 / S) rows of
// D columns), narrow enough that the S x COLS loaded bf16 values stay in
// registers, so every load of an item is in flight at once.
template <int S>
constexpr int combine_cols() {
  return S <= 3 ? 64 : (S <= 6 ? 32 : 16);
}
static_assert(kAttnMaxSplits == 10, "combine_rows is instantiated for 2..10 splits");

// Merge the S partial rows of the rows this CTA owns (Sec. 3.1 attention as
// a softmax over the union of the splits' keys).  Split s holds O_s / l_s
// (bf16), its max m_s (base 2) and sum l_s: with w_s = 2^(m_s - M) l_s,
// M = max_s m_s, the row is o = sum_s w_s (O_s / l_s) / sum_s w_s and
// lse = ln 2 (M + log2 sum_s w_s).
template <int D, int S>
__device__ __forceinline__ void combine_rows(const char* slabs, int split, int r0, int G, int n,
                                             int off, int h, const AttnArgs& a) {
  using L = Layout<D>;
  constexpr int COLS = combine_cols<S>() < D ? combine_cols<S>() : D;
  constexpr int NV = COLS / 8;  // groups of 8 bf16 per split per item
  constexpr int CG = D / COLS;
  const float NEG_INF = __int_as_float(0xff800000);
  const int rpc = (kBM + S - 1) / S;  // tile rows owned by each CTA of the work item
  const int row_lo = split * rpc;
  const int my_rows = max(0, min(kBM, row_lo + rpc) - row_lo);
  // items run row-fastest so that a warp reads consecutive rows of one
  // column group: contiguous in the slab layout
  for (int item = threadIdx.x; item < my_rows * CG; item += kThreads) {
    const int rr = row_lo + item % my_rows, cg = item / my_rows;
    const int rg = r0 + rr;
    const int uu = rg / G, g = rg % G;
    if (uu >= n) continue;
    float mv[S], lv[S];
    uint4 ov[S][NV];
#pragma unroll
    for (int sp = 0; sp < S; ++sp) {
      const char* src = slabs + (size_t)sp * L::kSlabBytes;
      const uint4* src8 = reinterpret_cast<const uint4*>(src);
      mv[sp] = __ldcg(reinterpret_cast<const float*>(src + L::kSlabM) + rr);
      lv[sp] = __ldcg(reinterpret_cast<const float*>(src + L::kSlabL) + rr);
#pragma unroll
      for (int q = 0; q < NV; ++q) ov[sp][q] = __ldcg(src8 + (cg * NV + q) * kBM + rr);
    }
    float M = NEG_INF;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) M = fmaxf(M, mv[sp]);
    float Ls = 0.f;
    float acc[COLS];
#pragma unroll
    for (int q = 0; q < COLS; ++q) acc[q] = 0.f;
#pragma unroll
    for (int sp = 0; sp < S; ++sp) {
      const float w = (mv[sp] == NEG_INF) ? 0.f : ex2(mv[sp] - M) * lv[sp];
      Ls += w;
#pragma unroll
      for (int q = 0; q < NV; ++q) {
        const uint32_t wd[4] = {ov[sp][q].x, ov[sp][q].y, ov[sp][q].z, ov[sp][q].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          acc[8 * q + 2 * j] += w * __uint_as_float(wd[j] << 16);
          acc[8 * q + 2 * j + 1] += w * __uint_as_float(wd[j] & 0xFFFF0000u);
        }
      }
    }
    const float inv = (Ls > 0.f) ? 1.f / Ls : 0.f;
    const size_t orow = (size_t)(off + uu) * a.Hq + (size_t)(h * G + g);
    uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.out) + orow * D + cg * COLS);
#pragma unroll
    for (int q = 0; q < NV; ++q)
      dst[q] = make_uint4(pack_bf16(acc[8 * q + 0] * inv, acc[8 * q + 1] * inv),
                          pack_bf16(acc[8 * q + 2] * inv, acc[8 * q + 3] * inv),
                          pack_bf16(acc[8 * q + 4] * inv, acc[8 * q + 5] * inv),
                          pack_bf16(acc[8 * q + 6] * inv, acc[8 * q + 7] * inv));
    if (cg == 0 && a.lse_out) a.lse_out[orow] = (M == NEG_INF) ? M : (M + log2f(Ls)) * kLn2;
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_split_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const AttnArgs a) {
  using L = Layout<D>;
  constexpr int DH = D / 2;  // O columns per softmax thread
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  cg::cluster_group cluster = cg::this_cluster();
  // the S_kv CTAs of a work item: a cluster, or (cooperative launch) the
  // gridDim.x CTAs along x
  const int S_kv = a.coop ? (int)gridDim.x : (int)cluster.num_blocks();
  const int split = a.coop ? (int)blockIdx.x : (int)cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.Hq / a.Hkv;
  const int b = blockIdx.z / a.Hkv, h = blockIdx.z % a.Hkv;
  const int r0 = blockIdx.y * kBM;

  int* par_s = reinterpret_cast<int*>(smem + L::kOffPar);
  uint32_t* anc_s = reinterpret_cast<uint32_t*>(smem + L::kOffAnc);
  float* red_max = reinterpret_cast<float*>(smem + L::kOffRedMax);
  float* red_l = reinterpret_cast<float*>(smem + L::kOffRedL);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kOffMisc);
  int* bad_flag = reinterpret_cast<int*>(smem + L::kOffMisc + 4);
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
  // ---- the tree's extent (global reads in flight while the barriers are set up)
  const int off = a.node_off[b];
  const int n = a.node_off[b + 1] - off;
  const int P = a.prefix_len[b];

  // ---- barriers; the first K/V copies go out before any global read returns
  const int kv_row0 = (b * a.Hkv + h) * a.S_max;
  auto load_k = [&](int it) {  // it-th tile of this split = tile split + it * S_kv
    const int st = it & 1;
    mbar_arrive_expect_tx(bar(BAR_K_FULL + st), L::kKVBytes);
    const int y = kv_row0 + (split + it * S_kv) * kBN;
#pragma unroll
    for (int c = 0; c < D / 64; ++c)
      tma_load_2d(k_base + st * L::kKVBytes + c * kRegion, &tm_k, c * 64, y, bar(BAR_K_FULL + st));
  };
  auto load_v = [&](int it) {
    const int st = it & 1;
    mbar_arrive_expect_tx(bar(BAR_V_FULL + st), L::kKVBytes);
    const int y = kv_row0 + (split + it * S_kv) * kBN;
#pragma unroll
    for (int c = 0; c < D / 64; ++c)
      tma_load_2d(v_base + st * L::kKVBytes + c * kRegion, &tm_v, c * 64, y, bar(BAR_V_FULL + st));
  };
  // Early copies are issued only for boxes that start inside the tensors (a
  // box past the last row is never requested), and every issued copy is
  // awaited before the buffers are reused or the CTA exits.
  const int kv_rows = a.B * a.Hkv * a.S_max;
  bool kv_early[kStages];
#pragma unroll
  for (int s = 0; s < kStages; ++s) kv_early[s] = kv_row0 + (split + s * S_kv) * kBN < kv_rows;
  auto load_q = [&](int node0) {
    mbar_arrive_expect_tx(bar(BAR_Q_FULL), L::kQBytes);
#pragma unroll
    for (int c = 0; c < D / 64; ++c)
      tma_load_3d(q_base + c * kRegion, &tm_q, c * 64, h * G, node0, bar(BAR_Q_FULL));
  };
  // tree 0 starts at node 0 (node_off[0] = 0), so its q tile is known up front
  const bool q_early = (b == 0) && (r0 / G < a.n_total);
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(BAR_K_FULL + s), 1);
      mbar_init(bar(BAR_V_FULL + s), 1);
      mbar_init(bar(BAR_K_EMPTY + s), 1);
      mbar_init(bar(BAR_V_EMPTY + s), 1);
      mbar_init(bar(BAR_S_FULL + s), 1);
    }
    mbar_init(bar(BAR_Q_FULL), 1);
    mbar_init(bar(BAR_P_FULL), kSoftmaxThreads);
    mbar_init(bar(BAR_O_DONE), 1);
    mbar_init(bar(BAR_O_DONE + 1), 1);
    fence_mbar_init();
    *bad_flag = 0;
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
    tma_prefetch_desc(&tm_q);
    if (q_early) load_q(r0 / G);
#pragma unroll
    for (int s = 0; s < kStages; ++s)
      if (kv_early[s]) {  // used when this split has that many tiles
        load_k(s);
        load_v(s);
      }
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 512);  // S buffers: [0,128) [128,256); O: [256, 256 + D)
    tmem_relinquish();
  }

  // ---- shape checks (uniform over the cluster)
  const bool bad_shape = (n < 1 || n > 256 || P < 0 || P + n > a.S_max || off < 0 ||
                          off + n > a.n_total || (b == 0 && off != 0) ||
                          (b == a.B - 1 && off + n != a.n_total));
  const bool skip = bad_shape || r0 >= G * n;
  const int Lk = P + n;
  const int T = (Lk + kBN - 1) / kBN;
  const int nt = skip ? 0 : (split < T ? (T - split + S_kv - 1) / S_kv : 0);
  const int u_base = r0 / G;
  if (tid == 0 && !q_early && nt > 0) load_q(off + u_base);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (skip) {
    // nothing to compute (uniform over the cluster): let the early copies land, leave
    if (tid == 0) {
      bool ok = true;
      for (int s = 0; s < kStages; ++s)
        if (kv_early[s]) {
          ok = mbar_wait(bar(BAR_K_FULL + s), 0) && ok;
          ok = mbar_wait(bar(BAR_V_FULL + s), 0) && ok;
        }
      if (q_early) ok = mbar_wait(bar(BAR_Q_FULL), 0) && ok;
      if (!ok) raise_status(a.status, kStTimeout);
      if (bad_shape && split == 0 && blockIdx.y == 0) raise_status(a.status, kStTree);
    }
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, 512);
    return;
  }

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane < 2) {
      // real tiles always lie inside the tensors, so an early stage was issued
      // for each of the first min(nt, kStages) tiles.  Lane 0 refills K
      // (after the S product of the tile two back), lane 1 refills V (after
      // its PV product).
      const int empty = lane == 0 ? BAR_K_EMPTY : BAR_V_EMPTY;
      for (int it = kStages; it < nt; ++it) {
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
      const uint32_t tmem_O = tmem + 256u;
      // Operand descriptors as base + offset / 16: the start-address field
      // (bits 0-13, 16-byte units) of a base descriptor plus the byte offset
      // of the operand, exact while the address stays below 256 KB: a few
      // integer ops per MMA instead of a full descriptor build keep the
      // tensor pipe fed.
      const uint64_t dq0 = smem_desc_sw128(q_base, 16, 1024);
      const uint64_t dk0 = smem_desc_sw128(k_base, 16, 1024);
      const uint64_t dv0 = smem_desc_sw128(v_base, kRegion, 1024);
      bool ok = mbar_wait_warp(bar(BAR_Q_FULL), 0);
      for (int it = 0; ok && it <= nt; ++it) {
        if (it < nt) {
          // S buffer it&1 holds P(it-2): S(it) may overwrite it once PV(it-2)
          // is done (MMAs with different accumulators are not ordered)
          const int st = it & 1;
          ok = mbar_wait_warp(bar(BAR_K_FULL + st), (it >> 1) & 1);
          if (ok && it >= 2) ok = mbar_wait_warp(bar(BAR_O_DONE + st), ((it - 2) >> 1) & 1);
          if (!ok) break;
          tc_fence_after();
          const uint64_t dk = dk0 + (uint64_t)((st * L::kKVBytes) >> 4);
          const uint32_t ts = tmem + (uint32_t)(st * 128);
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t o = (uint32_t)((kk >> 2) * kRegion + (kk & 3) * 32) >> 4;
            tc_mma_f16(ts, dq0 + o, dk + o, kIdS, kk > 0 ? 1u : 0u);
          }
          tc_commit(bar(BAR_S_FULL + st));
          tc_commit(bar(BAR_K_EMPTY + st));
        }
        if (it > 0) {
          const int jt = it - 1, sp = jt & 1;
          const int jkey0 = (split + jt * S_kv) * kBN;
          if (jkey0 + kBN > Lk) {
            // last tile of the sequence: V rows past the end may hold
            // anything; the warp zeroes them while the softmax of the tile
            // runs, so that 0-weight rows contribute exactly 0
            if (!(ok = mbar_wait_warp(bar(BAR_V_FULL + sp), (jt >> 1) & 1))) break;
            const int row0 = Lk - jkey0, chunks = (kBN - row0) * (D / 64) * 8;
            for (int i = lane; i < chunks; i += 32) {
              const int rr = row0 + i / ((D / 64) * 8), c = (i >> 3) % (D / 64), q = i & 7;
              st_shared_v4(v_base + sp * L::kKVBytes + c * kRegion + rr * 128 + q * 16,
                           make_uint4(0u, 0u, 0u, 0u));
            }
            fence_proxy_async_smem();  // the zeroed rows (generic stores) for the PV product
            __syncwarp();
          }
          ok = mbar_wait_warp(bar(BAR_P_FULL), jt & 1) && mbar_wait_warp(bar(BAR_V_FULL + sp), (jt >> 1) & 1);
          if (!ok) break;
          tc_fence_after();
          const uint64_t dv = dv0 + (uint64_t)((sp * L::kKVBytes) >> 4);
          const uint32_t pa = tmem + (uint32_t)(sp * 128);
          const uint32_t acc0 = jt > 0 ? 1u : 0u;
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk) {
            // P(jt) in S buffer jt&1: 16 keys per MMA = 8 TMEM columns
            tc_mma_f16_ts(tmem_O, pa + (uint32_t)(kk * 8), dv + (uint64_t)((kk * 16 * 128) >> 4),
                          kIdO, kk > 0 ? 1u : acc0);
          }
          tc_commit(bar(BAR_O_DONE + sp));
          tc_commit(bar(BAR_V_EMPTY + sp));
        }
      }
      if (!ok && lane == 0) raise_status(a.status, kStTimeout);
    }
    __syncwarp();
  }

  // ------------------------------------------------ softmax warps
  const int sidx = tid - 64;           // 0..255 for softmax threads
  const int q4 = warp & 3;             // TMEM lane quarter of this warp
  const int half = sidx >> 7;          // key / O column half
  const int r = q4 * 32 + lane;        // tile row = TMEM lane
  const float sl2 = a.scale_log2;      // softmax scale * log2(e): scores in base 2
  if (warp >= 2) {
    // parent array, validation and ancestor bitmasks, while the first
    // copies and products are in flight (row kBM, for rows past the tree,
    // stays zero)
    int bad = 0;
    for (int v = sidx; v < n; v += kSoftmaxThreads) {
      const int p = a.parent[off + v];
      par_s[v] = p;
      bad |= (v == 0) ? (p != -1) : (p < 0 || p >= v);
    }
    if (sidx < kAncWords) anc_s[kBM * kAncWords + sidx] = 0u;
    if (__any_sync(0xffffffffu, bad) && lane == 0) atomicOr(bad_flag, 1);
    softmax_bar();
    // Only a split whose tiles reach the tree's keys reads the bitmasks.
    // Each node's bits gather in registers along its parent chain (the walk
    // of Algorithm 3) and its row is stored once.  A malformed tree keeps
    // every tree slot masked; its outputs are undefined.
    if (nt > 0 && (split + (nt - 1) * S_kv + 1) * kBN > P) {
      const bool good = *bad_flag == 0;
      const int tile_nodes = min(kBM / G, n - u_base);
      for (int t = sidx; t < tile_nodes; t += kSoftmaxThreads) {
        uint32_t m[kAncWords - 1];
#pragma unroll
        for (int k = 0; k < kAncWords - 1; ++k) m[k] = 0u;
        if (good)
          for (int v = u_base + t; v >= 0; v = par_s[v]) {
            const int wi = v >> 5;
            const uint32_t bit = 1u << (v & 31);
#pragma unroll
            for (int k = 0; k < kAncWords - 1; ++k) m[k] |= (k == wi) ? bit : 0u;
          }
        uint32_t* w = anc_s + t * kAncWords;
#pragma unroll
        for (int k = 0; k < kAncWords - 1; ++k) w[k] = m[k];
        w[kAncWords - 1] = 0u;
      }
    }
    if (sidx == 0 && split == 0 && *bad_flag != 0) raise_status(a.status, kStTree);
    softmax_bar();

    const int u = (r0 + r) / G;
    const uint32_t anc = smem_u32(anc_s + (u < n ? (u - u_base) : kBM) * kAncWords);
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const uint32_t tmem_O = tmem + 256u;
    float m_run = NEG_INF, l_run = 0.f;  // m_run in raw score units
    // PV products observed so far, in order (PV(j): barrier j & 1, phase j >> 1)
    int o_seen = 0;
    auto observe = [&](int upto) -> bool {
      bool good = true;
      while (good && o_seen < upto) {
        good = mbar_wait(bar(BAR_O_DONE + (o_seen & 1)), (o_seen >> 1) & 1);
        if (good) ++o_seen;
      }
      return good;
    };
    // Every softmax warp runs the same number of iterations and meets the
    // named barrier in each one, also after a timed-out wait (then it only
    // skips the work), so no warp is ever left waiting at that barrier.
    bool ok = true;
    for (int it = 0; it < nt; ++it) {
      const int st = it & 1;
      const int tile_key0 = (split + it * S_kv) * kBN;
      const int key0 = tile_key0 + half * 64;  // first key of this thread's columns
      // the ancestor-mask words of this thread's tree columns, read from
      // shared memory while S is still being computed
      const bool tree_cols = key0 + 64 > P;
      uint32_t mw0 = 0xFFFFFFFFu, mw1 = 0xFFFFFFFFu;
      if (tree_cols) {
        mw0 = mask_word(anc, key0 - P);
        mw1 = mask_word(anc, key0 + 32 - P);
      }
      float s[64];
      float mx = NEG_INF;
      if (ok) ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_S_FULL + st), (it >> 1) & 1));
      // S(it) began after PV(it-2) finished: observing PV(0..it-2) returns at once
      if (ok) ok = __all_sync(0xffffffffu, observe(it - 1));
      if (ok) {
        tc_fence_after();
        const uint32_t ts = tmem + (uint32_t)(st * 128) + lane_off + half * 64;
        tmem_ld32f(ts, *reinterpret_cast<float(*)[32]>(&s[0]));
        tmem_ld32f(ts + 32, *reinterpret_cast<float(*)[32]>(&s[32]));
        tc_wait_ld();
        if (tree_cols) {
#pragma unroll
          for (int c = 0; c < 64; ++c) {
            const bool vis = ((c < 32) ? mw0 : mw1) & (1u << (c & 31));
            s[c] = vis ? s[c] : NEG_INF;
          }
        }
        mx = max64(s);
      }
      // row max over both halves (double-buffered by tile parity)
      float* rm = red_max + st * 2 * kBM;
      rm[half * kBM + r] = mx;
      softmax_bar();
      if (!ok) continue;
      // The reference max only moves when the row max grows by more than 8
      // (base 2): P = 2^(s - m_ref) stays below 2^8, exact enough in bf16 and
      // far from fp32 overflow, and most tiles skip the rescale of O.  O, l
      // and the partial rows all use the same reference.
      const float m_max = fmaxf(m_run, fmaxf(rm[r], rm[kBM + r]));
      const float m_new = (m_run == NEG_INF || (m_max - m_run) * sl2 > 8.f) ? m_max : m_run;
      const float m_use = (m_new == NEG_INF) ? 0.f : m_new;
      const float nb = -m_use * sl2;
      const float corr = ex2(fmaf(m_run, sl2, nb));
      const float2 sl2v = make_float2(sl2, sl2), nbv = make_float2(nb, nb);
      // row sum in eight independent chains (four paired accumulators)
      float2 racc[4];
#pragma unroll
      for (int c = 0; c < 64; c += 2) {
        const float2 x = fma2(make_float2(s[c], s[c + 1]), sl2v, nbv);
        s[c] = ex2(x.x);
        s[c + 1] = ex2(x.y);
        const float2 e = make_float2(s[c], s[c + 1]);
        racc[(c >> 1) & 3] = c < 8 ? e : add2(racc[(c >> 1) & 3], e);
      }
      const float2 rsum = add2(add2(racc[0], racc[1]), add2(racc[2], racc[3]));
      l_run = l_run * corr + (rsum.x + rsum.y);
      if (it > 0 && __any_sync(0xffffffffu, m_new > m_run)) {
        // PV(it-1) must finish before O is rescaled
        ok = __all_sync(0xffffffffu, observe(it));
        if (!ok) continue;
        tc_fence_after();
        {
#pragma unroll
          for (int c = 0; c < DH / 32; ++c) {
            uint32_t o[32];
            tmem_ld32(tmem_O + lane_off + half * DH + c * 32, o);
            tc_wait_ld();
#pragma unroll
            for (int q = 0; q < 32; ++q) o[q] = __float_as_uint(__uint_as_float(o[q]) * corr);
            tmem_st32(tmem_O + lane_off + half * DH + c * 32, o);
          }
          tc_wait_st();
        }
      }
      // this thread's 64 P values as bf16 pairs over its half of the S
      // buffer: columns st*128 + half*32 .. +32 (both halves have read their
      // S past the row-max barrier above)
      {
        uint32_t pw[32];
#pragma unroll
        for (int w = 0; w < 32; ++w) pw[w] = pack_bf16(s[2 * w], s[2 * w + 1]);
        tmem_st32(tmem + (uint32_t)(st * 128 + half * 32) + lane_off, pw);
        tc_wait_st();
      }
      tc_fence_before();
      mbar_arrive(bar(BAR_P_FULL));
      m_run = m_new;
    }
    if (ok && nt > 0) {
      ok = __all_sync(0xffffffffu, observe(nt));
      if (ok) tc_fence_after();
    }
    // speculative K/V copies this split did not use land in the buffers the
    // staging below reuses: wait for them first
    for (int it = nt; it < kStages; ++it)
      if (kv_early[it] && !(mbar_wait(bar(BAR_K_FULL + it), 0) && mbar_wait(bar(BAR_V_FULL + it), 0)))
        ok = false;
    if (nt == 0 && q_early && !mbar_wait(bar(BAR_Q_FULL), 0)) ok = false;  // no MMA waited it
    ok = __all_sync(0xffffffffu, ok);
    if (!ok && lane == 0) raise_status(a.status, kStTimeout);
    // row sum over both halves; every MMA of the CTA is done past this barrier
    red_l[half * kBM + r] = l_run;
    softmax_bar();
    const float l_tot = red_l[r] + red_l[kBM + r];
    const bool live = ok && nt > 0 && m_run != NEG_INF;

    if (S_kv == 1) {
      // ---- single split: normalise this row's O columns and write them
      const int rg = r0 + r;
      const int uu = rg / G, g = rg % G;
      const float inv = (live && l_tot > 0.f) ? 1.f / l_tot : 0.f;
      const size_t orow = (size_t)(off + uu) * a.Hq + (size_t)(h * G + g);
#pragma unroll
      for (int c = 0; c < DH / 32; ++c) {
        float o[32];
        tmem_ld32f(tmem_O + lane_off + half * DH + c * 32, o);
        tc_wait_ld();
        if (uu < n) {
          uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(a.out) + orow * D +
                                                half * DH + c * 32);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            dst[q] = make_uint4(pack_bf16(o[8 * q + 0] * inv, o[8 * q + 1] * inv),
                                pack_bf16(o[8 * q + 2] * inv, o[8 * q + 3] * inv),
                                pack_bf16(o[8 * q + 4] * inv, o[8 * q + 5] * inv),
                                pack_bf16(o[8 * q + 6] * inv, o[8 * q + 7] * inv));
        }
      }
      if (half == 0 && uu < n && a.lse_out)
        a.lse_out[orow] = live ? (m_run * sl2 + log2f(l_tot)) * kLn2 : NEG_INF;
    } else {
      // ---- this row's partial straight into the workspace, read back
      //      after the split barrier: O / l as bf16 plus (m base 2, l) in
      //      fp32.  Rows past the tree's last node are never read.
      const size_t unit = (size_t)blockIdx.z * gridDim.y + blockIdx.y;
      char* slab = reinterpret_cast<char*>(attn_slabs(a.ws, gridDim.y * gridDim.z)) +
                   (unit * (size_t)S_kv + (size_t)split) * L::kSlabBytes;
      uint4* slab8 = reinterpret_cast<uint4*>(slab);  // [D / 8][kBM] groups of 8 bf16
      const bool store = u < n;
      const float inv = (live && l_tot > 0.f) ? 1.f / l_tot : 0.f;
      // tcgen05.ld / wait::ld are warp-collective: the condition must be the
      // same for the 32 lanes (ok and nt are); per-row liveness only selects
      // what is stored
      if (ok && nt > 0) {
#pragma unroll
        for (int c = 0; c < DH / 32; ++c) {
          float o[32];
          tmem_ld32f(tmem_O + lane_off + half * DH + c * 32, o);
          tc_wait_ld();
          if (store) {
#pragma unroll
            for (int q = 0; q < 4; ++q)
              __stcg(slab8 + ((half * DH + c * 32) / 8 + q) * kBM + r,
                     make_uint4(pack_bf16(o[8 * q + 0] * inv, o[8 * q + 1] * inv),
                                pack_bf16(o[8 * q + 2] * inv, o[8 * q + 3] * inv),
                                pack_bf16(o[8 * q + 4] * inv, o[8 * q + 5] * inv),
                                pack_bf16(o[8 * q + 6] * inv, o[8 * q + 7] * inv)));
          }
        }
      } else if (store) {
        for (int c8 = 0; c8 < DH / 8; ++c8)
          __stcg(slab8 + (half * DH / 8 + c8) * kBM + r, make_uint4(0u, 0u, 0u, 0u));
      }
      if (half == 0 && store) {
        __stcg(reinterpret_cast<float*>(slab + L::kSlabM) + r, live ? m_run * sl2 : NEG_INF);
        __stcg(reinterpret_cast<float*>(slab + L::kSlabL) + r, live ? l_tot : 0.f);
      }
    }
  }
  tc_fence_before();
  if (S_kv == 1) {
    __syncthreads();  // TMEM reads are done
    if (warp == 1) {
      tc_fence_after();
      tmem_dealloc(tmem, 512);
    }
    return;
  }

  // ---- combine through L2: every CTA has written its partial rows.  The
  // cluster barrier (release / acquire at cluster scope) makes them visible
  // to the other CTAs of the cluster.  In a cooperative launch the CTAs of
  // a work item meet on a counter instead: thread 0 adds with release
  // semantics (after the block barrier, so it covers every thread's
  // stores) and waits, bounded, until all S_kv have arrived (acquire).
  const size_t unit = (size_t)blockIdx.z * gridDim.y + blockIdx.y;
  if (a.coop) {
    __syncthreads();
    if (tid == 0) {
      int* cnt = reinterpret_cast<int*>(a.ws) + 2 * unit;
      red_add_release_gpu(cnt, 1);
      const long long t0 = clock64();
      bool ok = true;
      while (ld_acquire_gpu(cnt) < S_kv) {
        if (clock64() - t0 > a.split_wait_cycles) {
          ok = false;
          break;
        }
        __nanosleep(64);
      }
      if (!ok) raise_status(a.status, kStTimeout);
      // every CTA of the item has passed the wait once the second counter
      // reaches S_kv: its last arrival returns both counters to zero for
      // the next launch
      if (atomicAdd(cnt + 1, 1) == S_kv - 1) {
        atomicExch(cnt, 0);
        atomicExch(cnt + 1, 0);
      }
    }
    __syncthreads();
  } else {
    cluster.sync();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  const char* slabs = reinterpret_cast<const char*>(attn_slabs(a.ws, gridDim.y * gridDim.z)) +
                      unit * (size_t)S_kv * L::kSlabBytes;
  switch (S_kv) {
    case 2: combine_rows<D, 2>(slabs, split, r0, G, n, off, h, a); break;
    case 3: combine_rows<D, 3>(slabs, split, r0, G, n, off, h, a); break;
    case 4: combine_rows<D, 4>(slabs, split, r0, G, n, off, h, a); break;
    case 5: combine_rows<D, 5>(slabs, split, r0, G, n, off, h, a); break;
    case 6: combine_rows<D, 6>(slabs, split, r0, G, n, off, h, a); break;
    case 7: combine_rows<D, 7>(slabs, split, r0, G, n, off, h, a); break;
    case 8: combine_rows<D, 8>(slabs, split, r0, G, n, off, h, a); break;
    case 9: combine_rows<D, 9>(slabs, split, r0, G, n, off, h, a); break;
    default: combine_rows<D, 10>(slabs, split, r0, G, n, off, h, a); break;
  }
}

template <int D>
cudaError_t launch_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                     const AttnArgs& a, SplitPlan plan, cudaStream_t s) {
  using L = Layout<D>;
  auto kern = tree_attn_split_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc);
  if (e != cudaSuccess) return e;
  const int G = a.Hq / a.Hkv;
  const int mtiles = (G * a.max_nodes + kBM - 1) / kBM;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(plan.splits, mtiles, a.B * a.Hkv);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kAlloc;
  cfg.stream = s;
  // programmatic dependent launch: this launch is dispatched while the
  // previous kernel on the stream finishes (its reads wait in the kernel)
  cudaLaunchAttribute attr[2];
  if (plan.coop) {
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
  } else {
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = plan.splits;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
  }
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, tq, tk, tv, a);
}

// clusters of `splits` CTAs of this kernel that can be resident at once
template <int D>
int max_active_clusters_d(int splits) {
  using L = Layout<D>;
  auto kern = tree_attn_split_kernel<D>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc) !=
      cudaSuccess)
    return 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits, 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kAlloc;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

// CTAs of this kernel resident on one SM
template <int D>
int blocks_per_sm_d() {
  using L = Layout<D>;
  auto kern = tree_attn_split_kernel<D>;
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

// How to split the keys.  Cost model: waves of resident work items times
// the per-CTA time, a fixed part plus one part per 128-key tile of its
// split, plus the combine when the keys are split.  The constants are fitted
// to a measured timeline of the Llama-3-8B-shaped launch (9 splits of 17
// key tiles): launch to first S product 3.5 us, 1.05 us per key tile, and
// 4.7 us from the last product to the merged rows (partials through L2, the
// counter barrier, the merge).  A cluster path holds up to 8 splits, with
// the resident clusters per split count from the occupancy API; a
// cooperative path holds up to kAttnMaxSplits when the whole grid is
// resident at once (one wave).  On a tie the cluster path wins (no
// counters).  Occupancy figures are cached per device and head size.
SplitPlan tree_attn_split_plan(int D, int B, int Hkv, int mtiles, int S_max, int num_sms,
                                double* cost_us) {
  static int cache[64][2][kClusterMaxSplits + 1] = {};
  static int bps_cache[64][2] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = 0;
  const int di = D == 64 ? 0 : 1;
  const long long units = (long long)B * Hkv * mtiles;
  const int tiles = (S_max + kBN - 1) / kBN;
  const double kFixed = 3.5, kCombine = 4.7, kPerTile = 1.05;  // microseconds
  int& bps = bps_cache[dev][di];
  if (bps == 0) bps = di ? blocks_per_sm_d<128>() : blocks_per_sm_d<64>();
  const long long coop_cap = (long long)(bps > 0 ? bps : 1) * num_sms;
  SplitPlan best{1, 0};
  double best_cost = 1e30;
  for (int s = 1; s <= kAttnMaxSplits; ++s) {
    if (s > 1 && s > tiles) break;
    const double per_cta = kFixed + (s > 1 ? kCombine : 0.0) + kPerTile * (double)((tiles + s - 1) / s);
    if (s <= kClusterMaxSplits) {
      int& fit = cache[dev][di][s];
      if (fit == 0) fit = di ? max_active_clusters_d<128>(s) : max_active_clusters_d<64>(s);
      const int resident = fit > 0 ? fit : (s == 1 ? num_sms : num_sms / (2 * s));
      if (resident > 0) {
        const double cost = (double)((units + resident - 1) / resident) * per_cta;
        if (cost < best_cost - 1e-9) {
          best_cost = cost;
          best = SplitPlan{s, 0};
        }
      }
    }
    if (s > 1 && units * s <= coop_cap && per_cta < best_cost - 1e-9) {
      best_cost = per_cta;
      best = SplitPlan{s, 1};
    }
  }
  if (cost_us) *cost_us = best_cost;
  return best;
}

size_t tree_attn_split_ws_bytes(int D, int B, int Hkv, int mtiles, int splits) {
  if (splits <= 1) return 0;
  const size_t slab = D == 64 ? (size_t)Layout<64>::kSlabBytes : (size_t)Layout<128>::kSlabBytes;
  const long long units = (long long)B * Hkv * mtiles;
  return attn_counter_bytes(units) + (size_t)units * splits * slab;
}

cudaError_t launch_tree_attn_split(const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                                   const CUtensorMap& tm_v, const AttnArgs& a, SplitPlan plan,
                                   cudaStream_t s) {
  if (a.D == 64) return launch_d<64>(tm_q, tm_k, tm_v, a, plan, s);
  return launch_d<128>(tm_q, tm_k, tm_v, a, plan, s);
}

}  // namespace tg
