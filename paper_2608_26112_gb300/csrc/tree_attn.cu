// tree_attn: ancestor-masked GQA tree attention on the 5th-generation tensor
// cores (Sec. 3.1 tree attention; Algorithm 3 tree mask).
//
// Work item = (tree b, kv-head h, 128-row query tile, KV split).  The
// query rows of one kv-head are the G * n pairs (node u, q-head h*G + g),
// row index u*G + g, so the tile is a dense 128 x D bf16 operand: a single
// 3-D TMA box {64, G, 128/G} of q gathers it.  The key axis (prefix
// [0, P) followed by the tree slots [P, P+n)) is cut into 128-key tiles;
// the S_kv CTAs of a thread-block cluster split those tiles and combine
// their partial (max, sum, O) rows over DSMEM at the end, so nothing but
// the final bf16 output and the lse touch global memory.
//
// Warp roles (192 threads, one CTA per SM):
//   warp 0      TMA producer: Q once, then K and V tiles into a 2-stage ring;
//   warp 1      TMEM owner and MMA issuer: S = Q K^T (M=128, N=128, K=D) and
//               O += P V (M=128, N=D, K=128), bf16 in, fp32 accumulate in
//               TMEM, completion signalled by tcgen05.commit on mbarriers;
//   warps 2..5  softmax: one query row per thread (TMEM lane = row), read
//               S with tcgen05.ld, apply the ancestor mask from a per-node
//               bitmask in shared memory, online max / sum in base 2, write
//               P as bf16 into the swizzled operand layout, rescale O in
//               TMEM when the running max grows; finally the combine.
// The MMA thread issues S(i+1) before PV(i), so the softmax of tile i+1
// overlaps the PV product of tile i.  Every mbarrier wait is bounded.
#include <cooperative_groups.h>

#include "common.cuh"
#include "launch.h"

namespace cg = cooperative_groups;

namespace tg {
namespace {

constexpr int kBM = 128;     // query rows per tile (TMEM lanes)
constexpr int kBN = 128;     // keys per KV tile
constexpr int kStages = 2;   // K/V ring depth
constexpr int kThreads = 192;
constexpr int kAncWords = 9; // 256 tree slots + one zero word
constexpr int kRegion = 128 * 128;  // 128 rows x 128 bytes: one swizzled operand region
constexpr float kLn2 = 0.6931471805599453f;

enum { BAR_KV_FULL = 0, BAR_KV_EMPTY = 2, BAR_Q_FULL = 4, BAR_S_FULL = 5, BAR_P_FULL = 6,
       BAR_O_DONE = 7, kNumBars = 8 };

constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

template <int D>
struct Layout {
  static constexpr int kQBytes = kBM * D * 2;
  static constexpr int kKVBytes = kBN * D * 2;
  static constexpr int kPBytes = kBM * kBN * 2;
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQBytes;
  static constexpr int kOffV = kOffK + kStages * kKVBytes;
  static constexpr int kOffP = kOffV + kStages * kKVBytes;
  static constexpr int kOffAnc = kOffP + kPBytes;                  // (kBM + 1) rows
  static constexpr int kOffPar = align_up(kOffAnc + (kBM + 1) * kAncWords * 4, 16);
  static constexpr int kOffM = align_up(kOffPar + 256 * 4, 16);
  static constexpr int kOffL = align_up(kOffM + kBM * 4, 16);
  static constexpr int kOffBar = align_up(kOffL + kBM * 4, 16);    // mbarriers: 8-byte aligned
  static constexpr int kOffTmem = align_up(kOffBar + kNumBars * 8, 16);
  static constexpr int kBytes = kOffTmem + 16;
  static constexpr int kAlloc = kBytes + 1024;                     // 1024-byte alignment slack
  // fp32 O staging for the combine, padded rows, reusing the K/V ring
  static constexpr int kOStride = D + 4;
  static constexpr int kOffO = kOffK;
  static_assert(kBM * kOStride * 4 <= 2 * kStages * kKVBytes, "O staging must fit in K/V ring");
  static_assert(kAlloc <= 227 * 1024, "shared memory budget");
  static_assert(kOffQ % 1024 == 0 && kOffK % 1024 == 0 && kOffV % 1024 == 0 && kOffP % 1024 == 0,
                "128-byte-swizzled operand tiles need 1024-byte alignment");
  static_assert(kOffBar % 8 == 0 && kOffTmem % 4 == 0 && kOffM % 16 == 0 && kOffL % 16 == 0,
                "mbarrier / scalar alignment");
  static_assert((kOStride * 4) % 16 == 0, "float4 rows of the O staging");
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

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    tree_attn_kernel(const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ CUtensorMap tm_v, const AttnArgs a) {
  using L = Layout<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  cg::cluster_group cluster = cg::this_cluster();
  const int S_kv = (int)cluster.num_blocks();
  const int split = (int)cluster.block_rank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = a.Hq / a.Hkv;
  const int b = blockIdx.z / a.Hkv, h = blockIdx.z % a.Hkv;
  const int r0 = blockIdx.y * kBM;

  int* par_s = reinterpret_cast<int*>(smem + L::kOffPar);
  uint32_t* anc_s = reinterpret_cast<uint32_t*>(smem + L::kOffAnc);
  float* m_s = reinterpret_cast<float*>(smem + L::kOffM);
  float* l_s = reinterpret_cast<float*>(smem + L::kOffL);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kOffTmem);
  const uint32_t bar0 = smem_u32(smem + L::kOffBar);
  auto bar = [&](int i) -> uint32_t { return bar0 + 8u * (uint32_t)i; };
  const uint32_t q_base = smem_u32(smem + L::kOffQ);
  const uint32_t k_base = smem_u32(smem + L::kOffK);
  const uint32_t v_base = smem_u32(smem + L::kOffV);
  const uint32_t p_base = smem_u32(smem + L::kOffP);

  // ---- shape checks; every exit here is uniform over the cluster
  const int off = a.node_off[b];
  const int n = a.node_off[b + 1] - off;
  const int P = a.prefix_len[b];
  if (n < 1 || n > 256 || P < 0 || P + n > a.S_max || off < 0 || off + n > a.n_total) {
    if (split == 0 && tid == 0 && blockIdx.y == 0) raise_status(a.status, kStTree);
    return;
  }
  if (r0 >= G * n) return;
  int bad = 0;
  for (int v = tid; v < n; v += kThreads) {
    const int p = a.parent[off + v];
    par_s[v] = p;
    bad |= (v == 0) ? (p != -1) : (p < 0 || p >= v);
  }
  if (__syncthreads_or(bad)) {
    if (split == 0 && tid == 0 && blockIdx.y == 0) raise_status(a.status, kStTree);
    return;
  }

  // ---- ancestor bitmasks of the nodes of this tile (row kBM stays zero)
  const int u_base = r0 / G;
  const int tile_nodes = min(kBM / G, n - u_base);
  for (int i = tid; i < (kBM + 1) * kAncWords; i += kThreads) anc_s[i] = 0u;
  __syncthreads();
  for (int t = tid; t < tile_nodes; t += kThreads) {
    uint32_t* w = anc_s + t * kAncWords;
    for (int v = u_base + t; v >= 0; v = par_s[v]) w[v >> 5] |= 1u << (v & 31);
  }

  // ---- barriers and TMEM (S: columns [0,128), O: columns [128, 128 + D))
  if (tid == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(BAR_KV_FULL + s), 1);
      mbar_init(bar(BAR_KV_EMPTY + s), 1);
    }
    mbar_init(bar(BAR_Q_FULL), 1);
    mbar_init(bar(BAR_S_FULL), 1);
    mbar_init(bar(BAR_P_FULL), 128);
    mbar_init(bar(BAR_O_DONE), 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), 256);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t tmem_S = tmem;
  const uint32_t tmem_O = tmem + 128u;

  // ---- this split's KV tiles
  const int Lk = P + n;
  const int T = (Lk + kBN - 1) / kBN;
  const int t0 = (int)((long long)split * T / S_kv);
  const int t1 = (int)((long long)(split + 1) * T / S_kv);
  const int nt = t1 - t0;
  const int kv_row0 = (b * a.Hkv + h) * a.S_max;

  if (warp == 0) {
    // ------------------------------------------------ TMA producer
    if (lane == 0 && nt > 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      mbar_arrive_expect_tx(bar(BAR_Q_FULL), L::kQBytes);
#pragma unroll
      for (int c = 0; c < D / 64; ++c)
        tma_load_3d(q_base + c * kRegion, &tm_q, c * 64, h * G, off + u_base, bar(BAR_Q_FULL));
      for (int it = 0; it < nt; ++it) {
        const int st = it & 1;
        if (it >= kStages && !mbar_wait(bar(BAR_KV_EMPTY + st), ((it >> 1) - 1) & 1)) {
          raise_status(a.status, kStTimeout);
          break;
        }
        mbar_arrive_expect_tx(bar(BAR_KV_FULL + st), 2 * L::kKVBytes);
        const int y = kv_row0 + (t0 + it) * kBN;
#pragma unroll
        for (int c = 0; c < D / 64; ++c) {
          tma_load_2d(k_base + st * L::kKVBytes + c * kRegion, &tm_k, c * 64, y,
                      bar(BAR_KV_FULL + st));
          tma_load_2d(v_base + st * L::kKVBytes + c * kRegion, &tm_v, c * 64, y,
                      bar(BAR_KV_FULL + st));
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer
    if (lane == 0 && nt > 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(kBM, kBN, false);
      constexpr uint32_t kIdO = idesc_bf16_f32(kBM, D, true);
      bool ok = mbar_wait(bar(BAR_Q_FULL), 0);
      for (int it = 0; ok && it <= nt; ++it) {
        if (it < nt) {
          const int st = it & 1;
          ok = mbar_wait(bar(BAR_KV_FULL + st), (it >> 1) & 1);
          if (ok && it > 0) ok = mbar_wait(bar(BAR_P_FULL), (it - 1) & 1);
          if (!ok) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t qa = q_base + (kk >> 2) * kRegion + (kk & 3) * 32;
            const uint32_t ka = k_base + st * L::kKVBytes + (kk >> 2) * kRegion + (kk & 3) * 32;
            tc_mma_f16(tmem_S, smem_desc_sw128(qa, 16, 1024), smem_desc_sw128(ka, 16, 1024), kIdS,
                       kk > 0 ? 1u : 0u);
          }
          tc_commit(bar(BAR_S_FULL));
        } else {
          ok = mbar_wait(bar(BAR_P_FULL), (it - 1) & 1);
          if (!ok) break;
          tc_fence_after();
        }
        if (it > 0) {
          const int jt = it - 1, sp = jt & 1;
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk) {
            const uint32_t pa = p_base + (kk >> 2) * kRegion + (kk & 3) * 32;
            const uint32_t va = v_base + sp * L::kKVBytes + kk * 16 * 128;
            tc_mma_f16(tmem_O, smem_desc_sw128(pa, 16, 1024), smem_desc_sw128(va, kRegion, 1024),
                       kIdO, (jt > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(bar(BAR_O_DONE));
          tc_commit(bar(BAR_KV_EMPTY + sp));
        }
      }
      if (!ok) raise_status(a.status, kStTimeout);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------ softmax warps
    const int q4 = warp & 3;              // TMEM lane quarter of this warp
    const int r = q4 * 32 + lane;         // tile row = TMEM lane
    const int rg = r0 + r;
    const int u = rg / G;
    const uint32_t* anc = anc_s + (u < n ? (u - u_base) : kBM) * kAncWords;
    const uint32_t lane_off = (uint32_t)(q4 * 32) << 16;
    const float sl2 = a.scale_log2;
    const float NEG_INF = __int_as_float(0xff800000);
    float m_run = NEG_INF, l_run = 0.f;
    bool ok = true;
    for (int it = 0; it < nt; ++it) {
      const int st = it & 1;
      const int key0 = (t0 + it) * kBN;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_S_FULL), it & 1));
      if (!ok) break;
      tc_fence_after();
      float s[kBN];
#pragma unroll
      for (int c = 0; c < kBN / 32; ++c)
        tmem_ld32f(tmem_S + lane_off + c * 32, *reinterpret_cast<float(*)[32]>(&s[c * 32]));
      tc_wait_ld();
      float mx = NEG_INF;
      if (key0 + kBN <= P) {
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          s[c] *= sl2;
          mx = fmaxf(mx, s[c]);
        }
      } else {
        uint32_t mw[kBN / 32];
#pragma unroll
        for (int w = 0; w < kBN / 32; ++w) mw[w] = mask_word(anc, key0 + 32 * w - P);
#pragma unroll
        for (int c = 0; c < kBN; ++c) {
          const bool vis = (mw[c >> 5] >> (c & 31)) & 1u;
          s[c] = vis ? s[c] * sl2 : NEG_INF;
          mx = fmaxf(mx, s[c]);
        }
      }
      const float m_new = fmaxf(m_run, mx);
      const float m_use = (m_new == NEG_INF) ? 0.f : m_new;
      const float corr = ex2(m_run - m_use);
      float rs = 0.f;
#pragma unroll
      for (int c = 0; c < kBN; ++c) {
        s[c] = ex2(s[c] - m_use);
        rs += s[c];
      }
      l_run = l_run * corr + rs;
      if (it > 0) {
        // PV(it-1) must finish before O is rescaled and P is overwritten
        ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_O_DONE), (it - 1) & 1));
        if (!ok) break;
        tc_fence_after();
        if (__any_sync(0xffffffffu, m_new > m_run)) {
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            tmem_ld32(tmem_O + lane_off + c * 32, o);
            tc_wait_ld();
#pragma unroll
            for (int q = 0; q < 32; ++q) o[q] = __float_as_uint(__uint_as_float(o[q]) * corr);
            tmem_st32(tmem_O + lane_off + c * 32, o);
          }
          tc_wait_st();
        }
      }
      if (key0 + kBN > Lk) {
        // last tile of the sequence: V rows past the end may hold anything;
        // zero them so that 0-weight rows contribute exactly 0
        ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_KV_FULL + st), (it >> 1) & 1));
        if (!ok) break;
        if (key0 + r >= Lk) {
#pragma unroll
          for (int c = 0; c < D / 64; ++c)
#pragma unroll
            for (int q = 0; q < 8; ++q)
              st_shared_v4(v_base + st * L::kKVBytes + c * kRegion + r * 128 + q * 16,
                           make_uint4(0u, 0u, 0u, 0u));
        }
      }
      // P row -> shared memory, bf16, 128-byte swizzled K-major operand layout
#pragma unroll
      for (int ch = 0; ch < kBN / 8; ++ch) {
        const uint4 w = make_uint4(pack_bf16(s[ch * 8 + 0], s[ch * 8 + 1]),
                                   pack_bf16(s[ch * 8 + 2], s[ch * 8 + 3]),
                                   pack_bf16(s[ch * 8 + 4], s[ch * 8 + 5]),
                                   pack_bf16(s[ch * 8 + 6], s[ch * 8 + 7]));
        const int region = ch >> 3, chunk = ch & 7;
        st_shared_v4(p_base + region * kRegion + r * 128 + ((chunk ^ (r & 7)) << 4), w);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(bar(BAR_P_FULL));
      m_run = m_new;
    }
    if (ok && nt > 0) {
      ok = __all_sync(0xffffffffu, mbar_wait(bar(BAR_O_DONE), (nt - 1) & 1));
      if (ok) tc_fence_after();
    }
    float* ost = reinterpret_cast<float*>(smem + L::kOffO) + r * L::kOStride;
    if (ok && nt > 0) {
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t o[32];
        tmem_ld32(tmem_O + lane_off + c * 32, o);
        tc_wait_ld();
#pragma unroll
        for (int q = 0; q < 32; q += 4)
          *reinterpret_cast<float4*>(ost + c * 32 + q) =
              make_float4(__uint_as_float(o[q]), __uint_as_float(o[q + 1]),
                          __uint_as_float(o[q + 2]), __uint_as_float(o[q + 3]));
      }
    } else {
      for (int c = 0; c < D; c += 4) *reinterpret_cast<float4*>(ost + c) = make_float4(0, 0, 0, 0);
      m_run = NEG_INF;
      l_run = 0.f;
      if (!ok && lane == 0) raise_status(a.status, kStTimeout);
    }
    m_s[r] = m_run;
    l_s[r] = l_run;
  }

  // ---- combine the S_kv partials of each row over DSMEM
  tc_fence_before();
  cluster.sync();
  if (warp >= 2) {
    const int st = tid - 64;
    const int rpc = kBM / S_kv;
    const int rbeg = split * rpc;
    constexpr int C4 = D / 4;
    const float NEG_INF = __int_as_float(0xff800000);
    for (int item = st; item < rpc * C4; item += 128) {
      const int rr = rbeg + item / C4, c4 = item % C4;
      const int rg = r0 + rr;
      const int uu = rg / G, g = rg % G;
      if (uu >= n) continue;
      float M = NEG_INF;
      for (int s = 0; s < S_kv; ++s) M = fmaxf(M, cluster.map_shared_rank(m_s, s)[rr]);
      float Ls = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      if (M != NEG_INF) {
        for (int s = 0; s < S_kv; ++s) {
          const float ms = cluster.map_shared_rank(m_s, s)[rr];
          if (ms == NEG_INF) continue;
          const float w = ex2(ms - M);
          Ls += w * cluster.map_shared_rank(l_s, s)[rr];
          const float* po = reinterpret_cast<const float*>(smem + L::kOffO);
          const float4 o = *reinterpret_cast<const float4*>(
              cluster.map_shared_rank(po, s) + rr * L::kOStride + c4 * 4);
          acc.x += w * o.x;
          acc.y += w * o.y;
          acc.z += w * o.z;
          acc.w += w * o.w;
        }
      }
      const float inv = (Ls > 0.f) ? 1.f / Ls : 0.f;
      const size_t orow = (size_t)(off + uu) * a.Hq + (size_t)(h * G + g);
      uint2 pk;
      pk.x = pack_bf16(acc.x * inv, acc.y * inv);
      pk.y = pack_bf16(acc.z * inv, acc.w * inv);
      *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(a.out) + orow * D + c4 * 4) = pk;
      if (c4 == 0 && a.lse_out) a.lse_out[orow] = (M + log2f(Ls)) * kLn2;
    }
  }
  cluster.sync();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, 256);
  }
}

template <int D>
cudaError_t launch_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                     const AttnArgs& a, int splits, cudaStream_t s) {
  using L = Layout<D>;
  auto kern = tree_attn_kernel<D>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::kAlloc);
  if (e != cudaSuccess) return e;
  const int G = a.Hq / a.Hkv;
  const int mtiles = (G * a.max_nodes + kBM - 1) / kBM;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(splits, mtiles, a.B * a.Hkv);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = L::kAlloc;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = splits;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, tq, tk, tv, a);
}

}  // namespace

// KV splits per work item: the power of two in {1, 2, 4, 8} whose grid fills
// the SMs best (one CTA per SM), preferring fewer splits on near ties.
int tree_attn_pick_splits(int B, int Hkv, int mtiles, int S_max, int num_sms) {
  const long long units = (long long)B * Hkv * mtiles;
  const int max_tiles = (S_max + kBN - 1) / kBN;
  int best = 1;
  double best_eff = -1.0;
  for (int s = 1; s <= 8; s *= 2) {
    if (s > 1 && s > max_tiles) break;
    const long long ctas = units * s;
    const long long waves = (ctas + num_sms - 1) / num_sms;
    const double eff = (double)ctas / (double)(waves * num_sms);
    if (eff > best_eff + 0.03) {
      best_eff = eff;
      best = s;
    }
  }
  return best;
}

cudaError_t launch_tree_attn(const CUtensorMap& tm_q, const CUtensorMap& tm_k,
                             const CUtensorMap& tm_v, const AttnArgs& a, int kv_splits,
                             cudaStream_t s) {
  if (a.D == 64) return launch_d<64>(tm_q, tm_k, tm_v, a, kv_splits, s);
  return launch_d<128>(tm_q, tm_k, tm_v, a, kv_splits, s);
}

}  // namespace tg
