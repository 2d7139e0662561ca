// treegraft_accept_noalloc: the accept walk for callers that cannot allocate
// device memory.
//
// treegraft_accept needs a caller-provided scratch buffer (one int32 per
// node for the target argmax, one ticket counter per tree).  Some callers
// have no way to obtain one: a plugin that an inference engine hands only
// its inputs and outputs, or code running where every device allocation
// must go through a memory pool it cannot reach.  This entry point keeps
// that scratch in a fixed array that lives in the library itself, so the
// caller passes inputs and outputs only.
//
// The array below is a file-scope __device__ variable: every GPU that loads
// the library holds its kNoAllocScratchWords * 4 bytes (about 272 KB) until
// the process exits.  In host code the name `g_accept_scratch` is only a
// host-side stand-in, not a device address, so the host looks up the real
// device address once per device with cudaGetSymbolAddress and passes that
// pointer to the kernel.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/treegraft.h"
#include "launch.h"

namespace tg {
namespace {

constexpr int kNoAllocMaxNodes = TG_NOALLOC_MAX_NODES;
constexpr int kNoAllocMaxTrees = TG_NOALLOC_MAX_TREES;
constexpr int kNoAllocScratchWords = kNoAllocMaxNodes + kNoAllocMaxTrees;

// a call's B ticket counters, then the argmax slots of its n_total nodes
static __device__ __align__(256) int32_t g_accept_scratch[kNoAllocScratchWords];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
int32_t* g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch array on the current device; looked up once
// per device (the first call on that device does it).
int32_t* scratch_ptr() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!g_scratch_ptr[d]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_accept_scratch) != cudaSuccess || p == nullptr) return nullptr;
    g_scratch_ptr[d] = static_cast<int32_t*>(p);
  }
  return g_scratch_ptr[d];
}

}  // namespace
}  // namespace tg

extern "C" int treegraft_accept_noalloc(const void* target_logits, int dtype, int V, int64_t ld,
                                        const int32_t* token, const int32_t* parent,
                                        const int32_t* node_off, int B, int max_nodes,
                                        int n_total, int path_cap, int32_t* path,
                                        int32_t* accept_len, int32_t* bonus, void* stream) {
  using namespace tg;
  if (!target_logits || !token || !parent || !node_off || !path || !accept_len || !bonus)
    return TG_ERR_INVALID_ARG;
  if (dtype != TG_BF16 && dtype != TG_F32) return TG_ERR_INVALID_ARG;
  if (B < 1 || V < 1 || ld < V || n_total < 1 || path_cap < 1 || max_nodes < 1 ||
      max_nodes > TG_MAX_TREE_NODES || (long long)n_total > (long long)B * max_nodes)
    return TG_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(target_logits) & (dtype == TG_BF16 ? 1 : 3)) != 0)
    return TG_ERR_INVALID_ARG;  // elements must sit at their natural alignment
  // the fixed scratch array bounds the problem size
  if (n_total > kNoAllocMaxNodes || B > kNoAllocMaxTrees) return TG_ERR_UNSUPPORTED;
  if (V > (dtype == TG_BF16 ? 262144 : 131072)) return TG_ERR_UNSUPPORTED;
  int* st = status_word_ptr();
  int32_t* scratch = scratch_ptr();
  if (!st || !scratch) return TG_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the tickets and argmax slots must start at zero; a well-formed call
  // leaves them so, but the array keeps whatever a malformed one left, so
  // clear them (tickets [0, B), slots [B, B + n_total)) before the launch
  if (cudaMemsetAsync(scratch, 0, sizeof(int32_t) * ((size_t)B + (size_t)n_total), s) != cudaSuccess)
    return TG_ERR_CUDA;
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
  a.tickets = scratch;
  a.am = scratch + B;
  a.status = st;
  return launch_accept(a, s) == cudaSuccess ? TG_OK : TG_ERR_CUDA;
}
