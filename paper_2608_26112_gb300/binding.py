"""Python binding of libtreegraft.so (the C ABI in include/treegraft.h).

Argument marshalling only: each wrapper checks the torch tensors it is
given, passes their device pointers and the current CUDA stream to the C
entry point of the same name, and turns a non-zero status into an
exception.  Every step of the computation runs in the library's kernels;
there is no CPU fallback, and a missing library is an error.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtreegraft.so")

TG_OK = 0
TG_BF16, TG_F32 = 0, 1
MAX_TREE_NODES = 256
MAX_TOPK = 32
MAX_PRUNE_NODES = 1024
MAX_GROW_NODES = 1024
NGRAM_MAX_N = 8

_lib = None


class TreeGraftError(RuntimeError):
    def __init__(self, fn: str, status: int):
        msg = lib().treegraft_status_string(status).decode() if _lib else str(status)
        super().__init__(f"{fn} returned status {status} ({msg})")
        self.status = status


_c_int, _c_i64, _c_f32, _c_vp, _c_size = (ctypes.c_int, ctypes.c_int64, ctypes.c_float,
                                          ctypes.c_void_p, ctypes.c_size_t)

_SIGNATURES = {
    "treegraft_tree_attn": [_c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_int, _c_int, _c_int,
                            _c_int, _c_int, _c_int, _c_int, _c_f32, _c_vp, _c_vp, _c_vp, _c_size,
                            _c_vp],
    "treegraft_tree_attn_workspace_size": [_c_int, _c_int, _c_int, _c_int, _c_int],
    "treegraft_expand_topk": [_c_vp, _c_int, _c_int, _c_int, _c_i64, _c_int, _c_vp, _c_vp,
                              _c_int, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp],
    "treegraft_rescore_select": [_c_vp, _c_vp, _c_int, _c_i64, _c_vp, _c_vp, _c_vp, _c_vp,
                                 _c_int, _c_int, _c_int, _c_int, _c_vp, _c_vp, _c_vp, _c_vp,
                                 _c_vp],
    "treegraft_accept_workspace_size": [_c_int, _c_int],
    "treegraft_accept": [_c_vp, _c_int, _c_int, _c_i64, _c_vp, _c_vp, _c_vp, _c_int, _c_int,
                         _c_int, _c_int, _c_vp, _c_vp, _c_vp, _c_vp, _c_size, _c_vp],
    "treegraft_accept_noalloc": [_c_vp, _c_int, _c_int, _c_i64, _c_vp, _c_vp, _c_vp, _c_int,
                                 _c_int, _c_int, _c_int, _c_vp, _c_vp, _c_vp, _c_vp],
    "treegraft_global_prune": [_c_vp, _c_vp, _c_vp, _c_int, _c_int, _c_int, _c_int, _c_int,
                               _c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp],
    "treegraft_grow_workspace_size": [_c_int, _c_int, _c_int],
    "treegraft_grow_step": [_c_int, _c_vp, _c_int, _c_int, _c_i64, _c_int, _c_int, _c_int, _c_int,
                            _c_int, _c_int, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp,
                            _c_size, _c_vp],
    "treegraft_accept_sample_workspace_size": [_c_int, _c_int],
    "treegraft_accept_sample": [_c_vp, _c_int, _c_int, _c_i64, _c_f32, _c_vp, _c_vp, _c_vp, _c_int,
                                _c_int, _c_int, _c_vp, _c_int, _c_vp, _c_vp, _c_vp, _c_vp, _c_size,
                                _c_vp],
    "treegraft_ngram_index_bytes": [_c_int, _c_int, _c_int],
    "treegraft_ngram_build": [_c_vp, _c_vp, _c_int, _c_int, _c_int, _c_vp, _c_size, _c_vp],
    "treegraft_ngram_cache": [_c_vp, _c_int, _c_int, _c_int, _c_i64, _c_int, _c_vp, _c_vp, _c_vp],
    "treegraft_ngram_draft": [_c_vp, _c_size, _c_int, _c_int, _c_int, _c_vp, _c_vp, _c_int, _c_vp,
                              _c_vp, _c_vp, _c_vp, _c_int, _c_vp, _c_int, _c_vp, _c_int, _c_vp,
                              _c_vp, _c_vp, _c_vp, _c_vp, _c_vp],
    "treegraft_ngram_grow_step": [_c_vp, _c_size, _c_int, _c_int, _c_int, _c_vp, _c_vp, _c_int,
                                  _c_vp, _c_vp, _c_int, _c_int, _c_int, _c_int, _c_int, _c_vp,
                                  _c_vp, _c_vp, _c_vp, _c_vp, _c_vp],
    "treegraft_last_device_status": [_c_vp],
    "treegraft_set_wait_budget": [_c_i64],
    "treegraft_graft_expand": [_c_vp, _c_int, _c_int, _c_int, _c_i64, _c_int, _c_int, _c_vp,
                               _c_int, _c_int, _c_int, _c_vp, _c_vp, _c_vp, _c_vp, _c_vp],
    "treegraft_status_string": [_c_int],
}
_RESTYPES = {"treegraft_accept_workspace_size": _c_size,
             "treegraft_grow_workspace_size": _c_size,
             "treegraft_ngram_index_bytes": _c_size,
             "treegraft_accept_sample_workspace_size": _c_size,
             "treegraft_tree_attn_workspace_size": _c_size,
             "treegraft_status_string": ctypes.c_char_p}


def lib() -> ctypes.CDLL:
    """Load libtreegraft.so (built by paper_2608_26112_gb300.build)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build it with "
                "`python -m paper_2608_26112_gb300.build` (nvcc, sm_103a)")
        dll = ctypes.CDLL(LIB_PATH)
        for name, argt in _SIGNATURES.items():
            fn = getattr(dll, name)
            fn.argtypes = argt
            fn.restype = _RESTYPES.get(name, _c_int)
        _lib = dll
    return _lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(fn: str, st: int):
    if st != TG_OK:
        raise TreeGraftError(fn, st)


def _need(t, dtype, name, device=True):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if device and not t.is_cuda:
        raise ValueError(f"{name} must live on a CUDA device")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _logit_dtype(t):
    if t.dtype == torch.bfloat16:
        return TG_BF16
    if t.dtype == torch.float32:
        return TG_F32
    raise TypeError("logits must be bfloat16 or float32")


def tree_attn_workspace_size(B, max_nodes, Hq, Hkv, D) -> int:
    return int(lib().treegraft_tree_attn_workspace_size(B, int(max_nodes), Hq, Hkv, D))


def tree_attn(q, k_cache, v_cache, prefix_len, parent, node_off, max_nodes, *, scale=0.0,
              out=None, lse_out=None, ws=None, stream=None):
    """Ancestor-masked GQA tree attention.  q [n_total, Hq, D] bf16,
    k_cache / v_cache [B, Hkv, S_max, D] bf16, prefix_len [B] int32,
    parent [n_total] int32 (local ids), node_off [B+1] int32.  ws: uint8
    scratch of tree_attn_workspace_size() bytes (allocated here if None).
    Returns (out [n_total, Hq, D] bf16, lse_out or None)."""
    _need(q, torch.bfloat16, "q")
    _need(k_cache, torch.bfloat16, "k_cache")
    _need(v_cache, torch.bfloat16, "v_cache")
    for t, nm in ((prefix_len, "prefix_len"), (parent, "parent"), (node_off, "node_off")):
        _need(t, torch.int32, nm)
    n_total, Hq, D = q.shape
    B, Hkv, S_max, D2 = k_cache.shape
    if D2 != D or tuple(v_cache.shape) != tuple(k_cache.shape):
        raise ValueError("q / k_cache / v_cache shapes disagree")
    if out is None:
        out = torch.empty_like(q)
    _need(out, torch.bfloat16, "out")
    if lse_out is not None:
        _need(lse_out, torch.float32, "lse_out")
    if ws is None:
        ws = torch.zeros(max(16, tree_attn_workspace_size(B, max_nodes, Hq, Hkv, D)),
                         dtype=torch.uint8, device=q.device)
    _need(ws, torch.uint8, "ws")
    st = lib().treegraft_tree_attn(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(prefix_len),
                                   _ptr(parent), _ptr(node_off), B, int(max_nodes), n_total, Hq,
                                   Hkv, D, S_max, float(scale), _ptr(out), _ptr(lse_out),
                                   _ptr(ws), ws.numel(), _stream(stream))
    _check("treegraft_tree_attn", st)
    return out, lse_out


def expand_topk(logits, parent_score, k, *, row_idx=None, V=None, out=None, lse_out=None,
                stream=None):
    """Per-row log-softmax + exact top-k + cumulative score.  logits
    [logit_rows, ld] bf16/fp32 (V <= ld columns used), parent_score [rows]
    fp32, row_idx [rows] int32 or None.  Returns (tok, logprob, score, lse)."""
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise ValueError("logits must be 2-D with unit column stride")
    if not logits.is_cuda:
        raise ValueError("logits must live on a CUDA device")
    dt = _logit_dtype(logits)
    _need(parent_score, torch.float32, "parent_score")
    rows = parent_score.shape[0]
    if row_idx is not None:
        _need(row_idx, torch.int32, "row_idx")
    V = logits.shape[1] if V is None else int(V)
    dev = logits.device
    if out is None:
        out = (torch.empty(rows, k, dtype=torch.int32, device=dev),
               torch.empty(rows, k, dtype=torch.float32, device=dev),
               torch.empty(rows, k, dtype=torch.float32, device=dev))
    tok, lp, sc = out
    st = lib().treegraft_expand_topk(_ptr(logits), dt, logits.shape[0], V, logits.stride(0), rows,
                                     _ptr(row_idx), _ptr(parent_score), int(k), _ptr(tok),
                                     _ptr(lp), _ptr(sc), _ptr(lse_out), _stream(stream))
    _check("treegraft_expand_topk", st)
    return tok, lp, sc, lse_out


def rescore_select(weak_edge, strong_lp, parent, token, visited, node_off, max_nodes, N, *,
                   V=None, out=None, stream=None):
    """Stronger-drafter rescoring + top-N reselection.  Returns (edge, score,
    selected [B, N], n_selected [B])."""
    _need(weak_edge, torch.float32, "weak_edge")
    if strong_lp.dim() != 2 or strong_lp.stride(1) != 1 or strong_lp.dtype != torch.float32:
        raise ValueError("strong_lp must be 2-D float32 with unit column stride")
    for t, nm in ((parent, "parent"), (token, "token"), (node_off, "node_off")):
        _need(t, torch.int32, nm)
    _need(visited, torch.uint8, "visited")
    n_total = parent.shape[0]
    B = node_off.shape[0] - 1
    V = strong_lp.shape[1] if V is None else int(V)
    dev = parent.device
    if out is None:
        out = (torch.empty(n_total, dtype=torch.float32, device=dev),
               torch.empty(n_total, dtype=torch.float32, device=dev),
               torch.empty(B, N, dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev))
    e, s, sel, nsel = out
    st = lib().treegraft_rescore_select(_ptr(weak_edge), _ptr(strong_lp), V, strong_lp.stride(0),
                                        _ptr(parent), _ptr(token), _ptr(visited), _ptr(node_off),
                                        B, int(max_nodes), n_total, int(N), _ptr(e), _ptr(s),
                                        _ptr(sel), _ptr(nsel), _stream(stream))
    _check("treegraft_rescore_select", st)
    return e, s, sel, nsel


def accept_workspace_size(B: int, n_total: int) -> int:
    return int(lib().treegraft_accept_workspace_size(B, n_total))


def accept_workspace(B: int, n_total: int, device) -> torch.Tensor:
    """A zero-filled workspace for accept (zeroed once; calls keep it ready)."""
    nbytes = accept_workspace_size(B, n_total)
    return torch.zeros(nbytes, dtype=torch.uint8, device=device)


def accept(target_logits, token, parent, node_off, max_nodes, path_cap, ws, *, V=None,
           out=None, stream=None):
    """Greedy longest-accepted-path walk.  Returns (path [B, path_cap],
    accept_len [B], bonus [B])."""
    if target_logits.dim() != 2 or target_logits.stride(1) != 1 or not target_logits.is_cuda:
        raise ValueError("target_logits must be a 2-D CUDA tensor with unit column stride")
    dt = _logit_dtype(target_logits)
    for t, nm in ((parent, "parent"), (token, "token"), (node_off, "node_off")):
        _need(t, torch.int32, nm)
    _need(ws, torch.uint8, "ws")
    n_total = parent.shape[0]
    B = node_off.shape[0] - 1
    V = target_logits.shape[1] if V is None else int(V)
    dev = parent.device
    if out is None:
        out = (torch.empty(B, path_cap, dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev))
    path, alen, bonus = out
    st = lib().treegraft_accept(_ptr(target_logits), dt, V, target_logits.stride(0), _ptr(token),
                                _ptr(parent), _ptr(node_off), B, int(max_nodes), n_total,
                                int(path_cap), _ptr(path), _ptr(alen), _ptr(bonus), _ptr(ws),
                                ws.numel(), _stream(stream))
    _check("treegraft_accept", st)
    return path, alen, bonus


def accept_sample_workspace(B: int, n_total: int, device) -> torch.Tensor:
    """A zero-filled workspace for accept_sample (zeroed once; calls keep it
    ready)."""
    nbytes = int(lib().treegraft_accept_sample_workspace_size(int(B), int(n_total)))
    if nbytes == 0:
        raise ValueError("accept_sample workspace: invalid sizes")
    return torch.zeros(nbytes, dtype=torch.uint8, device=device)


def accept_sample(target_logits, token, parent, node_off, max_nodes, path_cap, u, temperature,
                  ws, *, V=None, out=None, stream=None):
    """Stochastic verification at temperature > 0 with the caller's uniforms
    u fp32 [n_total, 2].  Returns (path [B, path_cap], accept_len [B],
    bonus [B])."""
    if target_logits.dim() != 2 or target_logits.stride(1) != 1 or not target_logits.is_cuda:
        raise ValueError("target_logits must be a 2-D CUDA tensor with unit column stride")
    dt = _logit_dtype(target_logits)
    for t, nm in ((parent, "parent"), (token, "token"), (node_off, "node_off")):
        _need(t, torch.int32, nm)
    _need(u, torch.float32, "u")
    _need(ws, torch.uint8, "ws")
    n_total = parent.shape[0]
    if tuple(u.shape) != (n_total, 2):
        raise ValueError("u must be [n_total, 2]")
    B = node_off.shape[0] - 1
    V = target_logits.shape[1] if V is None else int(V)
    dev = parent.device
    if out is None:
        out = (torch.empty(B, path_cap, dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev))
    path, alen, bonus = out
    st = lib().treegraft_accept_sample(_ptr(target_logits), dt, V, target_logits.stride(0),
                                       float(temperature), _ptr(token), _ptr(parent),
                                       _ptr(node_off), B, int(max_nodes), n_total, _ptr(u),
                                       int(path_cap), _ptr(path), _ptr(alen), _ptr(bonus),
                                       _ptr(ws), ws.numel(), _stream(stream))
    _check("treegraft_accept_sample", st)
    return path, alen, bonus


def accept_noalloc(target_logits, token, parent, node_off, max_nodes, path_cap, *, V=None,
                   out=None, stream=None):
    """accept() without a workspace, for callers that cannot allocate device
    memory: the library keeps the scratch in a fixed per-device array
    (n_total <= 65536, B <= 4096).  Calls that overlap on the GPU race."""
    if target_logits.dim() != 2 or target_logits.stride(1) != 1 or not target_logits.is_cuda:
        raise ValueError("target_logits must be a 2-D CUDA tensor with unit column stride")
    dt = _logit_dtype(target_logits)
    for t, nm in ((parent, "parent"), (token, "token"), (node_off, "node_off")):
        _need(t, torch.int32, nm)
    n_total = parent.shape[0]
    B = node_off.shape[0] - 1
    V = target_logits.shape[1] if V is None else int(V)
    if out is None:
        raise ValueError("accept_noalloc writes into caller-provided outputs: pass out=")
    path, alen, bonus = out
    st = lib().treegraft_accept_noalloc(_ptr(target_logits), dt, V, target_logits.stride(0),
                                        _ptr(token), _ptr(parent), _ptr(node_off), B,
                                        int(max_nodes), n_total, int(path_cap), _ptr(path),
                                        _ptr(alen), _ptr(bonus), _stream(stream))
    _check("treegraft_accept_noalloc", st)
    return path, alen, bonus


def graft_expand(logits, selected, k, cap, n, parent, token, edge, score, *, V=None,
                 stream=None):
    """Expand the reselected grafting positions (selected [B, N] int32, local
    node ids) by their top-k tokens from the drafter's rows (logits row
    b * cap + v) and append the children to the capacity-layout tree arrays
    parent / token / edge / score [B * cap] at rows b * cap + n + i * k + j.
    In place; returns (parent, token, edge, score)."""
    _need(selected, torch.int32, "selected")
    for t, nm, dt in ((parent, "parent", torch.int32), (token, "token", torch.int32),
                      (edge, "edge", torch.float32), (score, "score", torch.float32)):
        _need(t, dt, nm)
    if logits.dim() != 2:
        raise ValueError("logits must be [rows, ld]")
    if not logits.is_cuda or logits.stride(1) != 1:
        raise ValueError("logits must be a CUDA tensor with unit element stride")
    B, N = selected.shape
    if parent.numel() < B * cap:
        raise ValueError("tree arrays hold fewer than B * cap nodes")
    V = logits.shape[1] if V is None else int(V)
    st = lib().treegraft_graft_expand(_ptr(logits), _logit_dtype(logits), logits.shape[0], V,
                                      logits.stride(0), B, N, _ptr(selected), int(k), int(cap),
                                      int(n), _ptr(parent), _ptr(token), _ptr(edge), _ptr(score),
                                      _stream(stream))
    _check("treegraft_graft_expand", st)
    return parent, token, edge, score


def set_wait_budget(cycles: int) -> None:
    """Bound (SM cycles) of the waits a kernel makes on other thread blocks
    (the split barrier of tree_attn); 0 restores the default."""
    _check("treegraft_set_wait_budget", lib().treegraft_set_wait_budget(int(cycles)))


def last_device_status(stream=None) -> int:
    """Synchronise the stream; return and clear the device status bits."""
    return int(lib().treegraft_last_device_status(_stream(stream)))


def global_prune(score, parent, node_off, max_nodes, budget, path_cap, *, out=None, stream=None):
    """GlobalPrune of each tree to budget + 1 nodes with its verification
    buffers (Algorithm 3).  score fp32 [n_total], parent / node_off int32.
    Returns (kept, n_kept, new_parent, position, mask, paths, n_paths) with
    Mo = min(budget + 1, max_nodes) rows per tree; mask holds the uint32 bit
    words as int32 [B, Mo, ceil(Mo / 32)]."""
    _need(score, torch.float32, "score")
    _need(parent, torch.int32, "parent")
    _need(node_off, torch.int32, "node_off")
    n_total = parent.shape[0]
    B = node_off.shape[0] - 1
    Mo = min(int(budget) + 1, int(max_nodes))
    W = (Mo + 31) // 32
    dev = parent.device
    if out is None:
        out = (torch.empty(B, Mo, dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev),
               torch.empty(B, Mo, dtype=torch.int32, device=dev),
               torch.empty(B, Mo, dtype=torch.int32, device=dev),
               torch.empty(B, Mo, W, dtype=torch.int32, device=dev),
               torch.empty(B, Mo, int(path_cap), dtype=torch.int32, device=dev),
               torch.empty(B, dtype=torch.int32, device=dev))
    kept, n_kept, new_parent, position, mask, paths, n_paths = out
    st = lib().treegraft_global_prune(_ptr(score), _ptr(parent), _ptr(node_off), B, int(max_nodes),
                                      n_total, int(budget), int(path_cap), _ptr(kept),
                                      _ptr(n_kept), _ptr(new_parent), _ptr(position), _ptr(mask),
                                      _ptr(paths), _ptr(n_paths), _stream(stream))
    _check("treegraft_global_prune", st)
    return kept, n_kept, new_parent, position, mask, paths, n_paths


def grow_workspace(B, cap, m, device):
    """Scratch for grow_step on B trees of capacity cap with m children per
    frontier node (uint8 tensor)."""
    nbytes = int(lib().treegraft_grow_workspace_size(int(B), int(cap), int(m)))
    if nbytes == 0:
        raise ValueError("grow workspace: unsupported sizes")
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def grow_step(mode, logits, W, m, parent, token, edge, score, n, pool_lo, *, lse_mid=None,
              frontier=None, ws=None, V=None, stream=None):
    """One drafting step of the shared tree (Algorithm 2; mode 0 = small
    drafter, 1 = middle drafter) on B trees of capacity cap: parent / token
    int32 and edge / score fp32 [B, cap] (updated in place), lse_mid fp32
    [B, cap], logits [B * cap, ld] bf16/fp32 (row b * cap + v follows node v
    of tree b).  n and pool_lo are the host-side sizes of the step (see
    treegraft_grow_step).  Returns the frontier int32 [B, W]."""
    for t, nm in ((parent, "parent"), (token, "token")):
        _need(t, torch.int32, nm)
    for t, nm in ((edge, "edge"), (score, "score")):
        _need(t, torch.float32, nm)
    if lse_mid is not None:
        _need(lse_mid, torch.float32, "lse_mid")
    if parent.dim() != 2:
        raise ValueError("tree arrays must be [B, cap]")
    B, cap = parent.shape
    if logits.dim() != 2 or logits.stride(1) != 1 or not logits.is_cuda:
        raise ValueError("logits must be a 2-D CUDA tensor with unit column stride")
    dt = _logit_dtype(logits)
    V = logits.shape[1] if V is None else int(V)
    dev = parent.device
    if frontier is None:
        frontier = torch.empty(B, int(W), dtype=torch.int32, device=dev)
    _need(frontier, torch.int32, "frontier")
    if ws is None:
        ws = grow_workspace(B, cap, m, dev)
    st = lib().treegraft_grow_step(int(mode), _ptr(logits), dt, V, logits.stride(0), B, cap, int(n),
                                   int(pool_lo), int(W), int(m), _ptr(parent), _ptr(token),
                                   _ptr(edge), _ptr(score), _ptr(lse_mid), _ptr(frontier), _ptr(ws),
                                   ws.numel(), _stream(stream))
    _check("treegraft_grow_step", st)
    return frontier


class NgramIndex:
    """The n-gram small drafter's prompt index (a device buffer built by
    ngram_build) with the shape it was built for."""

    def __init__(self, buf, B, n_tokens, max_n):
        self.buf, self.B, self.n_tokens, self.max_n = buf, int(B), int(n_tokens), int(max_n)


def ngram_index_bytes(B, n_tokens, max_n) -> int:
    return int(lib().treegraft_ngram_index_bytes(int(B), int(n_tokens), int(max_n)))


def ngram_build(tokens, seq_off, max_n, *, index=None, stream=None):
    """Build the n-gram index over packed prompts: tokens int32 [n_tokens],
    seq_off int32 [B + 1] (prompt b = tokens[seq_off[b]:seq_off[b + 1]])."""
    _need(tokens, torch.int32, "tokens")
    _need(seq_off, torch.int32, "seq_off")
    B, n_tokens = seq_off.numel() - 1, tokens.numel()
    nbytes = ngram_index_bytes(B, n_tokens, max_n)
    if nbytes == 0:
        raise ValueError("ngram index: unsupported sizes")
    buf = index.buf if index is not None else torch.empty(nbytes, dtype=torch.uint8,
                                                          device=tokens.device)
    st = lib().treegraft_ngram_build(_ptr(tokens), _ptr(seq_off), B, n_tokens, int(max_n),
                                     _ptr(buf), buf.numel(), _stream(stream))
    _check("treegraft_ngram_build", st)
    return NgramIndex(buf, B, n_tokens, max_n)


def ngram_cache(logits, m_cache, *, cache_tok=None, cache_lp=None, V=None, stream=None):
    """Prefill cache: the top-m_cache tokens (int32) and log-probabilities
    (fp32) of every row of the prefill logits [n_tokens, ld]."""
    if logits.dim() != 2 or logits.stride(1) != 1 or not logits.is_cuda:
        raise ValueError("logits must be a 2-D CUDA tensor with unit column stride")
    rows = logits.shape[0]
    V = logits.shape[1] if V is None else int(V)
    if cache_tok is None:
        cache_tok = torch.empty(rows, int(m_cache), dtype=torch.int32, device=logits.device)
    if cache_lp is None:
        cache_lp = torch.empty(rows, int(m_cache), dtype=torch.float32, device=logits.device)
    _need(cache_tok, torch.int32, "cache_tok")
    _need(cache_lp, torch.float32, "cache_lp")
    st = lib().treegraft_ngram_cache(_ptr(logits), _logit_dtype(logits), rows, V, logits.stride(0),
                                     int(m_cache), _ptr(cache_tok), _ptr(cache_lp), _stream(stream))
    _check("treegraft_ngram_cache", st)
    return cache_tok, cache_lp


def _ngram_common(index, cache_tok, cache_lp, ctx, ctx_len):
    _need(cache_tok, torch.int32, "cache_tok")
    _need(cache_lp, torch.float32, "cache_lp")
    _need(ctx, torch.int32, "ctx")
    _need(ctx_len, torch.int32, "ctx_len")
    if (cache_tok.dim() != 2 or cache_tok.shape != cache_lp.shape
            or cache_tok.shape[0] != index.n_tokens):
        raise ValueError("cache_tok / cache_lp must be [n_tokens, m_cache]")
    if tuple(ctx.shape) != (index.B, index.max_n):
        raise ValueError("ctx must be [B, max_n]")
    return (_ptr(index.buf), index.buf.numel(), index.B, index.n_tokens, index.max_n,
            _ptr(cache_tok), _ptr(cache_lp), cache_tok.shape[1], _ptr(ctx), _ptr(ctx_len))


def ngram_draft(index, cache_tok, cache_lp, ctx, ctx_len, parent, token, rows, parent_score, m,
                *, with_match=False, stream=None):
    """The n-gram drafter's expansion of tree nodes rows int32 [R] (= b * cap
    + v) on trees parent / token int32 [B, cap]: tok int32, logprob, score
    fp32 [R, m] (and the matched prompt position and order if with_match)."""
    for t, nm in ((parent, "parent"), (token, "token"), (rows, "rows")):
        _need(t, torch.int32, nm)
    _need(parent_score, torch.float32, "parent_score")
    if parent.dim() != 2:
        raise ValueError("tree arrays must be [B, cap]")
    R, dev = rows.numel(), rows.device
    tok = torch.empty(R, int(m), dtype=torch.int32, device=dev)
    lp = torch.empty(R, int(m), dtype=torch.float32, device=dev)
    sc = torch.empty(R, int(m), dtype=torch.float32, device=dev)
    pos = torch.empty(R, dtype=torch.int32, device=dev) if with_match else None
    nn = torch.empty(R, dtype=torch.int32, device=dev) if with_match else None
    st = lib().treegraft_ngram_draft(*_ngram_common(index, cache_tok, cache_lp, ctx, ctx_len),
                                     _ptr(parent), _ptr(token), parent.shape[1], _ptr(rows), R,
                                     _ptr(parent_score), int(m), _ptr(tok), _ptr(lp), _ptr(sc),
                                     _ptr(pos), _ptr(nn), _stream(stream))
    _check("treegraft_ngram_draft", st)
    return (tok, lp, sc, pos, nn) if with_match else (tok, lp, sc)


def ngram_grow_step(index, cache_tok, cache_lp, ctx, ctx_len, W, m, parent, token, edge, score, n,
                    pool_lo, *, frontier=None, stream=None):
    """One small-drafter step of Algorithm 2 with the n-gram drafter on trees
    parent / token int32, edge / score fp32 [B, cap] (updated in place).
    Returns the frontier int32 [B, W]."""
    for t, nm in ((parent, "parent"), (token, "token")):
        _need(t, torch.int32, nm)
    for t, nm in ((edge, "edge"), (score, "score")):
        _need(t, torch.float32, nm)
    if parent.dim() != 2:
        raise ValueError("tree arrays must be [B, cap]")
    B, cap = parent.shape
    if frontier is None:
        frontier = torch.empty(B, int(W), dtype=torch.int32, device=parent.device)
    _need(frontier, torch.int32, "frontier")
    st = lib().treegraft_ngram_grow_step(*_ngram_common(index, cache_tok, cache_lp, ctx, ctx_len),
                                         cap, int(n), int(pool_lo), int(W), int(m), _ptr(parent),
                                         _ptr(token), _ptr(edge), _ptr(score), _ptr(frontier),
                                         _stream(stream))
    _check("treegraft_ngram_grow_step", st)
    return frontier
