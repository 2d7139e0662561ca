"""The C-ABI library builds, loads and exports every entry point that
include/treegraft.h declares; host-side argument validation rejects bad
calls before anything reaches the GPU.  CPU only: no kernel is launched."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "treegraft.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(treegraft_\w+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_26112_gb300 import build
    build.build()
    from paper_2608_26112_gb300 import binding
    return binding.lib()


def test_header_declares_the_four_calls():
    fns = declared_functions()
    for name in ("treegraft_tree_attn", "treegraft_expand_topk", "treegraft_rescore_select",
                 "treegraft_accept"):
        assert name in fns


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    assert lib.treegraft_status_string(0) == b"ok"
    assert b"invalid" in lib.treegraft_status_string(1)


def test_tree_attn_workspace_size(lib):
    # The larger of the two kernels' needs.  Split kernel: two int counters per
    # (tree, kv-head, 128-row work item) padded to 256 bytes, then per (work item,
    # split) a slab of 128 rows x (D bf16 + 2 fp32), up to 10 splits.  Two-tile
    # kernel: one ticket per 128-row unit padded to 256 bytes, then 512 slabs of
    # 256 rows for the key chunks of long units (twice the 256 resident CTAs).
    def sizes(B, n, Hq, Hkv, D):
        units = B * Hkv * (((Hq // Hkv) * n + 127) // 128)
        split = (units * 8 + 255) // 256 * 256 + units * 10 * 128 * (2 * D + 8)
        whole = (units * 4 + 255) // 256 * 256 + 512 * 256 * (2 * D + 8)
        return max(split, whole)
    for args in ((1, 60, 32, 8, 128), (4, 128, 64, 8, 128), (64, 256, 32, 8, 128), (1, 16, 8, 8, 64)):
        assert lib.treegraft_tree_attn_workspace_size(*args) == sizes(*args), args
    assert lib.treegraft_tree_attn_workspace_size(1, 60, 32, 8, 96) == 0


def test_workspace_size(lib):
    assert lib.treegraft_accept_workspace_size(1, 60) >= 61 * 4
    assert lib.treegraft_accept_workspace_size(1, 60) % 256 == 0
    assert lib.treegraft_accept_workspace_size(0, 60) == 0


NULL = None


def test_tree_attn_rejects_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    # null pointer
    assert lib.treegraft_tree_attn(NULL, fake, fake, fake, fake, fake, 1, 16, 16, 8, 8, 64, 144,
                                   0.0, fake, NULL, NULL, 0, NULL) == 1
    # head_dim 96 unsupported, G = 3 unsupported, Hq % Hkv != 0 invalid
    assert lib.treegraft_tree_attn(fake, fake, fake, fake, fake, fake, 1, 16, 16, 8, 8, 96, 144,
                                   0.0, fake, NULL, NULL, 0, NULL) == 2
    assert lib.treegraft_tree_attn(fake, fake, fake, fake, fake, fake, 1, 16, 16, 12, 4, 64, 144,
                                   0.0, fake, NULL, NULL, 0, NULL) == 2
    assert lib.treegraft_tree_attn(fake, fake, fake, fake, fake, fake, 1, 16, 16, 8, 3, 64, 144,
                                   0.0, fake, NULL, NULL, 0, NULL) == 1
    # more than 256 nodes per tree
    assert lib.treegraft_tree_attn(fake, fake, fake, fake, fake, fake, 1, 300, 300, 8, 8, 64,
                                   400, 0.0, fake, NULL, NULL, 0, NULL) == 1
    # misaligned q
    assert lib.treegraft_tree_attn(ctypes.c_void_p(0x1002), fake, fake, fake, fake, fake, 1, 16,
                                   16, 8, 8, 64, 144, 0.0, fake, NULL, NULL, 0, NULL) == 1
    # negative scale
    assert lib.treegraft_tree_attn(fake, fake, fake, fake, fake, fake, 1, 16, 16, 8, 8, 64, 144,
                                   -1.0, fake, NULL, NULL, 0, NULL) == 1


def test_expand_topk_rejects_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    args = dict(logits=fake, dtype=0, logit_rows=4, V=100, ld=100, rows=4, row_idx=NULL,
                ps=fake, k=4)

    def call(**kw):
        a = dict(args, **kw)
        return lib.treegraft_expand_topk(a["logits"], a["dtype"], a["logit_rows"], a["V"],
                                         a["ld"], a["rows"], a["row_idx"], a["ps"], a["k"], fake,
                                         fake, fake, NULL, NULL)
    assert call(rows=0) == 0                 # empty call is a no-op
    assert call(logits=NULL) == 1
    assert call(k=101) == 1                  # k > V
    assert call(k=0) == 1
    assert call(k=33) == 2                   # beyond the top-k limit
    assert call(ld=50) == 1                  # ld < V
    assert call(dtype=7) == 1
    assert call(rows=5) == 1                 # more rows than logits, no row_idx
    assert call(V=300000, ld=300000) == 2


def test_rescore_and_accept_reject_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    assert lib.treegraft_rescore_select(fake, fake, 100, 100, fake, fake, fake, fake, 1, 64, 64,
                                        0, fake, fake, fake, fake, NULL) == 1      # N = 0
    assert lib.treegraft_rescore_select(fake, fake, 100, 100, fake, fake, fake, fake, 1, 300, 64,
                                        8, fake, fake, fake, fake, NULL) == 1      # max_nodes
    assert lib.treegraft_rescore_select(NULL, fake, 100, 100, fake, fake, fake, fake, 1, 64, 64,
                                        8, fake, fake, fake, fake, NULL) == 1
    ws = lib.treegraft_accept_workspace_size(1, 60)
    assert lib.treegraft_accept(fake, 0, 100, 100, fake, fake, fake, 1, 60, 60, 8, fake, fake,
                                fake, fake, ws - 1, NULL) == 1                     # ws too small
    assert lib.treegraft_accept(fake, 0, 100, 100, fake, fake, fake, 1, 60, 60, 0, fake, fake,
                                fake, fake, ws, NULL) == 1                         # path_cap 0
    assert lib.treegraft_accept(fake, 0, 100, 100, fake, fake, fake, 1, 60, 61, 8, fake, fake,
                                fake, fake, ws, NULL) == 1                         # n_total > B*max


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    from paper_2608_26112_gb300 import binding
    monkeypatch.setattr(binding, "_lib", None)
    monkeypatch.setattr(binding, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        binding.lib()


def test_global_prune_rejects_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)

    def call(B=1, max_nodes=100, n_total=100, budget=10, path_cap=8, score=fake):
        return lib.treegraft_global_prune(score, fake, fake, B, max_nodes, n_total, budget,
                                          path_cap, fake, fake, fake, fake, fake, fake, fake, NULL)
    assert call(score=NULL) == 1
    assert call(budget=0) == 1                   # empty verification budget
    assert call(budget=256) == 1                 # pruned tree beyond tree_attn's 256 nodes
    assert call(path_cap=0) == 1
    assert call(n_total=101) == 1                # more nodes than B * max_nodes
    assert call(max_nodes=2000, n_total=2000) == 2


def test_grow_step_rejects_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    ws_need = lib.treegraft_grow_workspace_size(2, 64, 4)
    assert ws_need > 0
    assert lib.treegraft_grow_workspace_size(2, 2000, 4) == 0      # beyond TG_MAX_GROW_NODES
    assert lib.treegraft_grow_workspace_size(2, 64, 33) == 0       # beyond TG_MAX_TOPK

    def call(mode=0, dtype=0, V=100, ld=100, B=2, cap=64, n=11, pool_lo=1, W=4, m=4,
             lse=fake, logits=fake, ws_bytes=None):
        return lib.treegraft_grow_step(mode, logits, dtype, V, ld, B, cap, n, pool_lo, W, m, fake,
                                       fake, fake, fake, lse, fake, fake,
                                       ws_need if ws_bytes is None else ws_bytes, NULL)
    assert call(logits=NULL) == 1
    assert call(mode=2) == 1
    assert call(mode=1, lse=NULL) == 1          # a middle step caches the log-sum-exp
    assert call(dtype=5) == 1
    assert call(ld=99) == 1
    assert call(n=0) == 1
    assert call(pool_lo=11) == 1                # empty candidate pool
    assert call(m=101) == 1                     # more children than tokens
    assert call(n=60) == 1                      # 60 + 4 * 4 children exceed the capacity
    assert call(ws_bytes=ws_need - 1) == 1
    assert call(cap=2000, n=11) == 2            # beyond TG_MAX_GROW_NODES
    assert call(m=33, V=100, cap=1024) == 2     # beyond TG_MAX_TOPK
    assert call(logits=ctypes.c_void_p(0x1001)) == 1  # misaligned bf16 elements


def test_ngram_rejects_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    need = lib.treegraft_ngram_index_bytes(2, 100, 4)
    # T = 256 slots per order (>= 2 * 100): tokens, offsets, 4 tables, counts, fallbacks
    assert need == 512 + 256 + 4 * 256 * 4 + 256 * 4 + 256 + 256
    assert lib.treegraft_ngram_index_bytes(2, 100, 9) == 0          # max_n > TG_NGRAM_MAX_N
    assert lib.treegraft_ngram_index_bytes(3, 2, 4) == 0            # an empty prompt
    assert lib.treegraft_ngram_index_bytes(1, (1 << 26) + 1, 4) == 0
    assert lib.treegraft_ngram_build(fake, fake, 2, 100, 4, fake, need - 1, NULL) == 1
    assert lib.treegraft_ngram_build(NULL, fake, 2, 100, 4, fake, need, NULL) == 1
    assert lib.treegraft_ngram_build(fake, fake, 2, 100, 9, fake, 1 << 20, NULL) == 1
    assert lib.treegraft_ngram_cache(fake, 0, 10, 100, 100, 33, fake, fake, NULL) == 2
    assert lib.treegraft_ngram_cache(fake, 0, 10, 100, 99, 4, fake, fake, NULL) == 1

    def draft(m=4, m_cache=8, nbytes=need, R=5, index=fake):
        return lib.treegraft_ngram_draft(index, nbytes, 2, 100, 4, fake, fake, m_cache, fake, fake,
                                         fake, fake, 16, fake, R, fake, m, fake, fake, fake, NULL,
                                         NULL, NULL)
    assert draft(R=0) == 0
    assert draft(m=9) == 1                   # m > m_cache
    assert draft(m_cache=33, m=4) == 2
    assert draft(nbytes=need - 256) == 1
    assert draft(index=NULL) == 1

    def grow(cap=64, n=5, pool_lo=1, W=4, m=4):
        return lib.treegraft_ngram_grow_step(fake, need, 2, 100, 4, fake, fake, 8, fake, fake, cap,
                                             n, pool_lo, W, m, fake, fake, fake, fake, fake, NULL)
    assert grow(cap=20) == 1                 # 5 + 4 * 4 children do not fit
    assert grow(pool_lo=5) == 1
    assert grow(cap=2048, n=5) == 2          # beyond TG_MAX_GROW_NODES


def test_accept_sample_rejects_bad_args_on_host(lib):
    fake = ctypes.c_void_p(0x1000)
    need = lib.treegraft_accept_sample_workspace_size(2, 100)
    assert need == 512 + 512 + 256          # flags, bonus candidates, tickets
    assert lib.treegraft_accept_sample_workspace_size(0, 100) == 0

    def call(T=1.0, u=fake, nbytes=need, V=100, max_nodes=64, B=2):
        return lib.treegraft_accept_sample(fake, 0, V, V, T, fake, fake, fake, B, max_nodes, 100,
                                           u, 8, fake, fake, fake, fake, nbytes, NULL)
    assert call(T=0.0) == 1
    assert call(T=-1.0) == 1
    assert call(T=float("inf")) == 1
    assert call(T=1e-39) == 2                     # log2(e) / T overflows fp32
    assert call(u=NULL) == 1
    assert call(nbytes=need - 1) == 1
    assert call(max_nodes=300) == 1
    assert call(V=300000) == 2
