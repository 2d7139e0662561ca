"""GB300 (sm_103a) kernels for the draft-tree verify-and-grow step of
TreeGraft (multi-drafter tree speculative decoding).

The compute lives in libtreegraft.so (C ABI, include/treegraft.h); this
package holds its build script, its Python binding and the seeded synthetic
input generator used by the tests and the benchmark.
"""
from .binding import (  # noqa: F401
    MAX_GROW_NODES, MAX_PRUNE_NODES, MAX_TOPK, MAX_TREE_NODES, NGRAM_MAX_N, NgramIndex,
    TreeGraftError, accept, accept_sample, accept_sample_workspace, accept_workspace,
    accept_workspace_size, expand_topk, global_prune, graft_expand,
    grow_step, grow_workspace, last_device_status, lib, ngram_build, ngram_cache, ngram_draft,
    ngram_grow_step, ngram_index_bytes, rescore_select, set_wait_budget, tree_attn,
    tree_attn_workspace_size)
