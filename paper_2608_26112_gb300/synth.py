"""Seeded synthetic inputs for the draft-tree verify-and-grow step.

This module only draws random numbers and lays them out; it holds none of the
step's arithmetic (no masks, softmax, top-k, path sums or acceptance).  Both
the CUDA path (through tests and the benchmark) and the CPU oracle (through
tests) are fed from it, so neither side ever produces the other's inputs.

Shapes follow the workloads of the paper's setting: Llama-3 vocabulary 128256,
GQA 32/8 and 64/8 with head_dim 128, a verification tree of B_ver + 1 = 64
nodes (Sec. 5 setup, Appendix E: D=5, W=m=10, B_ver=63), trees grown by top-m
expansion (Algorithm 1).  The paper's benchmarks and checkpoints are replaced
by random draws with these shapes.

Conventions shared by every array produced here:
  * trees are given by ``parent`` (int32, root = local node 0 with parent -1,
    parent[i] < i, nodes numbered level by level) and ``token`` (int32);
    batched trees are concatenated and ``node_off`` (int32, B+1) gives each
    tree's node range;
  * bf16 tensors are returned as their raw uint16 bit patterns, rounded to
    nearest-even from float32 draws;
  * K/V caches are [B, Hkv, S_max, D]; slots [0, P_b) hold the committed
    prefix and slots [P_b, P_b + n_b) hold the tree's nodes in node order.
"""
from __future__ import annotations

import json
import math
import os

import numpy as np

LLAMA3_VOCAB = 128256


def make_rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest-even) and return the uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    bias = 0x7FFF + ((u >> 16) & 1)
    return ((u + bias) >> 16).astype(np.uint16)


# --------------------------------------------------------------------------
# tree shapes
# --------------------------------------------------------------------------

def _level_sizes(rng, n_nonroot: int, depth: int, cap: int | None) -> list[int]:
    """Random composition of n_nonroot into `depth` positive level sizes.

    With a per-parent child cap, level d may hold at most cap * |level d-1|
    nodes; compositions violating that are redrawn.
    """
    if depth < 1 or n_nonroot < depth:
        raise ValueError("need at least one node per level")
    for _ in range(100000):
        cuts = np.sort(rng.choice(n_nonroot - 1, size=depth - 1, replace=False)) + 1
        sizes = np.diff(np.concatenate([[0], cuts, [n_nonroot]])).tolist()
        if cap is None:
            return sizes
        prev, ok = 1, True
        for s in sizes:
            if s > cap * prev:
                ok = False
                break
            prev = s
        if ok:
            return sizes
    raise RuntimeError("could not draw level sizes under the child cap")


def sample_tree(rng, n: int, depth: int, cap: int | None = None,
                rank_bias: float = 0.0) -> np.ndarray:
    """Parent array of a random tree with n nodes and exactly `depth` levels
    below the root.

    Each node of level d picks a parent among the nodes of level d-1.  With
    rank_bias = 0 the pick is uniform (the tiny workload); with rank_bias > 0
    earlier nodes of the previous level are preferred, which gives the
    top-heavy shape of trees grown by top-m expansion, and `cap` bounds the
    children per parent (m).  Nodes are renumbered so that each level lists
    its nodes grouped by parent, parents in order.
    """
    if n == 1:
        return np.array([-1], dtype=np.int32)
    sizes = _level_sizes(rng, n - 1, depth, cap)
    parent = [-1]
    prev_ids = [0]
    next_id = 1
    for s in sizes:
        counts = np.zeros(len(prev_ids), dtype=np.int64)
        w = np.exp(-rank_bias * np.arange(len(prev_ids)))
        picks = []
        for _ in range(s):
            free = np.ones(len(prev_ids), bool) if cap is None else counts < cap
            p = w * free
            j = int(rng.choice(len(prev_ids), p=p / p.sum()))
            counts[j] += 1
            picks.append(j)
        picks.sort()
        ids = []
        for j in picks:
            parent.append(prev_ids[j])
            ids.append(next_id)
            next_id += 1
        prev_ids = ids
    return np.asarray(parent, dtype=np.int32)


def expansion_tree(rng, D: int, W: int, m: int) -> np.ndarray:
    """Parent array with the shape of a tree grown by D expansion steps of
    frontier W and branching m (Algorithm 1's shape before pruning): the
    root gets m children; at every later step W nodes of the newest level
    (drawn at random here) get m children each.  Ids run level by level,
    children grouped by parent, so parent[i] < i."""
    parent = [-1]
    level = [0]
    for k in range(D):
        front = level if k == 0 else sorted(rng.choice(level, size=min(W, len(level)), replace=False).tolist())
        nxt = []
        for v in front:
            for _ in range(m):
                parent.append(int(v))
                nxt.append(len(parent) - 1)
        level = nxt
    return np.asarray(parent, dtype=np.int32)


def path_scores(rng, parent: np.ndarray, step: float = 0.5, levels: int = 4) -> np.ndarray:
    """fp32 scores that never increase from a node to its children, as
    sums of log-probabilities along a path are: s(root) = 0 and
    s(v) = s(parent) - step * j with j uniform in {0, .., levels - 1}
    (zero steps give exact ties between a node and its child)."""
    s = np.zeros(len(parent), dtype=np.float64)
    drop = rng.integers(0, levels, size=len(parent)) * step
    for v in range(1, len(parent)):
        s[v] = s[parent[v]] - drop[v]
    return s.astype(np.float32)


def sample_tokens(rng, n: int, V: int) -> np.ndarray:
    return rng.integers(0, V, size=n, dtype=np.int64).astype(np.int32)


def children_lists(parent: np.ndarray) -> list[list[int]]:
    ch = [[] for _ in range(len(parent))]
    for v in range(1, len(parent)):
        ch[int(parent[v])].append(v)
    return ch


# --------------------------------------------------------------------------
# dense inputs
# --------------------------------------------------------------------------

def normal_f32(rng, shape, sigma: float = 1.0, mean: float = 0.0) -> np.ndarray:
    return (rng.standard_normal(size=shape, dtype=np.float32) * np.float32(sigma)
            + np.float32(mean))


def plant_child_bump(rng, logits: np.ndarray, parent: np.ndarray, token: np.ndarray,
                     row_of_node: np.ndarray, prob: float = 0.7,
                     bump: float = 8.0) -> None:
    """For each node with at least one child, with probability `prob` pick one
    child uniformly and add `bump` to that node's logit of the child's token
    (in place, float32 logits [rows, V])."""
    for v, ch in enumerate(children_lists(parent)):
        if ch and rng.random() < prob:
            c = ch[int(rng.integers(0, len(ch)))]
            logits[row_of_node[v], token[c]] += np.float32(bump)


# --------------------------------------------------------------------------
# prompts for the n-gram small drafter
# --------------------------------------------------------------------------

def prompt_stream(rng, L: int, V: int, *, copy_prob: float = 0.1, seg: tuple = (2, 12),
                  zipf_a: float = 1.1, active: int = 4096) -> np.ndarray:
    """A synthetic prompt of L tokens (int32) with the reuse that makes an
    n-gram drafter useful: each new piece is, with probability copy_prob, a
    copy of an earlier segment of length uniform in [seg[0], seg[1]],
    otherwise one token drawn from a Zipf(zipf_a) law over `active` tokens
    of a random permutation of the vocabulary."""
    active = min(active, V)
    vocab = rng.permutation(V)[:active]
    w = 1.0 / np.arange(1, active + 1) ** zipf_a
    draws = vocab[rng.choice(active, size=L, p=w / w.sum())]
    out = np.empty(L, np.int64)
    i = 0
    while i < L:
        if i >= seg[0] and rng.random() < copy_prob:
            ln = int(rng.integers(seg[0], seg[1] + 1))
            st = int(rng.integers(0, i - seg[0] + 1))
            ln = min(ln, L - i, i - st)
            out[i:i + ln] = out[st:st + ln]
            i += ln
        else:
            out[i] = draws[i]
            i += 1
    return out.astype(np.int32)


def plant_next_token_bump(rng, logits: np.ndarray, prompt: np.ndarray, prob: float = 0.7,
                          bump: float = 8.0) -> None:
    """Prefill logits that often predict the text: for each position j but
    the last, with probability `prob` add `bump` to row j's logit of the
    prompt's next token prompt[j + 1] (in place, float32 [L, V])."""
    for j in range(len(prompt) - 1):
        if rng.random() < prob:
            logits[j, prompt[j + 1]] += np.float32(bump)


def kv_cache(rng, B: int, Hkv: int, S_max: int, D: int, valid: list[int],
             tail: str = "zero") -> np.ndarray:
    """bf16 bits [B, Hkv, S_max, D] drawn N(0,1) over the valid slots of each
    sequence.  Slots past valid[b] hold zeros, or NaN bit patterns when
    tail == 'nan' (to check that a kernel never lets them reach the output)."""
    out = np.zeros((B, Hkv, S_max, D), dtype=np.uint16)
    for b in range(B):
        L = valid[b]
        out[b, :, :L] = f32_to_bf16_bits(normal_f32(rng, (Hkv, L, D)))
        if tail == "nan":
            out[b, :, L:] = 0x7FC0
    return out


# --------------------------------------------------------------------------
# workloads
# --------------------------------------------------------------------------

WORKLOADS = {
    # name: shape parameters (the synthetic stand-ins described in the module doc)
    "tiny": dict(B=1, P=128, n=16, depth=4, cap=None, rank_bias=0.0, Hq=8, Hkv=8,
                 D=64, V=1024, logit_dtype="f32", k=4, N=8),
    # the tree is one of the stored trees grown by Algorithm 1 + GlobalPrune
    # (tests/golden/llama3_8b_grown_trees.json), chosen by the seed
    "llama3-8b-verify": dict(B=1, P=2048, n=60, depth=6, cap=10, rank_bias=0.35, Hq=32,
                             Hkv=8, D=128, V=LLAMA3_VOCAB, logit_dtype="bf16", k=10, N=10,
                             tree="grown"),
    "graft-mha": dict(B=1, P=1024, n=64, depth=7, cap=8, rank_bias=0.35, Hq=32, Hkv=32,
                      D=128, V=32000, logit_dtype="f32", k=8, N=16),
    "llama3-70b-verify": dict(B=4, P=8192, n=128, depth=8, cap=16, rank_bias=0.25, Hq=64,
                              Hkv=8, D=128, V=LLAMA3_VOCAB, logit_dtype="bf16", k=16, N=16),
}


def serving_shape(B: int, seed: int) -> dict:
    """Ragged serving point: prefixes log-uniform in [512, 32768], tree sizes
    uniform in [32, 256], depths uniform in [4, 10]; GQA 32/8, head_dim 128."""
    rng = make_rng(1000 + B + 7919 * seed)
    P = np.exp(rng.uniform(math.log(512), math.log(32768), size=B)).astype(np.int64)
    n = rng.integers(32, 257, size=B)
    depth = rng.integers(4, 11, size=B)
    return dict(B=B, P=P.tolist(), n=n.tolist(), depth=depth.tolist(), cap=10,
                rank_bias=0.3, Hq=32, Hkv=8, D=128, V=LLAMA3_VOCAB, logit_dtype="bf16",
                k=10, N=10)


def _as_list(x, B):
    return list(x) if isinstance(x, (list, tuple)) else [x] * B


GROWN_TREES = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "tests",
                           "golden", "llama3_8b_grown_trees.json")
_grown_cache: list = []


def grown_trees() -> list:
    """The stored draft trees of the Llama-3-8B-shaped verify workload: each
    grown by Algorithm 1 (6 top-10 expansion steps by cumulative
    log-probability) and pruned to 60 nodes by GlobalPrune, written by
    tests/golden/make_grown_trees.py.  Loaded, not computed, here."""
    if not _grown_cache:
        with open(GROWN_TREES) as f:
            _grown_cache.extend(json.load(f)["trees"])
    return _grown_cache


def make_trees(rng, shape: dict, seed: int = 0):
    """Concatenated trees of a workload: (parent, token, node_off).  With
    shape["tree"] == "grown", tree b is stored tree (seed + b) mod count."""
    B = shape["B"]
    ns = _as_list(shape["n"], B)
    depths = _as_list(shape["depth"], B)
    parents, tokens, off = [], [], [0]
    for b in range(B):
        if shape.get("tree") == "grown":
            t = grown_trees()[(seed + b) % len(grown_trees())]
            p, tk = np.asarray(t["parent"], np.int32), np.asarray(t["token"], np.int32)
            if len(p) != ns[b]:
                raise ValueError("stored grown tree has the wrong size")
            parents.append(p)
            tokens.append(tk)
            off.append(off[-1] + ns[b])
            continue
        p = sample_tree(rng, ns[b], depths[b], shape.get("cap"), shape.get("rank_bias", 0.0))
        parents.append(p)
        tokens.append(sample_tokens(rng, ns[b], shape["V"]))
        off.append(off[-1] + ns[b])
    return (np.concatenate(parents).astype(np.int32), np.concatenate(tokens).astype(np.int32),
            np.asarray(off, dtype=np.int32))


def make_workload(name_or_shape, seed: int = 0, *, kv_tail: str = "zero",
                  with_logits: bool = True, with_strong: bool = True,
                  S_max: int | None = None, kv_trees: list[int] | None = None) -> dict:
    """All inputs of one verify-and-grow step for a named workload (or a
    shape dict), drawn from PCG64(seed).

    Returns a dict with
      shape, parent, token, node_off, prefix_len (int32 [B]), S_max,
      q (bf16 bits [n_total, Hq, D]), k_cache / v_cache (bf16 bits),
      logits ([n_total, V], float32 or bf16 bits; N(0, 3^2) plus the planted
        child bump with probability 0.7) used as the per-node next-token
        distributions (drafter rows for expansion, target rows for accept),
      parent_score (float32 [n_total], a path log-prob stand-in per row),
      weak_edge (float32 [n_total]) and strong_lp (float32 [n_total, V]):
        stored edge log-probs and a stronger drafter's log-probs, drawn
        log-prob shaped (mean -ln V - 4.5, sd 3, capped at 0),
      visited (uint8 [n_total]): nodes of depth <= 2 marked visited.
    With kv_trees, K/V are drawn only for those trees and k_cache / v_cache
    hold just their rows ([len(kv_trees), Hkv, S_max, D]); every other tree's
    K/V is all zeros (large serving batches stay cheap to build).
    """
    shape = dict(WORKLOADS[name_or_shape]) if isinstance(name_or_shape, str) else dict(name_or_shape)
    rng = make_rng(seed)
    B = shape["B"]
    parent, token, node_off = make_trees(rng, shape, seed)
    n_total = int(node_off[-1])
    Ps = _as_list(shape["P"], B)
    ns = [int(node_off[b + 1] - node_off[b]) for b in range(B)]
    valid = [Ps[b] + ns[b] for b in range(B)]
    if S_max is None:
        S_max = max(valid)
    Hq, Hkv, D, V = shape["Hq"], shape["Hkv"], shape["D"], shape["V"]
    out = dict(shape=shape, parent=parent, token=token, node_off=node_off,
               prefix_len=np.asarray(Ps, dtype=np.int32), S_max=S_max)
    out["q"] = f32_to_bf16_bits(normal_f32(rng, (n_total, Hq, D)))
    if kv_trees is None:
        out["k_cache"] = kv_cache(rng, B, Hkv, S_max, D, valid, kv_tail)
        out["v_cache"] = kv_cache(rng, B, Hkv, S_max, D, valid, kv_tail)
    else:
        sel = [valid[b] for b in kv_trees]
        out["kv_trees"] = list(kv_trees)
        out["k_cache"] = kv_cache(rng, len(sel), Hkv, S_max, D, sel, kv_tail)
        out["v_cache"] = kv_cache(rng, len(sel), Hkv, S_max, D, sel, kv_tail)
    # depth <= 2 nodes are marked visited (older nodes of a shared tree)
    vis = np.zeros(n_total, dtype=np.uint8)
    for b in range(B):
        o = node_off[b]
        d = np.zeros(ns[b], dtype=np.int64)
        for v in range(1, ns[b]):
            d[v] = d[parent[o + v]] + 1
        vis[o:o + ns[b]] = (d <= 2).astype(np.uint8)
    out["visited"] = vis
    out["parent_score"] = -np.abs(normal_f32(rng, (n_total,), 4.0))
    out["weak_edge"] = np.minimum(normal_f32(rng, (n_total,), 3.0, -math.log(V) - 4.5), 0).astype(np.float32)
    if with_logits:
        lg = np.empty((n_total, V), dtype=np.float32)
        for r0 in range(0, n_total, 256):
            r1 = min(n_total, r0 + 256)
            lg[r0:r1] = normal_f32(rng, (r1 - r0, V), 3.0)
        for b in range(B):
            o = int(node_off[b])
            rows = np.arange(o, o + ns[b])
            plant_child_bump(rng, lg, parent[o:o + ns[b]], token[o:o + ns[b]], rows)
        out["logits"] = lg if shape["logit_dtype"] == "f32" else f32_to_bf16_bits(lg)
    if with_strong:
        st = np.empty((n_total, V), dtype=np.float32)
        for r0 in range(0, n_total, 256):
            r1 = min(n_total, r0 + 256)
            st[r0:r1] = np.minimum(normal_f32(rng, (r1 - r0, V), 3.0, -math.log(V) - 4.5), 0)
        out["strong_lp"] = st
    return out
