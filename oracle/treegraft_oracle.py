"""CPU oracle for TreeGraft's verify-and-grow step (test infrastructure only).

This is a plain, slow statement of what the step computes, written from the
paper's definitions in fp64 (attention, log-sum-exp) and fp32 (path-score
sums, whose summation order the definition fixes).  Only the test-suite, the
package smoke check and the benchmark's CPU-baseline leg may import it; the
product path never calls it.  It shares no code with the CUDA library: it
takes plain numpy arrays (bf16 tensors as their uint16 bit patterns) and
decodes them itself.

Every function is pinned against something other than itself by the
CPU-only tests in tests/test_oracle_pins.py (brute force, closed forms,
invariants).  Parity status per function:
  ancestor_mask, tree_attention, expand_topk, rescore_select, accept,
  global_prune, grow_state / grow_step / grow_tree: pinned (grow_tree is
  grow_step applied over a schedule; its pins exercise every branch of it).

Readings of the paper taken here (where it is silent or loose):
  * depth(root) = 0; mask row u has P + depth(u) + 1 ones (Algorithm 3 mask:
    root, ancestors, self; plus the whole committed prefix);
  * every tree node, the root included, has its K/V at cache slot P + node;
  * scale = D^-1/2, q-head h reads kv-head floor(h / G), G = Hq / Hkv;
  * edge scores are natural-log probabilities (Sec. 3.1 defines s(v) as a
    product of probabilities; the log of it is a sum), s(root) = 0;
  * top-k and Top_W rank by the input value, ties to the lower token / node
    id;
  * the stronger drafter rescores a non-root node v from the row of its
    parent: p(v) = q_m(token(v) | prefix ending at pa(v)) (Sec. 3.1, 3.2);
  * verification at temperature 0 is greedy matching against the target's
    argmax (lowest token on ties); the accepted node is the deepest fully
    matching node, ties to the lowest id; the bonus token is the argmax of
    the accepted node's own row;
  * GlobalPrune (Algorithm 3) re-indexes the kept nodes in their original
    order and lists retrieval paths by leaf in ascending new index.
"""
from __future__ import annotations

import numpy as np

NEG_INF = float("-inf")


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode raw bf16 bit patterns (uint16) exactly into float64."""
    b = np.ascontiguousarray(bits).view(np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def _tree_slices(node_off):
    node_off = np.asarray(node_off, dtype=np.int64)
    return [(int(node_off[b]), int(node_off[b + 1])) for b in range(len(node_off) - 1)]


def check_tree(parent: np.ndarray) -> None:
    """Raise if a tree's parent array is not in parents-before-children form
    (Algorithm 3 re-indexes the verification tree so that it is)."""
    parent = np.asarray(parent)
    if len(parent) == 0 or parent[0] != -1:
        raise ValueError("root must be node 0 with parent -1")
    for i in range(1, len(parent)):
        if not (0 <= parent[i] < i):
            raise ValueError(f"parent[{i}] = {parent[i]} is not an earlier node")


def node_depth(parent: np.ndarray) -> np.ndarray:
    """Depth of every node, root depth 0 (position id, Algorithm 3)."""
    check_tree(parent)
    d = np.zeros(len(parent), dtype=np.int64)
    for u in range(len(parent)):
        v, k = u, 0
        while parent[v] != -1:
            v = parent[v]
            k += 1
        d[u] = k
    return d


def ancestor_mask(parent: np.ndarray) -> np.ndarray:
    """Tree-attention mask of Algorithm 3: mask[u, v] is true iff v is the
    root, an ancestor of u, or u itself.  Computed by walking parent pointers
    from u up to the root."""
    check_tree(parent)
    n = len(parent)
    m = np.zeros((n, n), dtype=bool)
    for u in range(n):
        m[u, 0] = True
        v = u
        while v != -1:
            m[u, v] = True
            v = int(parent[v])
    return m


def tree_attention(q, k_cache, v_cache, prefix_len, parent, node_off, Hkv: int,
                   scale: float | None = None, *, bf16: bool = True):
    """Ancestor-masked GQA tree attention in fp64.

    For tree b, q-head h and node u the keys are the committed prefix
    [0, P_b) and the tree slots P_b + v of the nodes v allowed by the
    Algorithm-3 mask of u (root, ancestors, self); the tree is verified
    through tree attention (Sec. 3.1; Algorithm 1/2 verification step).

      s_j = scale * <q, k_j>,  o = sum_j softmax(s)_j v_j,  lse = log sum_j e^{s_j}

    q: [n_total, Hq, D]; k_cache, v_cache: [B, Hkv, S_max, D] (bf16 bits if
    bf16 else float arrays).  Returns (o float64 [n_total, Hq, D],
    lse float64 [n_total, Hq]).
    """
    if bf16:
        q, k_cache, v_cache = (bf16_bits_to_f64(x) for x in (q, k_cache, v_cache))
    else:
        q, k_cache, v_cache = (np.asarray(x, dtype=np.float64) for x in (q, k_cache, v_cache))
    n_total, Hq, D = q.shape
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    o = np.zeros((n_total, Hq, D))
    lse = np.zeros((n_total, Hq))
    for b, (a, e) in enumerate(_tree_slices(node_off)):
        n, P = e - a, int(prefix_len[b])
        allowed = np.concatenate([np.ones((n, P), bool), ancestor_mask(parent[a:e])], axis=1)
        for h in range(Hq):
            kv = h // G
            K = k_cache[b, kv, :P + n]
            Vv = v_cache[b, kv, :P + n]
            s = (q[a:e, h] @ K.T) * scale
            s[~allowed] = NEG_INF
            m = s.max(axis=1, keepdims=True)
            p = np.exp(s - m)
            l = p.sum(axis=1, keepdims=True)
            o[a:e, h] = (p @ Vv) / l
            lse[a:e, h] = (m + np.log(l))[:, 0]
    return o, lse


def _row_values(logits, r: int, bf16: bool) -> np.ndarray:
    row = logits[r]
    return bf16_bits_to_f64(row) if bf16 else np.asarray(row, dtype=np.float64)


def expand_topk(logits, parent_score, k: int, row_idx=None, *, bf16: bool = False):
    """Per-row log-softmax, top-k child tokens and cumulative path score.

    For each logical row i (physical row row_idx[i], or i):
      lse = log sum_t exp(l_t)                         (fp64)
      tok = the k tokens of largest l_t, ordered by (l desc, token asc)
      logprob = fp32(l_tok - lse)       edge score p(u) in log form (Alg. 1/2)
      score = fp32(parent_score + l_tok - lse)   s(u) = s(v) * p(u) in log form
    A row whose logits are all -inf has lse = -inf and logprob = score = -inf.
    Returns tok int32 [rows, k], logprob f32, score f32, lse f64 [rows].
    """
    rows = len(parent_score)
    tok = np.zeros((rows, k), dtype=np.int32)
    lp = np.zeros((rows, k), dtype=np.float32)
    sc = np.zeros((rows, k), dtype=np.float32)
    lse = np.zeros(rows)
    for i in range(rows):
        r = int(row_idx[i]) if row_idx is not None else i
        x = _row_values(logits, r, bf16)
        V = len(x)
        m = x.max()
        if m == NEG_INF:
            lse[i] = NEG_INF
        else:
            lse[i] = m + np.log(np.exp(x - m).sum())
        order = np.lexsort((np.arange(V), -x))[:k]
        tok[i] = order
        if lse[i] == NEG_INF:
            lp[i] = NEG_INF
            sc[i] = NEG_INF
        else:
            lp[i] = (x[order] - lse[i]).astype(np.float32)
            sc[i] = (float(np.float32(parent_score[i])) + (x[order] - lse[i])).astype(np.float32)
    return tok, lp, sc, lse


def rescore_select(weak_edge, strong_lp, parent, token, visited, node_off, N: int):
    """Stronger-drafter rescoring of the candidate pool and global top-N.

    Per tree (Sec. 3.2, Algorithm 2 middle-drafter step): the candidate pool
    is C = {v : not visited[v]} = V(T) \\ P_k.  For non-root v in C the edge
    score becomes the stronger drafter's log-prob of token(v) under the
    prefix ending at pa(v): strong_lp[pa(v), token(v)]; other nodes keep
    weak_edge[v].  Scores are recomputed as fp32 sums from the root,
    s(root) = 0, s(v) = fp32(s(pa(v)) + edge(v)) in node order.  The
    frontier is Top_N(C, s) ordered by (s desc, id asc).

    Returns edge f32 [n_total] (root entries 0), score f32 [n_total],
    selected int32 [B, N] (local node ids, -1 padded), n_selected int32 [B].
    """
    n_total = len(parent)
    edge = np.zeros(n_total, dtype=np.float32)
    score = np.zeros(n_total, dtype=np.float32)
    slices = _tree_slices(node_off)
    sel = np.full((len(slices), N), -1, dtype=np.int32)
    nsel = np.zeros(len(slices), dtype=np.int32)
    for b, (a, e) in enumerate(slices):
        check_tree(parent[a:e])
        for v in range(1, e - a):
            if visited[a + v]:
                edge[a + v] = np.float32(weak_edge[a + v])
            else:
                edge[a + v] = np.float32(strong_lp[a + int(parent[a + v]), int(token[a + v])])
        score[a] = np.float32(0.0)
        for v in range(1, e - a):
            score[a + v] = np.float32(score[a + int(parent[a + v])]) + np.float32(edge[a + v])
        cand = [v for v in range(e - a) if not visited[a + v]]
        cand.sort(key=lambda v: (-float(score[a + v]), v))
        take = cand[:N]
        sel[b, :len(take)] = take
        nsel[b] = len(take)
    return edge, score, sel, nsel


def target_argmax(target_logits, rows, *, bf16: bool = False) -> np.ndarray:
    """Greedy target token per row: argmax with the lowest token on ties."""
    return np.array([int(np.argmax(_row_values(target_logits, r, bf16))) for r in rows],
                    dtype=np.int64)


def accept(target_logits, token, parent, node_off, path_cap: int, *, bf16: bool = False):
    """Greedy longest-accepted-path walk at temperature 0 (Sec. 5 setting;
    the verification step of Algorithms 1 and 2).

    Brute force: enumerate every root-to-node path; a path is accepted when
    each of its non-root nodes' token equals the target argmax of its
    parent's row.  The accepted node a* is the deepest fully matching node,
    ties to the lowest id; A = depth(a*); the bonus token is the argmax of
    row a*.  Returns path int32 [B, path_cap] (root-first local ids, -1
    padded), accept_len int32 [B], bonus int32 [B].
    """
    slices = _tree_slices(node_off)
    path = np.full((len(slices), path_cap), -1, dtype=np.int32)
    alen = np.zeros(len(slices), dtype=np.int32)
    bonus = np.zeros(len(slices), dtype=np.int32)
    for b, (a, e) in enumerate(slices):
        par = parent[a:e]
        check_tree(par)
        am = target_argmax(target_logits, range(a, e), bf16=bf16)
        best = None
        for v in range(e - a):
            chain = [v]
            while par[chain[-1]] != -1:
                chain.append(int(par[chain[-1]]))
            chain.reverse()
            ok = all(int(token[a + w]) == am[int(par[w])] for w in chain[1:])
            if ok:
                key = (len(chain) - 1, -v)
                if best is None or key > best[0]:
                    best = (key, chain)
        chain = best[1]
        if len(chain) > path_cap:
            raise ValueError("accepted path longer than path_cap")
        path[b, :len(chain)] = chain
        alen[b] = len(chain) - 1
        bonus[b] = am[chain[-1]]
    return path, alen, bonus


def global_prune(parent, score, node_off, budget: int, path_cap: int):
    """Global score-based pruning with ancestor closure (Algorithm 3), per
    tree, with the verification buffers it returns.

    M = budget + 1 (the root is the extra node).  A tree with at most M
    nodes is returned unchanged.  Otherwise the non-root nodes are ranked by
    (-s(v), d(v), id(v)); starting from K = {root}, each ranked node's chain
    up to the first node already in K is added whole when |K| + |chain| <= M,
    and the loop stops once |K| = M.  The kept nodes are re-indexed in their
    original order (parents keep coming before children), the mask is the
    Algorithm 3 mask of the pruned tree, a node's position id is its depth,
    and the retrieval paths are the root-to-leaf paths of the pruned tree
    (leaves in ascending new index, root first, -1 padded to path_cap).
    Scores are log-domain path scores (larger is better) in fp32.

    Returns per tree b (arrays of stride Mo = min(M, max tree size)):
      kept int32 [B, Mo] (old local ids in new order, -1 padded),
      n_kept int32 [B], new_parent int32 [B, Mo] (-1 for the root and pad),
      position int32 [B, Mo] (-1 pad), mask bool [B, Mo, Mo],
      paths int32 [B, Mo, path_cap] (-1 padded), n_paths int32 [B].
    """
    slices = _tree_slices(node_off)
    M = budget + 1
    Mo = min(M, max(e - a for a, e in slices))
    B = len(slices)
    kept_o = np.full((B, Mo), -1, dtype=np.int32)
    n_kept = np.zeros(B, dtype=np.int32)
    par_o = np.full((B, Mo), -1, dtype=np.int32)
    pos_o = np.full((B, Mo), -1, dtype=np.int32)
    mask_o = np.zeros((B, Mo, Mo), dtype=bool)
    paths_o = np.full((B, Mo, path_cap), -1, dtype=np.int32)
    n_paths = np.zeros(B, dtype=np.int32)
    for b, (a, e) in enumerate(slices):
        par = [int(x) for x in parent[a:e]]
        s = [float(x) for x in np.asarray(score[a:e], dtype=np.float32)]
        check_tree(np.asarray(par))
        n = e - a
        d = node_depth(np.asarray(par))
        if n <= M:
            kept = list(range(n))
        else:
            ranked = sorted(range(1, n), key=lambda v: (-s[v], int(d[v]), v))
            K = {0}
            for v in ranked:
                chain = []
                w = v
                while w not in K:
                    chain.append(w)
                    w = par[w]
                if len(K) + len(chain) <= M:
                    K.update(chain)
                if len(K) == M:
                    break
            kept = sorted(K)
        new = {old: i for i, old in enumerate(kept)}
        new_par = [-1] + [new[par[v]] for v in kept[1:]]
        k = len(kept)
        n_kept[b] = k
        kept_o[b, :k] = kept
        par_o[b, :k] = new_par
        pos_o[b, :k] = [int(d[v]) for v in kept]
        mask_o[b, :k, :k] = ancestor_mask(np.asarray(new_par))
        has_child = set(new_par[1:])
        leaves = [i for i in range(k) if i not in has_child]
        for j, leaf in enumerate(leaves):
            chain = [leaf]
            while new_par[chain[-1]] != -1:
                chain.append(new_par[chain[-1]])
            chain.reverse()
            if len(chain) > path_cap:
                raise ValueError("retrieval path longer than path_cap")
            paths_o[b, j, :len(chain)] = chain
        n_paths[b] = len(leaves)
    return kept_o, n_kept, par_o, pos_o, mask_o, paths_o, n_paths


def _row_log_softmax(logits, r: int, bf16: bool):
    """(values, lse) of one logit row in fp64."""
    x = _row_values(logits, r, bf16)
    m = x.max()
    lse = NEG_INF if m == NEG_INF else m + np.log(np.exp(x - m).sum())
    return x, lse


def grow_state():
    """Initial shared tree of Algorithm 2: the root alone, N_1 = {r}, P_1 empty,
    s(r) = 0 (log of 1)."""
    return dict(parent=[-1], token=[0], edge=[np.float32(0.0)], score=[np.float32(0.0)],
                new=[0], P=set(), lse_m={})


def grow_step(state, a: int, W: int, m: int, small_logits, middle_logits, *, bf16: bool = False,
              small_draft=None):
    """One drafting step k of Algorithm 2 on `state` (see grow_state), in place.

    The drafters' next-token logits under the prefix ending at node v are
    rows v of small_logits and middle_logits (tables indexed by node id, the
    stand-in for the drafter forwards).  Scores are log-domain: s(u) =
    fp32(s(v) + p(u)) with p(u) = fp32(l_u - lse) the drafter's
    log-probability of u's token.  a = 0 (small drafter): C = N_k (the nodes
    made at the previous step), F = Top_W(C, s) by (s desc, id asc), and
    each v in F gets its m best small-drafter tokens (logit desc, token asc)
    as new children.  a = 1 (middle drafter): C = V(T) \\ P; the log-sum-exp
    of every row in C is taken (and cached: it is the forward pass over C);
    every non-root v in C is rescored, p(v) = fp32(l_m[pa(v), token(v)] -
    lse_m[pa(v)]), and s is recomputed in node order; F = Top_W(C, s); each
    v in F gets its m best middle-drafter tokens; then P = P u C.  Children
    are appended in frontier order, then child rank, never replacing an
    existing node.  Returns the frontier F.

    small_draft, if given, replaces the small drafter's table: a callable
    (state, v, m) -> (tokens, log-probabilities) giving v's m children (the
    training-free n-gram drafter of the Appendix; oracle/ngram_oracle.py).
    """
    parent, token, edge, score = state["parent"], state["token"], state["edge"], state["score"]
    P, lse_m = state["P"], state["lse_m"]
    n = len(parent)
    if a == 0:
        C = list(state["new"])
        table = small_logits
    else:
        C = [v for v in range(n) if v not in P]
        for v in C:
            lse_m[v] = _row_log_softmax(middle_logits, v, bf16)[1]
        for v in C:
            if v == 0:
                continue
            row = _row_values(middle_logits, parent[v], bf16)
            edge[v] = np.float32(row[token[v]] - lse_m[parent[v]])
            score[v] = np.float32(score[parent[v]] + edge[v])
        table = middle_logits
    F = sorted(C, key=lambda v: (-float(score[v]), v))[:W]
    made = []
    for v in F:
        if a == 0 and small_draft is not None:
            toks, lps = small_draft(state, v, m)
            for y, lp in zip(toks, lps):
                parent.append(v)
                token.append(int(y))
                edge.append(np.float32(lp))
                score.append(np.float32(score[v] + np.float32(lp)))
                made.append(len(parent) - 1)
            continue
        x, lse = _row_log_softmax(table, v, bf16)
        order = np.lexsort((np.arange(len(x)), -x))[:m]
        for y in order:
            lp = np.float32(x[y] - lse)
            parent.append(v)
            token.append(int(y))
            edge.append(lp)
            score.append(np.float32(score[v] + lp))
            made.append(len(parent) - 1)
    if a == 1:
        P.update(C)
    state["new"] = made
    return F


def grow_tree(schedule, W: int, m: int, small_logits, middle_logits, *, bf16: bool = False):
    """TreeGraft shared-tree construction (Algorithm 2) for one sequence: the
    steps of `schedule` (0 = small drafter, 1 = middle drafter) applied in
    order by grow_step from the root alone.

    Returns parent int32, token int32, edge f32, score f32 (per node), the
    visited set P as uint8, and the list of frontiers (one per step).
    """
    state = grow_state()
    frontiers = [grow_step(state, a, W, m, small_logits, middle_logits, bf16=bf16)
                 for a in schedule]
    parent = state["parent"]
    visited = np.zeros(len(parent), dtype=np.uint8)
    visited[sorted(state["P"])] = 1
    return (np.asarray(parent, np.int32), np.asarray(state["token"], np.int32),
            np.asarray(state["edge"], np.float32), np.asarray(state["score"], np.float32),
            visited, frontiers)
