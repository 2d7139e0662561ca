"""CPU oracle for stochastic tree verification at temperature T > 0 (test
infrastructure only).

The verification step of Algorithms 1 and 2 is the usual rejection sampling
of tree speculative decoding, and Sec. 3.2 (Distribution preservation) rests
on it keeping the target's output distribution; the paper prints no formula.
This is that rule for a tree whose children are deterministic proposals
(TreeGraft drafts by Top_m, not by sampling), the form used by tree-SD
verifiers that draft without replacement:

  at node v (from the root), with p = softmax(l_v / T) and the residual
  r = p, visit v's children in ascending node id; child c with token x is
  accepted with probability r(x) / sum(r), decided by the caller's uniform
  u[c, 0]: accept iff u[c, 0] * sum(r) < r(x); a rejected child's token
  leaves the residual (r(x) = 0).  An accepted child becomes v and the walk
  goes on; when every child is rejected (or v is a leaf) the bonus token is
  drawn from r / sum(r) by inversion with u[v, 1]: the first token t (in
  token order) whose cumulative residual mass exceeds u[v, 1] * sum(r).

Each emitted token is then distributed exactly as p (a child's token is
emitted with probability p(x), any other token t with probability
(1 - sum of children's p) * p(t) / (1 - sum of children's p)); a child whose
token repeats an earlier sibling's has r(x) = 0 and is never accepted.  At
T -> 0 the rule becomes the greedy walk of treegraft_oracle.accept.

Only the test-suite, the package smoke check and the benchmark's CPU-baseline
leg may import it; the product path never calls it.  It shares no code with
the CUDA library.  Pinned by tests/test_oracle_sample.py (hand-worked cases,
inversion against numpy's searchsorted, the T -> 0 limit against the greedy
oracle, and the distribution of the emitted tokens by Monte Carlo).
Parity status: target_probs, accept_sample: pinned.
"""
from __future__ import annotations

import numpy as np

from oracle import treegraft_oracle as O


def target_probs(target_logits, r: int, T: float, *, bf16: bool = False) -> np.ndarray:
    """softmax(l_r / T) of one target row in fp64."""
    x = O._row_values(target_logits, r, bf16)
    m = x.max()
    e = np.exp((x - m) / T)
    return e / e.sum()


def accept_sample(target_logits, token, parent, node_off, u, T: float, path_cap: int, *,
                  bf16: bool = False):
    """Stochastic verification walk of every tree (see the module text).

    u is fp32 [n_total, 2] in [0, 1): u[c, 0] decides child c, u[v, 1] the
    bonus draw at v.  Returns path int32 [B, path_cap] (root-first local
    ids, -1 padded), accept_len int32 [B] (non-root nodes accepted), bonus
    int32 [B], and per tree a dict with the accepted node `astar`, the
    smallest decision margin |u * sum(r) - r(x)| / sum(r) met on the walk
    (`margin`), the bonus row's residual `resid` (fp64 [V]) and the draw's
    target mass `target` = u * sum(resid).
    """
    slices = O._tree_slices(node_off)
    B = len(slices)
    path = np.full((B, path_cap), -1, dtype=np.int32)
    alen = np.zeros(B, dtype=np.int32)
    bonus = np.zeros(B, dtype=np.int32)
    info = []
    for b, (a, e) in enumerate(slices):
        par = np.asarray(parent[a:e])
        O.check_tree(par)
        n = e - a
        children = [[] for _ in range(n)]
        for c in range(1, n):
            children[int(par[c])].append(c)          # ascending id
        v, chain, margin = 0, [0], np.inf
        while True:
            p = target_probs(target_logits, a + v, T, bf16=bf16)
            R = 1.0
            rejected = set()
            nxt = None
            for c in children[v]:
                x = int(token[a + c])
                if x in rejected:
                    continue                             # r(x) = 0
                lhs = float(u[a + c, 0]) * R
                margin = min(margin, abs(lhs - p[x]) / R)
                if lhs < p[x]:
                    nxt = c
                    break
                rejected.add(x)
                R -= p[x]
            if nxt is None:
                break
            v = nxt
            chain.append(v)
        resid = p.copy()
        for c in children[v]:
            resid[int(token[a + c])] = 0.0
        total = resid.sum()
        target = float(u[a + v, 1]) * total
        cum = np.cumsum(resid)
        hits = np.flatnonzero(cum > target)
        if len(hits):
            y = int(hits[0])
        else:                       # u * sum(r) rounded up to sum(r): the last token with mass
            pos = np.flatnonzero(resid > 0)
            y = int(pos[-1]) if len(pos) else int(np.argmax(p))
        if len(chain) > path_cap:
            raise ValueError("accepted path longer than path_cap")
        path[b, :len(chain)] = chain
        alen[b] = len(chain) - 1
        bonus[b] = y
        info.append(dict(astar=v, margin=margin, resid=resid, target=target))
    return path, alen, bonus, info
