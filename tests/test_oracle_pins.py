"""Pins for the CPU oracle: each oracle function is checked against something
other than itself (brute force, closed forms, invariants, an independently
written algorithm), so that a dropped term, a sign or index slip or a
transposed operand in the oracle fails here.  CPU only."""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import treegraft_oracle as O
from paper_2608_26112_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def all_trees(n):
    """Every parent vector with parent[0] = -1 and 0 <= parent[i] < i."""
    for tail in itertools.product(*[range(i) for i in range(1, n)]):
        yield np.array((-1,) + tail, dtype=np.int32)


# --------------------------------------------------------------------------
# mask (Algorithm 3)
# --------------------------------------------------------------------------

def closure_mask(parent):
    """Independent mask: reflexive-transitive closure of the child->parent
    relation by repeated boolean matrix products, plus the root column."""
    n = len(parent)
    A = np.eye(n, dtype=bool)
    for v in range(1, n):
        A[v, parent[v]] = True
    R = A.copy()
    for _ in range(n):
        R = (R.astype(np.int64) @ A.astype(np.int64)) > 0
    R[:, 0] = True
    return R


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6, 7])
def test_mask_matches_closure_on_every_tree(n):
    count = 0
    for parent in all_trees(n):
        m = O.ancestor_mask(parent)
        assert np.array_equal(m, closure_mask(parent))
        count += 1
    assert count == math.factorial(n - 1)


def test_mask_row_count_is_depth_plus_one():
    rng = synth.make_rng(3)
    for _ in range(20):
        parent = synth.sample_tree(rng, 40, 6, 10, 0.3)
        m = O.ancestor_mask(parent)
        d = O.node_depth(parent)
        assert np.array_equal(m.sum(1), d + 1)
        # the mask of u contains the mask of its parent, plus u itself
        for u in range(1, len(parent)):
            assert m[u, u] and np.all(m[u] >= m[parent[u]])
            assert m[u].sum() == m[parent[u]].sum() + 1


def test_mask_star_tree():
    parent = np.array([-1] + [0] * 9, dtype=np.int32)
    m = O.ancestor_mask(parent)
    for u in range(1, 10):
        assert set(np.nonzero(m[u])[0]) == {0, u}


def test_depth_enumeration_against_paths():
    for parent in all_trees(6):
        d = O.node_depth(parent)
        for u in range(6):
            k, v = 0, u
            while v:
                v = parent[v]
                k += 1
            assert d[u] == k


def test_check_tree_rejects_bad_parents():
    for bad in ([0, 0], [-1, 1], [-1, 0, 3], [-1, -1]):
        with pytest.raises(ValueError):
            O.check_tree(np.array(bad))


# --------------------------------------------------------------------------
# tree attention
# --------------------------------------------------------------------------

def _rand_attn(seed, B, P, n, Hq, Hkv, D, parent=None, depth=3):
    rng = synth.make_rng(seed)
    Ps = [P] * B if np.isscalar(P) else list(P)
    ns = [n] * B if np.isscalar(n) else list(n)
    parents, off = [], [0]
    for b in range(B):
        parents.append(parent if parent is not None else synth.sample_tree(rng, ns[b], min(depth, ns[b] - 1) if ns[b] > 1 else 0, None))
        off.append(off[-1] + ns[b])
    par = np.concatenate(parents).astype(np.int32)
    S = max(Ps[b] + ns[b] for b in range(B))
    q = synth.f32_to_bf16_bits(synth.normal_f32(rng, (off[-1], Hq, D)))
    k = synth.kv_cache(rng, B, Hkv, S, D, [Ps[b] + ns[b] for b in range(B)])
    v = synth.kv_cache(rng, B, Hkv, S, D, [Ps[b] + ns[b] for b in range(B)])
    return q, k, v, np.array(Ps, np.int32), par, np.array(off, np.int32)


def causal_loop(q, K, V, scale):
    """Plain causal attention written with Python loops: query i attends to
    keys 0..i of its own sequence."""
    out = []
    for i in range(len(q)):
        s = [scale * sum(q[i][d] * K[j][d] for d in range(len(q[i]))) for j in range(i + 1)]
        m = max(s)
        w = [math.exp(x - m) for x in s]
        z = math.fsum(w)
        out.append([math.fsum(w[j] * V[j][d] for j in range(i + 1)) / z for d in range(len(V[0]))])
    return np.array(out)


def test_chain_tree_is_causal_attention_loop():
    # a chain (parent[i] = i - 1) sees prefix + all earlier nodes: causal attention
    P, n, D = 5, 6, 8
    chain = np.arange(-1, n - 1, dtype=np.int32)
    q, k, v, Ps, par, off = _rand_attn(11, 1, P, n, 2, 1, D, parent=chain)
    o, _ = O.tree_attention(q, k, v, Ps, par, off, Hkv=1)
    K = O.bf16_bits_to_f64(k)[0, 0, :P + n]
    Vv = O.bf16_bits_to_f64(v)[0, 0, :P + n]
    qq = O.bf16_bits_to_f64(q)
    for h in range(2):
        # queries of the prefix are irrelevant; pad with the keys themselves
        full_q = np.concatenate([np.zeros((P, D)), qq[:, h]], axis=0)
        ref = causal_loop(full_q.tolist(), K.tolist(), Vv.tolist(), 1 / math.sqrt(D))[P:]
        np.testing.assert_allclose(o[:, h], ref, rtol=1e-12, atol=1e-12)


def test_chain_tree_is_torch_causal_sdpa():
    P, n, Hq, Hkv, D = 64, 32, 8, 2, 16
    chain = np.arange(-1, n - 1, dtype=np.int32)
    q, k, v, Ps, par, off = _rand_attn(12, 1, P, n, Hq, Hkv, D, parent=chain)
    o, lse = O.tree_attention(q, k, v, Ps, par, off, Hkv=Hkv)
    qq = torch.tensor(O.bf16_bits_to_f64(q)).permute(1, 0, 2)            # [Hq, n, D]
    K = torch.tensor(O.bf16_bits_to_f64(k)[0, :, :P + n]).repeat_interleave(Hq // Hkv, 0)
    Vv = torch.tensor(O.bf16_bits_to_f64(v)[0, :, :P + n]).repeat_interleave(Hq // Hkv, 0)
    allowed = torch.ones(n, P + n, dtype=torch.bool)
    allowed[:, P:] = torch.tril(torch.ones(n, n, dtype=torch.bool))
    ref = torch.nn.functional.scaled_dot_product_attention(qq, K, Vv, attn_mask=allowed)
    np.testing.assert_allclose(o, ref.permute(1, 0, 2).numpy(), rtol=1e-10, atol=1e-12)
    s = (qq @ K.transpose(1, 2)) / math.sqrt(D)
    s = s.masked_fill(~allowed, float("-inf"))
    np.testing.assert_allclose(lse, torch.logsumexp(s, -1).T.numpy(), rtol=1e-12)


def test_single_node_is_decode_attention():
    P, D = 40, 32
    q, k, v, Ps, par, off = _rand_attn(13, 1, P, 1, 4, 4, D)
    o, _ = O.tree_attention(q, k, v, Ps, par, off, Hkv=4)
    qq, K, Vv = (O.bf16_bits_to_f64(x) for x in (q, k, v))
    for h in range(4):
        s = K[0, h, :P + 1] @ qq[0, h] / math.sqrt(D)
        w = np.exp(s - s.max())
        np.testing.assert_allclose(o[0, h], w @ Vv[0, h, :P + 1] / w.sum(), rtol=1e-12)


def test_gqa_equals_repeated_kv_heads():
    Hq, Hkv = 8, 2
    q, k, v, Ps, par, off = _rand_attn(14, 2, [17, 30], [9, 12], Hq, Hkv, 16)
    o, lse = O.tree_attention(q, k, v, Ps, par, off, Hkv=Hkv)
    k_rep = np.repeat(k, Hq // Hkv, axis=1)   # kv head j serves q heads j*G .. j*G+G-1
    v_rep = np.repeat(v, Hq // Hkv, axis=1)
    o2, lse2 = O.tree_attention(q, k_rep, v_rep, Ps, par, off, Hkv=Hq)
    np.testing.assert_array_equal(o, o2)
    np.testing.assert_array_equal(lse, lse2)


def test_identical_value_rows_give_that_row():
    q, k, v, Ps, par, off = _rand_attn(15, 1, 20, 10, 2, 2, 8)
    row = synth.f32_to_bf16_bits(np.linspace(-1, 1, 8, dtype=np.float32))
    v[:] = row
    o, _ = O.tree_attention(q, k, v, Ps, par, off, Hkv=2)
    np.testing.assert_allclose(o, np.broadcast_to(O.bf16_bits_to_f64(row), o.shape), rtol=1e-14)


def test_relabelling_nodes_permutes_outputs():
    # swap the labels of two sibling subtrees' roots: a topological relabelling
    rng = synth.make_rng(16)
    P, n, D, H = 12, 7, 8, 2
    parent = np.array([-1, 0, 0, 1, 2, 3, 4], dtype=np.int32)
    perm = np.array([0, 2, 1, 4, 3, 6, 5])        # new label -> old label
    inv = np.argsort(perm)
    par2 = np.array([-1] + [inv[parent[perm[i]]] for i in range(1, n)], dtype=np.int32)
    O.check_tree(par2)
    q = synth.f32_to_bf16_bits(synth.normal_f32(rng, (n, H, D)))
    k = synth.kv_cache(rng, 1, H, P + n, D, [P + n])
    v = synth.kv_cache(rng, 1, H, P + n, D, [P + n])
    o, _ = O.tree_attention(q, k, v, [P], parent, [0, n], Hkv=H)
    k2, v2 = k.copy(), v.copy()
    k2[:, :, P:] = k[:, :, P + perm]
    v2[:, :, P:] = v[:, :, P + perm]
    o2, _ = O.tree_attention(q[perm], k2, v2, [P], par2, [0, n], Hkv=H)
    np.testing.assert_allclose(o2, o[perm], rtol=1e-13)


def test_zero_prefix_root_attends_only_to_itself():
    q, k, v, Ps, par, off = _rand_attn(17, 1, 0, 5, 2, 2, 8)
    o, lse = O.tree_attention(q, k, v, Ps, par, off, Hkv=2)
    Vv = O.bf16_bits_to_f64(v)
    np.testing.assert_allclose(o[0], Vv[0, :, 0], rtol=1e-14)


# --------------------------------------------------------------------------
# expand_topk
# --------------------------------------------------------------------------

def brute_topk(x, k, parent_score):
    idx = sorted(range(len(x)), key=lambda t: (-x[t], t))[:k]
    m = max(x)
    lse = m + math.log(math.fsum(math.exp(t - m) for t in x))
    return idx, [x[t] - lse for t in idx], [parent_score + x[t] - lse for t in idx], lse


def test_expand_topk_brute_force():
    rng = synth.make_rng(21)
    x = synth.normal_f32(rng, (6, 300), 3.0)
    ps = synth.normal_f32(rng, (6,), 2.0)
    tok, lp, sc, lse = O.expand_topk(x, ps, 7)
    for r in range(6):
        i, l, s, z = brute_topk([float(t) for t in x[r]], 7, float(ps[r]))
        assert list(tok[r]) == i
        np.testing.assert_allclose(lp[r], l, rtol=1e-6)
        np.testing.assert_allclose(sc[r], s, rtol=1e-6)
        assert abs(lse[r] - z) < 1e-12 * max(1, abs(z))


def test_expand_topk_uniform_row():
    V = 1000
    tok, lp, sc, lse = O.expand_topk(np.zeros((1, V), np.float32), np.zeros(1, np.float32), 5)
    assert list(tok[0]) == [0, 1, 2, 3, 4]
    np.testing.assert_allclose(lp[0], -math.log(V), rtol=1e-7)
    np.testing.assert_allclose(lse[0], math.log(V), rtol=1e-15)


def test_expand_topk_spike_and_row_idx_and_bf16():
    x = np.zeros((3, 64), np.float32)
    x[1, 17] = 1e4
    bits = synth.f32_to_bf16_bits(x)
    tok, lp, sc, _ = O.expand_topk(bits, np.array([-1.0, -2.0], np.float32), 2,
                                   row_idx=[1, 0], bf16=True)
    assert tok[0, 0] == 17 and abs(lp[0, 0]) < 1e-6 and abs(sc[0, 0] + 1.0) < 1e-6
    assert list(tok[1]) == [0, 1]
    assert tok[0, 1] == 0 and lp[0, 1] < -9000


def test_expand_topk_ties_and_neg_inf():
    x = np.array([[-1, 0, 1, 1, 0, -1, 1, 0]], np.float32)
    tok, lp, _, _ = O.expand_topk(x, np.zeros(1, np.float32), 5)
    assert list(tok[0]) == [2, 3, 6, 1, 4]
    y = np.full((2, 6), -np.inf, np.float32)
    y[0, 3] = 0.5
    tok, lp, sc, lse = O.expand_topk(y, np.zeros(2, np.float32), 3)
    assert tok[0, 0] == 3 and lp[0, 0] == 0.0 and np.isneginf(lp[0, 1])
    assert list(tok[1]) == [0, 1, 2] and np.all(np.isneginf(lp[1])) and np.isneginf(lse[1])
    # negative zero ties with positive zero: the lower token wins
    z = np.array([[0.0, -0.0, -0.0, 0.0]], np.float32)
    z[0, 0] = -0.0
    tok, _, _, _ = O.expand_topk(z, np.zeros(1, np.float32), 4)
    assert list(tok[0]) == [0, 1, 2, 3]


# --------------------------------------------------------------------------
# rescore_select
# --------------------------------------------------------------------------

def brute_rescore(weak, strong, parent, token, visited, N):
    n = len(parent)
    edge = [0.0] * n
    for v in range(1, n):
        edge[v] = float(weak[v]) if visited[v] else float(strong[parent[v]][token[v]])
    score = []
    for v in range(n):
        chain = []
        w = v
        while w > 0:
            chain.append(w)
            w = parent[w]
        acc = np.float32(0)
        for w in reversed(chain):            # root-first fp32 additions
            acc = np.float32(acc + np.float32(edge[w]))
        score.append(acc)
    cand = [v for v in range(n) if not visited[v]]
    best = sorted(cand, key=lambda v: (-float(score[v]), v))[:N]
    return np.array(edge, np.float32), np.array(score, np.float32), best


def test_rescore_select_brute_force():
    rng = synth.make_rng(31)
    for trial in range(5):
        n, V = 30, 50
        parent = synth.sample_tree(rng, n, 5, 4, 0.3)
        token = synth.sample_tokens(rng, n, V)
        weak = synth.normal_f32(rng, (n,), 2.0, -3.0)
        strong = synth.normal_f32(rng, (n, V), 2.0, -4.0)
        visited = (rng.random(n) < 0.4).astype(np.uint8)
        e, s, sel, ns = O.rescore_select(weak, strong, parent, token, visited, [0, n], 8)
        e2, s2, best = brute_rescore(weak, strong, parent, token, visited, 8)
        np.testing.assert_array_equal(e, e2)
        np.testing.assert_array_equal(s, s2)
        assert list(sel[0, :ns[0]]) == best and np.all(sel[0, ns[0]:] == -1)


def test_rescore_select_unchanged_scores_when_strong_equals_weak():
    # strong rows carry exactly the stored edge scores: rescoring changes nothing,
    # so the scores are the plain cumulative sums and the selection is plain top-N
    rng = synth.make_rng(32)
    n, V = 40, 64
    parent = synth.sample_tree(rng, n, 6, 5, 0.3)
    token = synth.sample_tokens(rng, n, V)
    weak = synth.normal_f32(rng, (n,), 1.0, -2.0)
    strong = synth.normal_f32(rng, (n, V), 1.0, -9.0)
    for v in range(1, n):
        strong[parent[v], token[v]] = weak[v]
    dup = {}
    for v in range(1, n):            # duplicate sibling tokens would overwrite; skip them
        dup.setdefault((parent[v], token[v]), []).append(v)
    if any(len(x) > 1 for x in dup.values()):
        pytest.skip("duplicate sibling tokens in draw")
    vis = np.zeros(n, np.uint8)
    e, s, sel, ns = O.rescore_select(weak, strong, parent, token, vis, [0, n], 10)
    d = O.node_depth(parent)
    cum = np.zeros(n, np.float32)
    for v in np.argsort(d, kind="stable"):
        if v:
            cum[v] = np.float32(cum[parent[v]] + weak[v])
    np.testing.assert_array_equal(s, cum)
    assert list(sel[0]) == sorted(range(n), key=lambda v: (-float(cum[v]), v))[:10]


def test_rescore_select_all_visited_and_root_candidate():
    n = 6
    parent = np.array([-1, 0, 0, 1, 1, 2], np.int32)
    token = np.arange(n, dtype=np.int32)
    weak = np.array([0, -1, -2, -3, -4, -5], np.float32)
    strong = np.full((n, n), -100.0, np.float32)
    e, s, sel, ns = O.rescore_select(weak, strong, parent, token, np.ones(n, np.uint8), [0, n], 3)
    assert ns[0] == 0 and np.all(sel == -1)
    np.testing.assert_array_equal(s, [0, -1, -2, -4, -5, -7])
    # first middle step: nothing visited; the root (score 0) is the best candidate
    e, s, sel, ns = O.rescore_select(weak, strong, parent, token, np.zeros(n, np.uint8), [0, n], 3)
    assert list(sel[0]) == [0, 1, 2] and ns[0] == 3
    assert s[1] == -100 and s[3] == -200


# --------------------------------------------------------------------------
# accept
# --------------------------------------------------------------------------

def level_sweep_accept(am, token, parent):
    """Independent accept: one pass in node order (parents precede children)."""
    n = len(parent)
    full = [True] + [False] * (n - 1)
    depth = [0] * n
    for v in range(1, n):
        depth[v] = depth[parent[v]] + 1
        full[v] = full[parent[v]] and token[v] == am[parent[v]]
    best = max((depth[v], -v) for v in range(n) if full[v])
    a = -best[1]
    path = []
    while a != -1:
        path.append(a)
        a = parent[a]
    return path[::-1]


def logits_with_argmax(am, V, rng, ties=False):
    x = synth.normal_f32(rng, (len(am), V), 1.0)
    for r, t in enumerate(am):
        x[r, t] = 10.0
        if ties and t + 1 < V:
            x[r, t + 1] = 10.0            # tie: the lower token must win
    return x


def test_accept_matches_level_sweep():
    rng = synth.make_rng(41)
    for trial in range(30):
        n, V = int(rng.integers(1, 25)), 6
        parent = synth.sample_tree(rng, n, min(4, n - 1), None) if n > 1 else np.array([-1], np.int32)
        token = synth.sample_tokens(rng, n, V)
        am = rng.integers(0, V - 1, size=n)
        x = logits_with_argmax(am, V, rng, ties=True)
        path, A, bonus = O.accept(x, token, parent, [0, n], n)
        ref = level_sweep_accept(am, token, parent)
        assert list(path[0, :len(ref)]) == ref and np.all(path[0, len(ref):] == -1)
        assert A[0] == len(ref) - 1 and bonus[0] == am[ref[-1]]


def test_accept_chain_fully_planted():
    n, V = 9, 20
    parent = np.arange(-1, n - 1, dtype=np.int32)
    rng = synth.make_rng(42)
    token = synth.sample_tokens(rng, n, V)
    am = np.append(token[1:], 3)
    x = logits_with_argmax(am, V, rng)
    path, A, bonus = O.accept(x, token, parent, [0, n], n)
    assert A[0] == n - 1 and list(path[0]) == list(range(n)) and bonus[0] == 3


def test_accept_no_match():
    n, V = 7, 10
    parent = np.array([-1, 0, 0, 1, 1, 2, 2], np.int32)
    token = np.array([0, 1, 1, 2, 2, 3, 3], np.int32)
    rng = synth.make_rng(43)
    x = logits_with_argmax([5] * n, V, rng)
    path, A, bonus = O.accept(x, token, parent, [0, n], 4)
    assert A[0] == 0 and list(path[0]) == [0, -1, -1, -1] and bonus[0] == 5


def test_accept_duplicate_sibling_prefers_deeper_then_lower_id():
    # node 1 and node 2 carry the same token under the root; node 2 has a child
    parent = np.array([-1, 0, 0, 2], np.int32)
    token = np.array([0, 4, 4, 7], np.int32)
    am = [4, 1, 7, 2]
    x = logits_with_argmax(am, 9, synth.make_rng(44))
    path, A, bonus = O.accept(x, token, parent, [0, 4], 4)
    assert list(path[0]) == [0, 2, 3, -1] and A[0] == 2 and bonus[0] == 2
    x = logits_with_argmax([4, 1, 8, 2], 9, synth.make_rng(45))
    path, A, bonus = O.accept(x, token, parent, [0, 4], 4)
    assert list(path[0, :2]) == [0, 1] and A[0] == 1 and bonus[0] == 1


def test_accept_grafting_examples():
    """Tree shapes of the two non-destructive grafting traces (Appendix G):
    a grafting node that keeps a historical chain of four nodes next to newly
    attached siblings; the target follows the historical chain."""
    with open(os.path.join(GOLDEN, "grafting_examples.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        parent = np.array(case["parent"], np.int32)
        token = np.array(case["token"], np.int32)
        n, V = len(parent), case["vocab"]
        am = np.array(case["target_argmax"])
        x = logits_with_argmax(am, V, synth.make_rng(46))
        path, A, bonus = O.accept(x, token, parent, [0, n], n)
        exp = case["accepted_path"]
        assert list(path[0, :len(exp)]) == exp
        assert A[0] == len(exp) - 1 and bonus[0] == case["bonus"]


def test_accept_batched_trees_are_independent():
    rng = synth.make_rng(47)
    ns = [5, 1, 8]
    parents = [synth.sample_tree(rng, 5, 2), np.array([-1], np.int32), synth.sample_tree(rng, 8, 3)]
    par = np.concatenate(parents)
    tok = synth.sample_tokens(rng, 14, 5)
    x = synth.normal_f32(rng, (14, 5), 2.0)
    off = [0, 5, 6, 14]
    path, A, bonus = O.accept(x, tok, par, off, 8)
    for b in range(3):
        p1, a1, b1 = O.accept(x[off[b]:off[b + 1]], tok[off[b]:off[b + 1]], parents[b], [0, ns[b]], 8)
        assert np.array_equal(path[b], p1[0]) and A[b] == a1[0] and bonus[b] == b1[0]


# ------------------------------------------------------------------ GlobalPrune (Algorithm 3)

def top_nodes(parent, score, M):
    """Root plus the M - 1 best non-root nodes by (score desc, depth asc,
    id asc), by a library sort."""
    n = len(parent)
    d = O.node_depth(parent)
    ids = np.arange(1, n)
    order = np.lexsort((ids, d[1:], -np.asarray(score, np.float64)[1:]))
    return sorted([0] + ids[order[:M - 1]].tolist())


def check_prune_buffers(parent, kept, k, new_par, pos, mask, paths, n_paths):
    """Properties any GlobalPrune result must have."""
    kept = kept[:k].tolist()
    assert kept[0] == 0 and kept == sorted(kept)
    ks = set(kept)
    for v in kept[1:]:
        assert int(parent[v]) in ks                          # ancestor-closed
    d = O.node_depth(parent)
    for i, v in enumerate(kept):
        assert pos[i] == d[v]
        assert new_par[i] == (-1 if i == 0 else kept.index(int(parent[v])))
    np.testing.assert_array_equal(mask[:k, :k], O.ancestor_mask(new_par[:k]))
    assert not mask[k:].any() and not mask[:, k:].any()
    leaves = [i for i in range(k) if i not in set(new_par[1:k].tolist())]
    assert n_paths == len(leaves)
    for j, leaf in enumerate(leaves):
        row = paths[j]
        length = int((row >= 0).sum())
        assert row[length - 1] == leaf and row[0] == 0
        assert all(new_par[row[t]] == row[t - 1] for t in range(1, length))
        assert (row[length:] == -1).all()
    assert (paths[n_paths:] == -1).all()


def test_global_prune_small_tree_is_returned_unchanged():
    rng = synth.make_rng(60)
    parent = synth.sample_tree(rng, 12, 4)
    score = synth.normal_f32(rng, (12,), 2.0)
    kept, k, new_par, pos, mask, paths, npth = O.global_prune(parent, score, [0, 12], 11, 8)
    assert k[0] == 12 and list(kept[0]) == list(range(12))
    np.testing.assert_array_equal(new_par[0], parent)
    np.testing.assert_array_equal(pos[0], O.node_depth(parent))
    check_prune_buffers(parent, kept[0], 12, new_par[0], pos[0], mask[0], paths[0], npth[0])


@pytest.mark.parametrize("seed", range(6))
def test_global_prune_path_monotone_scores_keep_the_top_nodes(seed):
    """With scores that never increase from parent to child (sums of
    log-probabilities), every node ranks after its parent, each ranked chain
    is the node alone, and Algorithm 3 keeps exactly the root and the
    budget's best nodes."""
    rng = synth.make_rng(61 + seed)
    parent = synth.expansion_tree(rng, 5, 4, 3)
    score = synth.path_scores(rng, parent)
    n = len(parent)
    for budget in (1, 7, 20, n - 2):
        kept, k, new_par, pos, mask, paths, npth = O.global_prune(parent, score, [0, n], budget, 12)
        assert kept[0, :k[0]].tolist() == top_nodes(parent, score, budget + 1)
        check_prune_buffers(parent, kept[0], k[0], new_par[0], pos[0], mask[0], paths[0], npth[0])


def test_global_prune_chain_keeps_the_first_nodes():
    """On a chain every node's ancestors are the nodes before it, so only
    chains ending at nodes 1..M-1 fit: the first M nodes are kept, whatever
    the scores."""
    rng = synth.make_rng(62)
    n = 30
    parent = np.arange(-1, n - 1, dtype=np.int32)
    score = synth.normal_f32(rng, (n,), 5.0)
    kept, k, new_par, pos, mask, paths, npth = O.global_prune(parent, score, [0, n], 9, 12)
    assert kept[0, :k[0]].tolist() == list(range(10))
    assert npth[0] == 1 and paths[0, 0].tolist() == list(range(10)) + [-1, -1]


def test_global_prune_star_is_plain_top_k():
    rng = synth.make_rng(63)
    n = 40
    parent = np.zeros(n, dtype=np.int32)
    parent[0] = -1
    score = np.round(synth.normal_f32(rng, (n,), 2.0)).astype(np.float32)  # many ties
    kept, k, *_ = O.global_prune(parent, score, [0, n], 12, 3)
    ids = np.arange(1, n)
    order = np.lexsort((ids, -score[1:].astype(np.float64)))
    assert kept[0, :k[0]].tolist() == sorted([0] + ids[order[:12]].tolist())


def test_global_prune_skips_a_long_chain_and_keeps_ranking():
    """Worked by hand from Algorithm 3 with M = 3: the best node x sits at
    depth 3 and its chain (x, b, a) would make |K| = 4 > 3, so it is
    skipped; c and e then fit and fill K = {r, c, e}."""
    #          r   a  b  x  c  e
    parent = np.array([-1, 0, 1, 2, 0, 0], np.int32)
    score = np.array([0, -1, -2, 10, 5, 4], np.float32)
    kept, k, new_par, pos, mask, paths, npth = O.global_prune(parent, score, [0, 6], 2, 3)
    assert kept[0, :k[0]].tolist() == [0, 4, 5]
    assert new_par[0].tolist() == [-1, 0, 0] and pos[0].tolist() == [0, 1, 1]
    assert npth[0] == 2 and paths[0].tolist() == [[0, 1, -1], [0, 2, -1], [-1, -1, -1]]


def test_global_prune_ties_prefer_shallower_then_lower_id():
    """Equal scores: depth decides (shallower first), then the lower id."""
    #          r  a  b  c  d
    parent = np.array([-1, 0, 1, 0, 0], np.int32)
    score = np.array([0, 1, 3, 3, 3], np.float32)      # b (depth 2) ties c, d (depth 1)
    kept, k, *_ = O.global_prune(parent, score, [0, 5], 2, 4)
    assert kept[0, :k[0]].tolist() == [0, 3, 4]        # c, d before b; b's chain no longer fits
    kept, k, *_ = O.global_prune(parent, score, [0, 5], 1, 4)
    assert kept[0, :k[0]].tolist() == [0, 3]           # c before d by id


def test_global_prune_random_scores_batched_invariants():
    rng = synth.make_rng(64)
    parents, scores, off = [], [], [0]
    for n in (1, 9, 40, 77):
        p = synth.sample_tree(rng, n, min(n - 1, 6)) if n > 1 else np.array([-1], np.int32)
        parents.append(p)
        scores.append(synth.normal_f32(rng, (n,), 3.0))
        off.append(off[-1] + n)
    par, sc = np.concatenate(parents), np.concatenate(scores)
    out = O.global_prune(par, sc, off, 15, 10)
    for b in range(4):
        single = O.global_prune(parents[b], scores[b], [0, len(parents[b])], 15, 10)
        assert out[1][b] == single[1][0]
        Mo = out[0].shape[1]
        check_prune_buffers(parents[b], out[0][b], out[1][b], out[2][b], out[3][b], out[4][b],
                            out[5][b], out[6][b])
        assert out[1][b] <= 16


# ------------------------------------------------------------------ grow loop (Algorithm 2)

def _lsm(row):
    from scipy.special import log_softmax
    return log_softmax(np.asarray(row, np.float64))


def test_grow_tree_hand_worked_graft():
    """Worked by hand from Algorithm 2 with W = 1, m = 2 and schedule
    (small, middle, small).  Step 1 expands the root with the small drafter's
    two best tokens (1, 3).  Step 2: P is empty, so C = {r, 1, 2}; nodes 1
    and 2 are rescored from the middle drafter's root row, the root (score
    0, the largest possible) is the frontier and gets the middle drafter's
    two best tokens 3 and 0 (tie at 0 to the lower token) - a second child
    with token 3 is attached next to node 2, not over it.  Step 3 expands the
    better of the new nodes {3, 4}: node 3."""
    rng = synth.make_rng(70)
    small = synth.normal_f32(rng, (8, 4), 1.0)
    small[0] = [0.0, 3.0, 1.0, 2.0]
    middle = synth.normal_f32(rng, (8, 4), 1.0)
    middle[0] = [0.0, 0.0, 0.0, 5.0]
    par, tok, edge, score, vis, fr = O.grow_tree([0, 1, 0], 1, 2, small, middle)
    assert par.tolist() == [-1, 0, 0, 0, 0, 3, 3]
    t56 = np.lexsort((np.arange(4), -small[3].astype(np.float64)))[:2].tolist()
    assert tok.tolist() == [0, 1, 3, 3, 0] + t56
    assert fr == [[0], [0], [3]]
    assert vis.tolist() == [1, 1, 1, 0, 0, 0, 0]
    lm, ls3 = _lsm(middle[0]), _lsm(small[3])
    expect = [0.0, lm[1], lm[3], lm[3], lm[0], lm[3] + ls3[t56[0]], lm[3] + ls3[t56[1]]]
    np.testing.assert_allclose(score, expect, atol=2e-6)
    np.testing.assert_allclose(edge[1:3], [lm[1], lm[3]], atol=1e-6)   # rescored edges


def test_grow_tree_all_small_is_single_drafter_construction():
    """With every step on the small drafter, Algorithm 2 is Algorithm 1:
    each frontier is the best W of the previous step's nodes, every node's
    score is the sum of small-drafter log-probabilities along its path, and
    nothing is visited."""
    rng = synth.make_rng(71)
    V, W, m, D = 32, 2, 3, 3
    small = synth.normal_f32(rng, (64, V), 2.0)
    middle = synth.normal_f32(rng, (64, V), 2.0)
    par, tok, edge, score, vis, fr = O.grow_tree([0] * D, W, m, small, middle)
    assert len(par) == 1 + m + W * m + W * m and not vis.any()
    prev = [0]
    for k in range(D):
        best = sorted(prev, key=lambda v: (-float(score[v]), v))[:W]
        assert fr[k] == best
        prev = [v for v in range(len(par)) if par[v] in best and v > max(prev)]
    for v in range(1, len(par)):
        lp = _lsm(small[par[v]])[tok[v]]
        assert abs(edge[v] - lp) < 1e-6
        path, w = 0.0, v
        while w:
            path += _lsm(small[par[w]])[tok[w]]
            w = par[w]
        assert abs(score[v] - path) < 1e-5


def test_grow_tree_frontier_ties_go_to_the_lower_node_id():
    """Top_W ranks by (score desc, node id asc).  The root's children come
    from a row whose four best logits are equal, so they carry equal scores;
    the next small step's frontier of W = 2 is the two with the lowest ids,
    and a middle step over the same tree keeps that order among equals."""
    small = np.zeros((32, 8), np.float32)
    small[0, [2, 4, 5, 7]] = 3.0
    middle = np.zeros((32, 8), np.float32)
    par, tok, edge, score, vis, fr = O.grow_tree([0, 0], 2, 4, small, middle)
    assert tok[1:5].tolist() == [2, 4, 5, 7]
    assert len(set(score[1:5].tolist())) == 1
    assert fr == [[0], [1, 2]]
    # middle step: every row uniform, so all non-root scores tie; the root
    # (score 0, the largest) comes first, then the lowest ids
    par, tok, edge, score, vis, fr = O.grow_tree([0, 1], 3, 4, small, middle)
    assert fr[1] == [0, 1, 2]


def test_grow_tree_middle_first_step_expands_the_root():
    rng = synth.make_rng(72)
    small = synth.normal_f32(rng, (32, 16), 2.0)
    middle = synth.normal_f32(rng, (32, 16), 2.0)
    par, tok, edge, score, vis, fr = O.grow_tree([1, 0], 3, 2, small, middle)
    assert fr[0] == [0] and vis.tolist()[:1] == [1] and vis.sum() == 1
    top = np.lexsort((np.arange(16), -middle[0].astype(np.float64)))[:2].tolist()
    assert tok[1:3].tolist() == top and par[1:3].tolist() == [0, 0]


@pytest.mark.parametrize("seed", range(4))
def test_grow_tree_random_schedules_invariants(seed):
    rng = synth.make_rng(73 + seed)
    V, W, m, D = 24, 3, 2, 5
    sched = rng.integers(0, 2, size=D).tolist()
    cap = 1 + D * W * m
    small = synth.normal_f32(rng, (cap, V), 2.0)
    middle = synth.normal_f32(rng, (cap, V), 2.0)
    par, tok, edge, score, vis, fr = O.grow_tree(sched, W, m, small, middle)
    n = len(par)
    assert n == 1 + m * sum(len(f) for f in fr)
    O.check_tree(par)
    last_mid = max([k for k, a in enumerate(sched) if a == 1], default=-1)
    # P is every node that existed when the last middle step ran
    n_then = 1 + m * sum(len(f) for f in fr[:last_mid]) if last_mid >= 0 else 0
    assert vis.tolist() == [1] * n_then + [0] * (n - n_then)
    for v in range(1, n):
        # a visited node carries the middle drafter's edge; an unvisited one
        # the edge of the drafter whose step created it
        made_at = next(k for k in range(D) if par[v] in fr[k] and
                       v < 1 + m * sum(len(f) for f in fr[:k + 1]))
        table = middle if (vis[v] or sched[made_at] == 1) else small
        assert abs(edge[v] - _lsm(table[par[v]])[tok[v]]) < 1e-6
        assert score[v] == np.float32(score[par[v]] + edge[v])
