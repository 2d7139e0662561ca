"""Parity of stochastic verification (treegraft_accept_sample) with the
oracle's rule (oracle/sample_oracle.py) on the same trees, logits and
uniforms.

The decisions compare fp32 values on the device with fp64 values in the
oracle, so a draw within rounding of a threshold may fall either way.  Bars:
for every tree whose walk decisions all clear their thresholds by more than
1e-4 of the residual mass (the oracle reports the smallest margin), the path
and the accepted length are bit-exact; the bonus token must be a valid draw:
a token with residual mass whose cumulative residual range (fp64, token
order) holds u * sum(r) within 1e-5 of sum(r).  At least 90 % of the trees
of every case are compared exactly."""
import numpy as np
import pytest
import torch

import paper_2608_26112_gb300 as tg
from oracle import sample_oracle as S
from paper_2608_26112_gb300 import synth
from tests import _dev

pytestmark = pytest.mark.gpu

MARGIN = 1e-4
BONUS_TOL = 1e-5


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26112_gb300 import build
    build.build()
    return torch.device("cuda:0")


def _trees(rng, sizes, V, cap, dup_prob=0.0):
    parents, tokens = [], []
    for n in sizes:
        depth = max(1, min(6, n - 1)) if n > 1 else 0
        par = synth.sample_tree(rng, n, depth, cap=cap) if n > 1 else np.array([-1], np.int32)
        tok = rng.integers(0, V, size=n).astype(np.int32)
        if dup_prob:
            for c in range(2, n):       # repeat an earlier sibling's token now and then
                sib = [j for j in range(1, c) if par[j] == par[c]]
                if sib and rng.random() < dup_prob:
                    tok[c] = tok[sib[int(rng.integers(0, len(sib)))]]
        parents.append(par)
        tokens.append(tok)
    off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    return np.concatenate(parents).astype(np.int32), np.concatenate(tokens), off


def _logits(rng, parent, token, off, V, bf16, bump=6.0, prob=0.8):
    x = synth.normal_f32(rng, (len(parent), V), 3.0)
    for b in range(len(off) - 1):
        a, e = int(off[b]), int(off[b + 1])
        synth.plant_child_bump(rng, x[a:e], parent[a:e], token[a:e], np.arange(e - a), prob=prob,
                               bump=bump)
    return synth.f32_to_bf16_bits(x) if bf16 else x


def _run(dev, rng, sizes, V, bf16, T, cap=10, path_cap=12, dup_prob=0.0, bump=12.0):
    parent, token, off = _trees(rng, sizes, V, cap, dup_prob)
    host = _logits(rng, parent, token, off, V, bf16, bump=bump)
    u = rng.random((len(parent), 2)).astype(np.float32)
    lg = _dev.bf16(host, dev) if bf16 else _dev.f32(host, dev)
    B = len(sizes)
    ws = tg.accept_sample_workspace(B, len(parent), dev)
    for _ in range(2):      # the second call checks that the tickets were reset
        path, alen, bonus = tg.accept_sample(lg, _dev.i32(token, dev), _dev.i32(parent, dev),
                                             _dev.i32(off, dev), max(sizes), path_cap,
                                             _dev.f32(u, dev), T, ws)
        torch.cuda.synchronize()
        assert tg.last_device_status() == 0
        assert not torch.any(ws != 0)       # flags, candidates and tickets back to zero
    path, alen, bonus = (t.cpu().numpy() for t in (path, alen, bonus))
    op, oa, ob, info = S.accept_sample(host, token, parent, off, u, T, path_cap, bf16=bf16)
    exact = 0
    for b in range(B):
        if info[b]["margin"] <= MARGIN:
            continue
        exact += 1
        assert path[b].tolist() == op[b].tolist(), b
        assert alen[b] == oa[b]
        resid, target = info[b]["resid"], info[b]["target"]
        y = int(bonus[b])
        assert 0 <= y < V and resid[y] > 0, (b, y)
        cum = np.cumsum(resid)
        tol = BONUS_TOL * cum[-1]
        lo = cum[y - 1] if y > 0 else 0.0
        assert lo - tol <= target <= cum[y] + tol, (b, y, int(ob[b]), lo, target, cum[y])
    assert exact >= 0.9 * B
    return alen


@pytest.mark.parametrize("T", [0.6, 1.0, 1.5])
def test_sample_small_vocab(dev, T):
    rng = synth.make_rng(950 + int(T * 10))
    sizes = rng.integers(1, 41, size=24).tolist()
    alen = _run(dev, rng, sizes, 1024, False, T)
    assert alen.max() >= 2


def test_sample_llama3_vocab(dev):
    """The Llama-3-8B-shaped verify tree: 60 nodes, 128256-token bf16
    target rows, several trees."""
    rng = synth.make_rng(960)
    _run(dev, rng, [60] * 6, synth.LLAMA3_VOCAB, True, 1.0)


def test_sample_duplicate_siblings(dev):
    rng = synth.make_rng(970)
    sizes = [30] * 12
    _run(dev, rng, sizes, 64, False, 0.8, dup_prob=0.5)


def test_sample_low_temperature_matches_greedy(dev):
    """At T = 0.02 the rule is the greedy walk: the same path and bonus as
    treegraft_accept (every row's leading logit 1.0 clear of the next, and no
    repeated sibling tokens, where the greedy rule prefers the deeper
    branch and the walk the first child)."""
    rng = synth.make_rng(980)
    sizes = [40] * 16
    parent, token, off = _trees(rng, sizes, 512, 8)
    host = _logits(rng, parent, token, off, 512, False)
    host[np.arange(len(host)), host.argmax(axis=1)] += np.float32(1.0)   # a clear leader per row
    lg = _dev.f32(host, dev)
    u = _dev.f32(rng.random((len(parent), 2)).astype(np.float32) * np.float32(0.99), dev)
    args = (_dev.i32(token, dev), _dev.i32(parent, dev), _dev.i32(off, dev), 40, 12)
    sp, sa, sb = tg.accept_sample(lg, *args, u, 0.02, tg.accept_sample_workspace(16, 640, dev))
    gp, ga, gb = tg.accept(lg, *args, tg.accept_workspace(16, 640, dev))
    torch.cuda.synchronize()
    assert tg.last_device_status() == 0
    top2 = np.sort(host, axis=1)[:, -2:]
    clear = (top2[:, 1] - top2[:, 0]) > 0.5
    compared = 0
    for b in range(16):
        a, e = int(off[b]), int(off[b + 1])
        fam = [(int(parent[c]), int(token[c])) for c in range(a + 1, e)]
        if clear[a:e].all() and len(set(fam)) == len(fam):   # no repeated sibling token
            compared += 1
            assert sp[b].tolist() == gp[b].tolist() and sa[b] == ga[b] and sb[b] == gb[b]
    assert compared >= 8


def test_sample_single_node_trees_draw_from_the_row(dev):
    """Trees of the root alone: A = 0 and the bonus is an inversion draw of
    the root's row, checked against the cumulative distribution."""
    rng = synth.make_rng(990)
    _run(dev, rng, [1] * 40, 3000, False, 1.0)


def test_sample_rejects_bad_temperature(dev):
    x = torch.zeros(2, 8, device=dev)
    i = torch.zeros(2, dtype=torch.int32, device=dev)
    off = torch.tensor([0, 2], dtype=torch.int32, device=dev)
    u = torch.zeros(2, 2, device=dev)
    ws = tg.accept_sample_workspace(1, 2, dev)
    with pytest.raises(tg.TreeGraftError):
        tg.accept_sample(x, i, torch.tensor([-1, 0], dtype=torch.int32, device=dev), off, 2, 4,
                         u, 0.0, ws)


def test_sample_one_workspace_serves_any_shape(dev):
    """A workspace sized for a 24-tree batch serves a 3-tree batch next: its
    tickets then sit where the first call kept per-node flags, which the walk
    has returned to zero."""
    rng = synth.make_rng(977)
    sizes = rng.integers(20, 41, size=24).tolist()
    parent, token, off = _trees(rng, sizes, 1024, 10)
    ws = tg.accept_sample_workspace(len(sizes), len(parent), dev)
    for sz in (sizes, [5, 9, 3]):
        parent, token, off = _trees(rng, sz, 1024, 10)
        host = _logits(rng, parent, token, off, 1024, False, bump=12.0)
        u = rng.random((len(parent), 2)).astype(np.float32)
        path, alen, bonus = tg.accept_sample(_dev.f32(host, dev), _dev.i32(token, dev),
                                             _dev.i32(parent, dev), _dev.i32(off, dev), max(sz),
                                             12, _dev.f32(u, dev), 1.0, ws)
        torch.cuda.synchronize()
        assert tg.last_device_status() == 0
        assert not torch.any(ws != 0)
        op, oa, ob, info = S.accept_sample(host, token, parent, off, u, 1.0, 12, bf16=False)
        for b in range(len(sz)):
            if info[b]["margin"] > MARGIN:
                assert path[b].tolist() == op[b].tolist() and alen[b] == oa[b]
