"""Parity of the device grow step (treegraft_grow_step, Algorithm 2) with the
oracle's grow_step, step by step: before every device step the trees are
read back and the oracle applies the same step to that state, so every step
is checked on its own inputs.

Bars: a small step ranks stored fp32 scores, so its frontier, parents and
child tokens are bit-exact; child edges / scores within 1e-4 relative (they
hold a log-sum-exp).  A middle step rescores from a recomputed log-sum-exp,
so its rescored edges / scores and cached lse are compared within the same
tolerance and its frontier must be a valid Top_W of the pool under the
oracle's scores (equal to the oracle's frontier except where two scores are
within the tolerance); the children's parents and tokens are bit-exact for
the frontier the device chose."""
import numpy as np
import pytest
import torch

import paper_2608_26112_gb300 as tg
from oracle import treegraft_oracle as O
from paper_2608_26112_gb300 import synth
from tests import _dev

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-4, 1e-5


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26112_gb300 import build
    build.build()
    return torch.device("cuda:0")


def _tables(rng, B, cap, V, bf16, sigma=3.0):
    x = synth.normal_f32(rng, (B * cap, V), sigma)
    return synth.f32_to_bf16_bits(x) if bf16 else x


def _oracle_state(par, tok, edge, score, lse, n, new_lo, n_vis):
    return dict(parent=par[:n].tolist(), token=tok[:n].tolist(),
                edge=[np.float32(e) for e in edge[:n]], score=[np.float32(s) for s in score[:n]],
                new=list(range(new_lo, n)), P=set(range(n_vis)),
                lse_m={v: float(lse[v]) for v in range(n_vis)})


def _run_schedule(dev, sched, W, m, V, B, bf16, seed, root_scores=None):
    rng = synth.make_rng(seed)
    cap = 1
    c_lo, n_vis, nn = 0, 0, 1
    for a in sched:                       # capacity from the lock-step sizes
        pool = nn - (c_lo if a == 0 else n_vis)
        if a == 1:
            n_vis = nn
        c_lo, nn = nn, nn + min(W, pool) * m
    cap = nn
    small = _tables(rng, B, cap, V, bf16)
    middle = _tables(rng, B, cap, V, bf16)
    lg_small = _dev.bf16(small, dev) if bf16 else _dev.f32(small, dev)
    lg_middle = _dev.bf16(middle, dev) if bf16 else _dev.f32(middle, dev)
    parent = torch.full((B, cap), -1, dtype=torch.int32, device=dev)
    token = torch.zeros(B, cap, dtype=torch.int32, device=dev)
    edge = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    score = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    lse = torch.full((B, cap), float("nan"), dtype=torch.float32, device=dev)
    ws = tg.grow_workspace(B, cap, m, dev)
    n, new_lo, n_vis = 1, 0, 0
    for k, a in enumerate(sched):
        pool_lo = new_lo if a == 0 else n_vis
        snap = [t.cpu().numpy().copy() for t in (parent, token, edge, score, lse)]
        fr = tg.grow_step(a, lg_middle if a else lg_small, W, m, parent, token, edge, score, n,
                          pool_lo, lse_mid=lse, ws=ws)
        torch.cuda.synchronize()
        assert tg.last_device_status() == 0
        nf = min(W, n - pool_lo)
        n_next = n + nf * m
        got = [t.cpu().numpy() for t in (parent, token, edge, score, lse)]
        frs = fr.cpu().numpy()
        for b in range(B):
            st = _oracle_state(*(s[b] for s in snap), n, new_lo, n_vis)
            table_s = small[b * cap:(b + 1) * cap]
            table_m = middle[b * cap:(b + 1) * cap]
            F = O.grow_step(st, a, W, m, table_s, table_m, bf16=bf16)
            gF = frs[b][:nf].tolist()
            assert (frs[b][nf:] == -1).all()
            sc_o = np.asarray(st["score"][:n], np.float64)
            if a == 0:
                assert gF == F, (k, b)
            else:
                pool = list(range(pool_lo, n))
                # rescored pool: edges, scores, cached lse within tolerance
                np.testing.assert_allclose(got[3][b][pool_lo:n], sc_o[pool_lo:n], rtol=RTOL,
                                           atol=ATOL)
                np.testing.assert_allclose(got[2][b][max(pool_lo, 1):n],
                                           np.asarray(st["edge"][max(pool_lo, 1):n], np.float64),
                                           rtol=RTOL, atol=ATOL)
                np.testing.assert_allclose(got[4][b][pool_lo:n],
                                           [st["lse_m"][v] for v in pool], rtol=RTOL, atol=ATOL)
                # a valid Top_W under the oracle's scores, in the device's own order
                assert len(set(gF)) == nf and set(gF) <= set(pool)
                rest = [v for v in pool if v not in gF]
                tol = RTOL * max(1.0, float(np.abs(sc_o[pool]).max()))
                if rest:
                    assert min(sc_o[gF]) >= max(sc_o[rest]) - tol, (k, b)
                gs = got[3][b][gF]
                assert all(gs[i] >= gs[i + 1] for i in range(nf - 1))
                if gF != F:       # only near-ties may order differently
                    for x, y in zip(gF, F):
                        assert abs(sc_o[x] - sc_o[y]) <= tol, (k, b, gF, F)
            # children: the device's frontier expanded with the oracle's Top_m
            table = table_m if a else table_s
            for i, v in enumerate(gF):
                x, lse_v = O._row_log_softmax(table, v, bf16)
                top = np.lexsort((np.arange(V), -x))[:m]
                u = slice(n + i * m, n + (i + 1) * m)
                assert (got[0][b][u] == v).all()
                assert got[1][b][u].tolist() == top.tolist(), (k, b, v)
                lp = x[top] - lse_v
                np.testing.assert_allclose(got[2][b][u], lp, rtol=RTOL, atol=ATOL)
                np.testing.assert_allclose(got[3][b][u], float(got[3][b][v]) + lp, rtol=RTOL,
                                           atol=ATOL)
            # nodes outside the pool and the new children are untouched
            lo_keep = pool_lo if a else n
            assert (got[0][b][:n] == snap[0][b][:n]).all()
            assert (got[1][b][:n] == snap[1][b][:n]).all()
            assert (got[3][b][:lo_keep] == snap[3][b][:lo_keep]).all()
            assert (got[0][b][n_next:] == snap[0][b][n_next:]).all()
        if a == 1:
            n_vis = n
        new_lo, n = n, n_next
    return n


@pytest.mark.parametrize("bf16", [False, True])
@pytest.mark.parametrize("sched", [[0, 1, 0, 1, 0], [1, 0, 0, 1], [0, 0, 0], [1, 1, 0]])
def test_grow_step_schedules(dev, sched, bf16):
    n = _run_schedule(dev, sched, W=4, m=3, V=300, B=2, bf16=bf16, seed=500 + sum(sched))
    assert n > 1


def test_grow_step_paper_shape(dev):
    """Frontier W = 10 and branching m = 10 over D = 5 steps with the fixed
    schedule [1, 0, 1, 0, 1] of the paper's ablation, bf16 Llama-3 vocabulary
    rows (a 511-node tree by the last step)."""
    _run_schedule(dev, [1, 0, 1, 0, 1], W=10, m=10, V=128256, B=1, bf16=True, seed=510)


def test_grow_step_wide_frontier_and_single_child(dev):
    # W above the pool size (frontier padded with -1), one child per node
    _run_schedule(dev, [0, 1, 0, 1], W=50, m=1, V=64, B=3, bf16=False, seed=520)


def test_grow_step_ties_to_lower_ids(dev):
    """Quantised logits: many equal scores, so Top_W and Top_m ties decide
    (lower node id, lower token)."""
    rng = synth.make_rng(530)
    B, V, W, m = 1, 40, 3, 4
    sched = [0, 0, 1, 0]
    cap = 1 + 4 + 12 + 12 + 12 + 12
    q = rng.integers(-1, 2, size=(B * cap, V)).astype(np.float32)
    dev_q = _dev.f32(q, dev)
    parent = torch.full((B, cap), -1, dtype=torch.int32, device=dev)
    token = torch.zeros(B, cap, dtype=torch.int32, device=dev)
    edge = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    score = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    lse = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    st = O.grow_state()
    n, new_lo, n_vis = 1, 0, 0
    for a in sched:
        pool_lo = new_lo if a == 0 else n_vis
        fr = tg.grow_step(a, dev_q, W, m, parent, token, edge, score, n, pool_lo, lse_mid=lse)
        F = O.grow_step(st, a, W, m, q, q)
        nf = min(W, n - pool_lo)
        assert fr.cpu().numpy()[0][:nf].tolist() == F
        n_next = n + nf * m
        assert parent.cpu().numpy()[0][:n_next].tolist() == st["parent"]
        assert token.cpu().numpy()[0][:n_next].tolist() == st["token"]
        if a == 1:
            n_vis = n
        new_lo, n = n, n_next
    assert tg.last_device_status() == 0


def test_grow_step_malformed_tree_sets_status(dev):
    B, cap, V = 1, 16, 32
    q = torch.zeros(B * cap, V, dtype=torch.float32, device=dev)
    parent = torch.tensor([[-1, 0, 5, 1] + [-1] * 12], dtype=torch.int32, device=dev)  # 5 > 2
    token = torch.zeros(B, cap, dtype=torch.int32, device=dev)
    edge = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    score = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    lse = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    tg.last_device_status()
    tg.grow_step(1, q, 2, 2, parent, token, edge, score, 4, 0, lse_mid=lse)
    torch.cuda.synchronize()
    assert tg.last_device_status() & 4
