"""Pins of the stochastic-verification oracle (oracle/sample_oracle.py)
against what the rule fixes independently of the oracle's code: hand-worked
walks, the bonus draw against numpy's searchsorted on the cumulative
probabilities, the T -> 0 limit against the greedy oracle, and the
distribution of the emitted tokens (each must follow the target's
next-token distribution) by Monte Carlo."""
import numpy as np
import pytest

from oracle import sample_oracle as S
from oracle import treegraft_oracle as O
from paper_2608_26112_gb300 import synth


def _logits_for(p, T=1.0):
    """A logit row whose softmax at temperature T is p."""
    return (np.log(np.asarray(p, np.float64)) * T).astype(np.float64)


def _walk(rows, token, parent, u, T=1.0):
    lg = np.asarray(rows, np.float64)
    node_off = np.array([0, len(parent)], np.int32)
    u = np.asarray(u, np.float32)
    return S.accept_sample(lg, np.asarray(token), np.asarray(parent), node_off, u, T, 8)


P_ROOT = [0.5, 0.3, 0.2]


@pytest.mark.parametrize("u1,u2,want_path,want_bonus", [
    (0.40, 0.9, [0, 1], None),      # 0.40 < 0.5: child 1 (token 0) accepted
    (0.60, 0.50, [0, 2], None),     # child 1 rejected; R = 0.5, 0.25 < 0.3: child 2 accepted
    (0.60, 0.70, [0], 2),           # both rejected: the residual is all on token 2
])
def test_hand_walks(u1, u2, want_path, want_bonus):
    # root (children 1: token 0, 2: token 1); rows 1, 2 are leaves
    rows = [_logits_for(P_ROOT), _logits_for([0.1, 0.1, 0.8]), _logits_for([0.6, 0.2, 0.2])]
    u = [[0.0, 0.0], [u1, 0.05], [u2, 0.05]]
    path, alen, bonus, info = _walk(rows, [9, 0, 1], [-1, 0, 0], u)
    assert path[0][:len(want_path)].tolist() == want_path
    assert alen[0] == len(want_path) - 1
    if want_bonus is not None:
        assert bonus[0] == want_bonus
    else:   # bonus from the accepted leaf's row with u = 0.05: its first token
        assert bonus[0] == 0


def test_duplicate_sibling_is_never_accepted():
    # children 1 and 2 carry the same token 0; once 1 is rejected, 2 has no mass
    rows = [_logits_for(P_ROOT), _logits_for([1 / 3] * 3), _logits_for([1 / 3] * 3)]
    path, alen, bonus, _ = _walk(rows, [9, 0, 0], [-1, 0, 0], [[0, 0], [0.9, 0], [0.0, 0]])
    assert alen[0] == 0
    # residual (0, 0.3, 0.2) / 0.5 drawn at u = 0: token 1
    assert bonus[0] == 1


@pytest.mark.parametrize("T", [0.5, 1.0, 2.0])
def test_bonus_draw_is_inversion(T):
    rng = synth.make_rng(900)
    x = rng.normal(0, 3, size=(1, 50))
    p = np.exp((x[0] - x[0].max()) / T)
    p /= p.sum()
    cum = np.cumsum(p)
    for uu in rng.random(200):
        u = np.array([[0.0, uu]], np.float32)
        _, _, bonus, _ = S.accept_sample(x, np.array([0]), np.array([-1]), np.array([0, 1]), u,
                                         T, 4)
        assert bonus[0] == int(np.searchsorted(cum, float(np.float32(uu)), side="right"))


def test_small_temperature_is_greedy():
    rng = synth.make_rng(910)
    for seed in range(5):
        r = synth.make_rng(920 + seed)
        parent = synth.sample_tree(r, 30, 5, cap=4)
        V = 64
        token = r.integers(0, V, size=30).astype(np.int32)
        lg = synth.normal_f32(r, (30, V), 3.0)
        synth.plant_child_bump(r, lg, parent, token, np.arange(30), prob=0.8)
        off = np.array([0, 30], np.int32)
        u = rng.random((30, 2)).astype(np.float32) * np.float32(0.999)
        gp, ga, gb = O.accept(lg, token, parent, off, 12)
        sp, sa, sb, _ = S.accept_sample(lg, token, parent, off, u, 1e-3, 12)
        assert (gp == sp).all() and (ga == sa).all() and (gb == sb).all()


def test_emitted_tokens_follow_the_target():
    """Monte Carlo over the uniforms: the first emitted token (an accepted
    child's token or the bonus) follows p(.|root); given that it is child
    c's token, the next one follows p(.|c).  A duplicate sibling and a
    grandchild make every branch of the rule count."""
    V = 5
    rng = synth.make_rng(930)
    p_root = [0.35, 0.25, 0.2, 0.15, 0.05]
    #        node: 0 root, 1 tok 0, 2 tok 2, 3 tok 0 (duplicate of 1), 4 tok 3 under 1
    parent = np.array([-1, 0, 0, 0, 1])
    token = np.array([0, 0, 2, 0, 3])
    p1 = [0.1, 0.2, 0.3, 0.25, 0.15]
    rows = [_logits_for(p_root), _logits_for(p1), _logits_for([0.2] * 5),
            _logits_for([0.2] * 5), _logits_for([0.4, 0.3, 0.1, 0.1, 0.1])]
    lg = np.asarray(rows)
    off = np.array([0, 5], np.int32)
    N = 30000
    first = np.zeros(V)
    second = np.zeros(V)
    for _ in range(N):
        u = rng.random((5, 2)).astype(np.float32)
        path, alen, bonus, _ = S.accept_sample(lg, token, parent, off, u, 1.0, 4)
        seq = [int(token[v]) for v in path[0][1:alen[0] + 1]] + [int(bonus[0])]
        first[seq[0]] += 1
        if seq[0] == 0:                                  # came through node 1
            second[seq[1]] += 1
    for f, pr, n_eff in ((first / N, p_root, N), (second / first[0], p1, first[0])):
        sd = np.sqrt(np.asarray(pr) * (1 - np.asarray(pr)) / n_eff)
        assert (np.abs(f - pr) <= 5 * sd + 1e-9).all(), (f, pr)
