"""Pins of the n-gram small drafter's oracle (oracle/ngram_oracle.py) against
what its definition fixes, independently of the oracle's own code: cases
worked out by hand, a second formulation of the longest-suffix match (the
longest common suffix at every prompt position, taken with numpy), the
invariants of a match, a bincount statement of the fallback, and a copy
chain whose drafted tokens are known in closed form."""
import numpy as np
import pytest
from scipy.special import logsumexp

from oracle import ngram_oracle as NG
from oracle import treegraft_oracle as O
from paper_2608_26112_gb300 import synth

#              0  1  2  3  4  5  6  7  8  9  10
HAND_PROMPT = [5, 1, 2, 3, 1, 2, 4, 1, 2, 3, 7]


@pytest.mark.parametrize("query,max_n,want", [
    ([1, 2], 4, (8, 2)),            # (1,2) ends at 2, 5, 8: latest
    ([9, 1, 2, 3], 4, (9, 3)),      # (9,1,2,3) absent; (1,2,3) ends at 3, 9
    ([2, 4], 4, (6, 2)),
    ([3, 3], 4, (9, 1)),            # (3,3) absent; (3) ends at 3, 9
    ([1, 2, 3], 1, (9, 1)),         # max_n 1: only the last token
    ([4, 1, 2, 3], 4, (9, 4)),      # the whole 4-gram at 6..9
    ([8], 4, (7, 0)),               # absent: 1 and 2 occur 3 times, 1 wins, last at 7
    ([5], 3, (0, 1)),               # an n-gram at the very start
    ([3, 7], 2, (10, 2)),           # ... and at the very end
])
def test_match_hand_cases(query, max_n, want):
    assert NG.match(HAND_PROMPT, query, max_n) == want


def test_fallback_hand_cases():
    assert NG.most_frequent_position([4, 4, 2, 2, 9]) == 3     # tie 2 / 4 -> token 2
    assert NG.most_frequent_position([7]) == 0
    assert NG.most_frequent_position([3, 1, 3, 1, 1]) == 4


def _lcs_formulation(prompt, query, max_n):
    """The match as one maximum: the common suffix length of the query and
    the prompt prefix ending at j, capped at max_n, maximised over j (latest
    j among the maxima); numpy throughout."""
    p = np.asarray(prompt, np.int64)
    q = np.asarray(query, np.int64)[-max_n:]
    L, n = len(p), len(q)
    run = np.zeros(L, np.int64)          # run[j] = common suffix length at j
    alive = np.ones(L, bool)
    for i in range(n):                   # compare p[j - i] with q[n - 1 - i]
        js = np.arange(L) - i
        ok = (js >= 0) & alive
        ok[ok] = p[js[ok]] == q[n - 1 - i]
        alive = ok
        run += alive
    best = run.max() if L else 0
    if best == 0:
        counts = np.bincount(p)
        tok = int(np.argmax(counts))     # argmax: first (lowest) token among ties
        return int(np.flatnonzero(p == tok)[-1]), 0
    return int(np.flatnonzero(run == best)[-1]), int(best)


@pytest.mark.parametrize("seed", range(6))
def test_match_equals_longest_common_suffix(seed):
    rng = synth.make_rng(700 + seed)
    V = 4 + seed                          # small vocabularies: many partial matches
    prompt = rng.integers(0, V, size=60).tolist()
    for _ in range(80):
        ql = int(rng.integers(1, 9))
        if rng.random() < 0.5:            # half of the queries are cut from the prompt
            e = int(rng.integers(ql, len(prompt) + 1))
            query = prompt[e - ql:e]
            query[0] = int(rng.integers(0, V + 2))
        else:
            query = rng.integers(0, V + 2, size=ql).tolist()
        max_n = int(rng.integers(1, 7))
        assert NG.match(prompt, query, max_n) == _lcs_formulation(prompt, query, max_n)


@pytest.mark.parametrize("seed", range(3))
def test_match_invariants(seed):
    rng = synth.make_rng(720 + seed)
    prompt = rng.integers(0, 5, size=40).tolist()
    for _ in range(50):
        query = rng.integers(0, 6, size=int(rng.integers(1, 7))).tolist()
        max_n = int(rng.integers(1, 6))
        j, n = NG.match(prompt, query, max_n)
        q = query[-max_n:]
        if n == 0:
            continue
        assert prompt[j - n + 1:j + 1] == q[len(q) - n:]          # it is a match
        g = q[len(q) - n:]
        later = [k for k in range(j + 1, len(prompt)) if k >= n - 1 and prompt[k - n + 1:k + 1] == g]
        assert not later                                         # the latest one
        if n < len(q):                                           # nothing longer occurs
            g1 = q[len(q) - n - 1:]
            assert not any(prompt[k - n:k + 1] == g1 for k in range(n, len(prompt)))


def test_node_query_reads_path_then_context():
    # root 0; 1, 2 children of 0; 3 child of 1; 4 child of 3
    parent = [-1, 0, 0, 1, 3]
    token = [99, 11, 12, 13, 14]          # the root's token is not read
    ctx = [1, 2, 3]
    assert NG.node_query(parent, token, 4, ctx, 8) == [1, 2, 3, 11, 13, 14]
    assert NG.node_query(parent, token, 4, ctx, 4) == [3, 11, 13, 14]
    assert NG.node_query(parent, token, 2, ctx, 2) == [3, 12]
    assert NG.node_query(parent, token, 0, ctx, 2) == [2, 3]


def test_prefill_cache_is_top_m_log_softmax():
    rng = synth.make_rng(730)
    x = rng.normal(0, 3, size=(7, 50)).astype(np.float32)
    x[2, 5] = x[2, 9] = x[2].max() + 1.0          # a tie: token 5 first
    tok, lp = NG.prefill_cache(x, 4)
    for r in range(7):
        order = np.argsort(-x[r].astype(np.float64), kind="stable")[:4]
        assert tok[r].tolist() == order.tolist()
        lse = logsumexp(x[r].astype(np.float64))
        np.testing.assert_allclose(lp[r], x[r][order] - lse, rtol=1e-6)
    assert tok[2][:2].tolist() == [5, 9]


def test_draft_reads_the_matched_row():
    cache_tok = np.arange(11 * 3, dtype=np.int32).reshape(11, 3)
    cache_lp = -np.arange(11 * 3, dtype=np.float32).reshape(11, 3)
    tok, lp, j, n = NG.draft(HAND_PROMPT, cache_tok, cache_lp, [2, 4], 4, 2)
    assert (j, n) == (6, 2) and tok == [18, 19] and lp == [-18.0, -19.0]


def _copy_setup(rng, L=48, V=40, bump=12.0):
    """A prompt with no repeated 3-gram, and prefill logits whose top-1 at
    position j is the prompt's next token x[j + 1]."""
    while True:
        prompt = rng.integers(0, V, size=L).tolist()
        grams = [tuple(prompt[j:j + 3]) for j in range(L - 2)]
        if len(set(grams)) == len(grams):
            break
    logits = rng.normal(0, 1, size=(L, V)).astype(np.float32)
    for j in range(L - 1):
        logits[j, prompt[j + 1]] += bump
    return prompt, logits


def test_grow_chain_copies_the_prompt():
    """W = m = 1 small steps from a context equal to a prompt prefix: with
    unique 3-grams and a top-1 cache that predicts the next prompt token, the
    drafted chain is the prompt's own continuation, token for token."""
    rng = synth.make_rng(740)
    prompt, logits = _copy_setup(rng)
    tok_c, lp_c = NG.prefill_cache(logits, 2)
    k, D = 10, 8
    ctx = prompt[k - 3:k]
    st = O.grow_state()
    small = NG.small_drafter(prompt, tok_c, lp_c, ctx, 3)
    for _ in range(D):
        O.grow_step(st, 0, 1, 1, None, None, small_draft=small)
    assert st["parent"] == [-1] + list(range(D))
    assert st["token"][1:] == prompt[k:k + D]
    s = np.float32(0.0)
    for i in range(1, D + 1):                  # path score = fp32 running sum
        s = np.float32(s + lp_c[k - 1 + i - 1][0])
        assert st["score"][i] == s


def test_grow_step_with_small_drafter_branches():
    """A small step with W = 2, m = 2 on a hand tree: the frontier is Top_W of
    the new nodes and each gets the first two cached candidates at its own
    match."""
    prompt = HAND_PROMPT
    cache_tok = np.arange(11 * 3, dtype=np.int32).reshape(11, 3) + 100
    cache_lp = -(np.arange(11 * 3, dtype=np.float32).reshape(11, 3) + 1) / 8
    st = dict(parent=[-1, 0, 0, 0], token=[0, 2, 4, 9],
              edge=[np.float32(0), np.float32(-1), np.float32(-0.5), np.float32(-2)],
              score=[np.float32(0), np.float32(-1), np.float32(-0.5), np.float32(-2)],
              new=[1, 2, 3], P=set(), lse_m={})
    ctx = [3, 1]
    F = O.grow_step(st, 0, 2, 2, None, None,
                    small_draft=NG.small_drafter(prompt, cache_tok, cache_lp, ctx, 3))
    assert F == [2, 1]
    # node 2: query (3, 1, 4) -> (1, 4)? absent; (4) at 6 -> row 6
    # node 1: query (3, 1, 2) -> the whole 3-gram at 3..5 -> row 5
    assert st["parent"][4:] == [2, 2, 1, 1]
    assert st["token"][4:] == [118, 119, 115, 116]
    assert st["score"][4] == np.float32(np.float32(-0.5) + cache_lp[6][0])
