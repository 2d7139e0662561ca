"""Parity of the n-gram small drafter (treegraft_ngram_*) with the oracle's
n-gram drafter (oracle/ngram_oracle.py).

Bars: the prefill cache's tokens are bit-exact (top-m by exact logit order)
and its log-probabilities within 1e-4 relative; every lookup's matched
position and order are bit-exact (integer work); a draft's tokens and
log-probabilities are the device cache's row at that position, copied, and
its scores fp32(parent score + logprob) bit-exact; the grow step's frontier,
parents and tokens are bit-exact, its edges and scores within 1e-4 of the
oracle's (they hold the cached log-probabilities)."""
import numpy as np
import pytest
import torch

import paper_2608_26112_gb300 as tg
from oracle import ngram_oracle as NG
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


def _prompts(rng, lens, V, small_vocab=None):
    out = []
    for L in lens:
        if small_vocab:
            out.append(rng.integers(0, small_vocab, size=L).astype(np.int32))
        else:
            out.append(synth.prompt_stream(rng, L, V))
    return out


def _prefill(rng, prompts, V, bf16):
    """Packed prefill logits N(0, 3^2) with the next-token bump, as fp32
    values and as the device tensor (bf16 bits or fp32)."""
    rows = []
    for p in prompts:
        x = synth.normal_f32(rng, (len(p), V), 3.0)
        synth.plant_next_token_bump(rng, x, p)
        if bf16:                     # in blocks of rows: the rounding's temporaries stay small
            x = np.concatenate([synth.f32_to_bf16_bits(x[i:i + 128])
                                for i in range(0, len(x), 128)])
        rows.append(x)
    return np.concatenate(rows)


def _setup(dev, prompts, host_logits, bf16, max_n, m_cache):
    seq = np.concatenate([[0], np.cumsum([len(p) for p in prompts])]).astype(np.int32)
    toks = np.concatenate(prompts).astype(np.int32)
    lg = _dev.bf16(host_logits, dev) if bf16 else _dev.f32(host_logits, dev)
    index = tg.ngram_build(_dev.i32(toks, dev), _dev.i32(seq, dev), max_n)
    ctok, clp = tg.ngram_cache(lg, m_cache)
    torch.cuda.synchronize()
    assert tg.last_device_status() == 0
    return seq, index, ctok, clp


def _oracle_cache(host_logits, m_cache, bf16, rows=None):
    """The oracle's prefill cache at the given packed rows (all by default)."""
    if rows is None:
        return NG.prefill_cache(host_logits, m_cache, bf16=bf16)
    tok, lp, _, _ = O.expand_topk(host_logits, np.zeros(len(rows), np.float32), m_cache,
                                  row_idx=np.asarray(rows), bf16=bf16)
    return tok, lp


def _random_trees(rng, prompts, cap, vocab_extra):
    """Trees whose tokens are mostly prompt tokens (so suffixes match at
    several lengths), some unseen."""
    B = len(prompts)
    parent = np.full((B, cap), -1, np.int32)
    token = np.zeros((B, cap), np.int32)
    for b, p in enumerate(prompts):
        for v in range(1, cap):
            parent[b, v] = int(rng.integers(0, v))
            if rng.random() < 0.85:
                token[b, v] = p[int(rng.integers(0, len(p)))]
            else:
                token[b, v] = vocab_extra + int(rng.integers(0, 5))
    return parent, token


def _ctx(rng, prompts, max_n, full=False):
    B = len(prompts)
    ctx = np.zeros((B, max_n), np.int32)
    clen = np.zeros(B, np.int32)
    for b, p in enumerate(prompts):
        c = max_n if full else int(rng.integers(0, max_n + 1))
        e = int(rng.integers(min(c, len(p)), len(p) + 1))
        tail = p[max(0, e - c):e].tolist()
        tail = [int(p[0])] * (c - len(tail)) + tail
        ctx[b, :c] = tail
        clen[b] = c
    return ctx, clen


def _check_cache(ctok, clp, host_logits, m_cache, bf16, rows=None):
    g_tok, g_lp = ctok.cpu().numpy(), clp.cpu().numpy()
    if rows is not None:
        g_tok, g_lp = g_tok[rows], g_lp[rows]
    o_tok, o_lp = _oracle_cache(host_logits, m_cache, bf16, rows)
    assert (g_tok == o_tok).all()
    np.testing.assert_allclose(g_lp, o_lp, rtol=RTOL, atol=ATOL)


def _run_draft(dev, rng, prompts, host_logits, bf16, max_n, m_cache, m, cap):
    seq, index, ctok, clp = _setup(dev, prompts, host_logits, bf16, max_n, m_cache)
    _check_cache(ctok, clp, host_logits, m_cache, bf16)
    V = host_logits.shape[1]
    parent, token = _random_trees(rng, prompts, cap, V)
    ctx, clen = _ctx(rng, prompts, max_n)
    B = len(prompts)
    rows = np.arange(B * cap, dtype=np.int32)
    rng.shuffle(rows)
    ps = synth.normal_f32(rng, (B * cap,), 2.0)
    tok, lp, sc, pos, nn = tg.ngram_draft(index, ctok, clp, _dev.i32(ctx, dev), _dev.i32(clen, dev),
                                          _dev.i32(parent, dev), _dev.i32(token, dev),
                                          _dev.i32(rows, dev), _dev.f32(ps, dev), m,
                                          with_match=True)
    torch.cuda.synchronize()
    assert tg.last_device_status() == 0
    tok, lp, sc, pos, nn = (t.cpu().numpy() for t in (tok, lp, sc, pos, nn))
    g_tok, g_lp = ctok.cpu().numpy(), clp.cpu().numpy()
    orders = set()
    for r, node in enumerate(rows.tolist()):
        b, v = divmod(node, cap)
        q = NG.node_query(parent[b], token[b], v, ctx[b][:clen[b]].tolist(), max_n)
        j, n = NG.match(prompts[b], q, max_n)
        assert (pos[r], nn[r]) == (j, n), (b, v, q)
        orders.add(n)
        row = seq[b] + j
        assert tok[r].tolist() == g_tok[row][:m].tolist()
        assert (lp[r] == g_lp[row][:m]).all()
        assert (sc[r] == (np.float32(ps[r]) + g_lp[row][:m]).astype(np.float32)).all()
    return orders


@pytest.mark.parametrize("bf16", [False, True])
@pytest.mark.parametrize("max_n", [1, 3, 8])
def test_ngram_draft_matches_oracle(dev, bf16, max_n):
    """Ragged prompts (one of a single token), random trees, random context
    lengths (0 included): every row's match, tokens, logprobs and scores."""
    rng = synth.make_rng(800 + max_n + 10 * bf16)
    V = 300
    prompts = _prompts(rng, [1, 37, 300, 129], V)
    host = _prefill(rng, prompts, V, bf16)
    orders = _run_draft(dev, rng, prompts, host, bf16, max_n, m_cache=6, m=4, cap=40)
    assert 0 in orders and max(orders) >= min(2, max_n)


def test_ngram_draft_collisions_small_vocab(dev):
    """A three-token vocabulary: every n-gram recurs, so each table holds
    few keys with long runs of equal positions and the probes depend on the
    token comparison, not the hash, to tell keys apart."""
    rng = synth.make_rng(820)
    V = 16
    prompts = _prompts(rng, [3000, 2500], V, small_vocab=3)
    host = _prefill(rng, prompts, V, False)
    orders = _run_draft(dev, rng, prompts, host, False, 8, m_cache=3, m=3, cap=64)
    assert 8 in orders


def test_ngram_draft_many_prompts(dev):
    """64 prompts of 1..200 tokens in one index (equal n-grams across
    prompts must not match each other)."""
    rng = synth.make_rng(830)
    V = 64
    lens = rng.integers(1, 201, size=64).tolist()
    prompts = _prompts(rng, lens, V, small_vocab=8)
    host = _prefill(rng, prompts, V, False)
    _run_draft(dev, rng, prompts, host, False, 4, m_cache=2, m=2, cap=12)


def test_ngram_paper_shape(dev):
    """A 2048-token prompt with 128256-token bf16 prefill logits, top-10
    cache, max_n 4: the cache at 48 sampled rows against the oracle, every
    lookup of a 64-node tree bit-exact."""
    rng = synth.make_rng(840)
    V, L = synth.LLAMA3_VOCAB, 2048
    prompts = [synth.prompt_stream(rng, L, V)]
    host = _prefill(rng, prompts, V, True)
    max_n, m_cache = 4, 10
    seq, index, ctok, clp = _setup(dev, prompts, host, True, max_n, m_cache)
    rows = np.sort(rng.choice(L, size=48, replace=False))
    _check_cache(ctok, clp, host, m_cache, True, rows=rows)
    cap = 64
    parent, token = _random_trees(rng, prompts, cap, V - 10)
    ctx, clen = _ctx(rng, prompts, max_n, full=True)
    q_rows = np.arange(cap, dtype=np.int32)
    ps = np.zeros(cap, np.float32)
    _, _, _, pos, nn = tg.ngram_draft(index, ctok, clp, _dev.i32(ctx, dev), _dev.i32(clen, dev),
                                      _dev.i32(parent, dev), _dev.i32(token, dev),
                                      _dev.i32(q_rows, dev), _dev.f32(ps, dev), 10,
                                      with_match=True)
    torch.cuda.synchronize()
    assert tg.last_device_status() == 0
    pos, nn = pos.cpu().numpy(), nn.cpu().numpy()
    for v in range(cap):
        q = NG.node_query(parent[0], token[0], v, ctx[0].tolist(), max_n)
        assert (pos[v], nn[v]) == NG.match(prompts[0], q, max_n), v


def _grow_check(dev, rng, prompts, host, bf16, max_n, m_cache, W, m, steps, ctx_full=True):
    """Small steps of Algorithm 2 with the n-gram drafter on all trees at
    once; before every device step the trees are read back and the oracle
    applies the same step to that state with its own cache."""
    seq, index, ctok, clp = _setup(dev, prompts, host, bf16, max_n, m_cache)
    B = len(prompts)
    o_tok, o_lp = _oracle_cache(host, m_cache, bf16)
    ctx, clen = _ctx(rng, prompts, max_n, full=ctx_full)
    cap, nn_, lo_ = 1, 1, 0
    for _ in range(steps):
        cap = nn_ + min(W, nn_ - lo_) * m
        lo_, nn_ = nn_, cap
    parent = torch.full((B, cap), -1, dtype=torch.int32, device=dev)
    token = torch.zeros(B, cap, dtype=torch.int32, device=dev)
    edge = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    score = torch.zeros(B, cap, dtype=torch.float32, device=dev)
    d_ctx, d_clen = _dev.i32(ctx, dev), _dev.i32(clen, dev)
    n, lo = 1, 0
    for k in range(steps):
        snap = [t.cpu().numpy().copy() for t in (parent, token, edge, score)]
        fr = tg.ngram_grow_step(index, ctok, clp, d_ctx, d_clen, W, m, parent, token, edge, score,
                                n, lo)
        torch.cuda.synchronize()
        assert tg.last_device_status() == 0
        nf = min(W, n - lo)
        n_next = n + nf * m
        got = [t.cpu().numpy() for t in (parent, token, edge, score)]
        frs = fr.cpu().numpy()
        for b in range(B):
            st = dict(parent=snap[0][b][:n].tolist(), token=snap[1][b][:n].tolist(),
                      edge=[np.float32(e) for e in snap[2][b][:n]],
                      score=[np.float32(x) for x in snap[3][b][:n]],
                      new=list(range(lo, n)), P=set(), lse_m={})
            a, e = int(seq[b]), int(seq[b + 1])
            small = NG.small_drafter(prompts[b], o_tok[a:e], o_lp[a:e], ctx[b][:clen[b]].tolist(),
                                     max_n)
            F = O.grow_step(st, 0, W, m, None, None, small_draft=small)
            assert frs[b][:nf].tolist() == F, (k, b)
            assert (frs[b][nf:] == -1).all()
            assert got[0][b][:n_next].tolist() == st["parent"]
            assert got[1][b][:n_next].tolist() == st["token"], (k, b)
            np.testing.assert_allclose(got[2][b][n:n_next], np.asarray(st["edge"][n:], np.float64),
                                       rtol=RTOL, atol=ATOL)
            np.testing.assert_allclose(got[3][b][n:n_next],
                                       np.asarray(st["score"][n:], np.float64), rtol=RTOL,
                                       atol=ATOL)
            assert (got[3][b][:n] == snap[3][b][:n]).all()          # nothing rewritten
            assert (got[0][b][n_next:] == snap[0][b][n_next:]).all()
        lo, n = n, n_next
    return got


@pytest.mark.parametrize("bf16", [False, True])
def test_ngram_grow_steps_match_oracle(dev, bf16):
    rng = synth.make_rng(850 + bf16)
    V = 400
    prompts = _prompts(rng, [500, 64, 1, 230], V)
    host = _prefill(rng, prompts, V, bf16)
    _grow_check(dev, rng, prompts, host, bf16, max_n=4, m_cache=5, W=4, m=3, steps=5)


def test_ngram_grow_paper_shape(dev):
    """W = m = 10 over D = 5 small steps from the root (1 + 10 + 4 * 100 =
    411 nodes), a 512-token prompt, 128256-token bf16 prefill, max_n 4."""
    rng = synth.make_rng(860)
    V = synth.LLAMA3_VOCAB
    prompts = [synth.prompt_stream(rng, 512, V)]
    host = _prefill(rng, prompts, V, True)
    _grow_check(dev, rng, prompts, host, True, max_n=4, m_cache=10, W=10, m=10, steps=5)


def test_ngram_grow_chain_copies_the_prompt(dev):
    """W = m = 1 with a context cut from a prompt whose 3-grams are unique
    and whose cache predicts the next token: the chain drafted on the device
    is the prompt's own continuation."""
    rng = synth.make_rng(870)
    V, L = 40, 48
    while True:
        p = rng.integers(0, V, size=L).astype(np.int32)
        if len({tuple(p[j:j + 3]) for j in range(L - 2)}) == L - 2:
            break
    x = synth.normal_f32(rng, (L, V), 1.0)
    for j in range(L - 1):
        x[j, p[j + 1]] += np.float32(12.0)
    seq, index, ctok, clp = _setup(dev, [p], x, False, 3, 2)
    k, D = 10, 8
    ctx = _dev.i32(p[k - 3:k].reshape(1, 3), dev)
    clen = _dev.i32(np.array([3]), dev)
    parent = torch.full((1, D + 1), -1, dtype=torch.int32, device=dev)
    token = torch.zeros(1, D + 1, dtype=torch.int32, device=dev)
    edge = torch.zeros(1, D + 1, dtype=torch.float32, device=dev)
    score = torch.zeros(1, D + 1, dtype=torch.float32, device=dev)
    for i in range(D):
        tg.ngram_grow_step(index, ctok, clp, ctx, clen, 1, 1, parent, token, edge, score, i + 1,
                           i)
    torch.cuda.synchronize()
    assert tg.last_device_status() == 0
    assert parent.cpu().numpy()[0].tolist() == [-1] + list(range(D))
    assert token.cpu().numpy()[0][1:].tolist() == p[k:k + D].tolist()


def test_ngram_device_errors_set_status(dev):
    """A malformed seq_off, a row outside the trees, a context length above
    max_n and a malformed tree each raise their status bit."""
    rng = synth.make_rng(880)
    p = rng.integers(0, 5, size=20).astype(np.int32)
    tg.last_device_status()
    tg.ngram_build(_dev.i32(p, dev), _dev.i32(np.array([0, 12, 9]), dev), 3)
    assert tg.last_device_status() & 16
    x = synth.normal_f32(rng, (20, 8), 1.0)
    seq, index, ctok, clp = _setup(dev, [p[:12], p[12:]], x, False, 3, 2)
    parent = _dev.i32(np.array([[-1, 0, 1, 1], [-1, 0, 3, 0]]), dev)   # tree 1: 3 > 2
    token = _dev.i32(np.zeros((2, 4)), dev)
    ctx = _dev.i32(np.zeros((2, 3)), dev)
    ps = _dev.f32(np.zeros(1), dev)
    ok_len = _dev.i32(np.array([2, 2]), dev)
    tg.ngram_draft(index, ctok, clp, ctx, ok_len, parent, token, _dev.i32(np.array([9]), dev),
                   ps, 2)
    assert tg.last_device_status() & 16
    tg.ngram_draft(index, ctok, clp, ctx, _dev.i32(np.array([4, 2]), dev), parent, token,
                   _dev.i32(np.array([3]), dev), ps, 2)
    assert tg.last_device_status() & 16
    tg.ngram_draft(index, ctok, clp, ctx, ok_len, parent, token, _dev.i32(np.array([6]), dev),
                   ps, 2)
    assert tg.last_device_status() & 4
    tg.ngram_draft(index, ctok, clp, ctx, ok_len, parent, token, _dev.i32(np.array([3]), dev),
                   ps, 2)
    assert tg.last_device_status() == 0
