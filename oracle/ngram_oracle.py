"""CPU oracle for TreeGraft's n-gram small drafter (test infrastructure only).

A plain, slow statement of the training-free lookup drafter that TreeGraft
uses as its small drafter (Appendix, "n-gram small drafter"): at prefill the
target's top-m next-token candidates and their log-probabilities are cached
at every prompt position; at a small-drafter step the suffix of the current
prefix is matched against the prompt with the longest n-gram that occurs,
shortening it one token at a time, and the cached candidates of the matched
position become the expansion's children with their cached log-probabilities
as edge scores.  With no match at any length the candidates of the position
of the prompt's most frequent token are used.  Only the test-suite, the
package smoke check and the benchmark's CPU-baseline leg may import it; the
product path never calls it.  It shares no code with the CUDA library (no
hashing, no index: every lookup scans the prompt).

Every function is pinned by tests/test_oracle_ngram.py (hand-derived cases,
an independent longest-common-suffix formulation, invariants, a copy chain
whose drafted tokens are known in closed form).  Parity status: prefill_cache,
most_frequent_position, match, node_query, draft, small_drafter: pinned.

Readings taken where the paper is silent:
  * the index covers the prompt positions only (the only positions with
    cached candidates); an n-gram match must lie wholly inside the prompt;
  * an n-gram that occurs several times matches at its latest occurrence;
  * the longest order tried is a parameter max_n; a query shorter than max_n
    starts at its own length;
  * the current prefix at tree node v is the committed text (its last token
    is the root's) followed by the tokens of the non-root nodes on the path
    root -> v;
  * the most frequent prompt token breaks count ties to the lower token id
    and is used at its latest position;
  * the cache holds the top-m_cache tokens by (logit desc, token asc) with
    logprob = fp32(l - lse); an expansion takes the first m <= m_cache of
    them, score = fp32(s(v) + logprob).
"""
from __future__ import annotations

import numpy as np

from oracle import treegraft_oracle as T


def prefill_cache(logits, m: int, *, bf16: bool = False):
    """Top-m candidates and their log-probabilities at every prefill row:
    tok int32 [rows, m] by (logit desc, token asc), logprob f32 [rows, m]."""
    rows = len(logits)
    tok, lp, _, _ = T.expand_topk(logits, np.zeros(rows, np.float32), m, bf16=bf16)
    return tok, lp


def most_frequent_position(prompt) -> int:
    """Latest position of the prompt's most frequent token (count ties go to
    the lower token id)."""
    counts = {}
    for t in prompt:
        counts[int(t)] = counts.get(int(t), 0) + 1
    best = min(counts, key=lambda t: (-counts[t], t))
    return max(j for j, t in enumerate(prompt) if int(t) == best)


def match(prompt, query, max_n: int):
    """(position j, order n) of the longest suffix of `query` (at most max_n
    tokens) that ends somewhere in the prompt, at its latest end position j;
    shorter suffixes are tried only when a longer one has no occurrence.
    With no occurrence at any length: (most_frequent_position, 0)."""
    prompt = [int(t) for t in prompt]
    query = [int(t) for t in query]
    for n in range(min(max_n, len(query)), 0, -1):
        gram = query[len(query) - n:]
        hits = [j for j in range(n - 1, len(prompt)) if prompt[j - n + 1:j + 1] == gram]
        if hits:
            return max(hits), n
    return most_frequent_position(prompt), 0


def node_query(parent, token, v: int, ctx, max_n: int) -> list[int]:
    """The last max_n tokens of the prefix at node v: the committed context
    `ctx` (ending with the root's token) followed by the tokens of the
    non-root nodes on the path root -> v."""
    path = []
    w = v
    while w != 0:
        path.append(int(token[w]))
        w = int(parent[w])
    seq = [int(t) for t in ctx] + path[::-1]
    return seq[-max_n:]


def draft(prompt, cache_tok, cache_lp, query, max_n: int, m: int):
    """The small drafter's expansion for one query: the first m cached
    candidates (tokens, log-probabilities) at the matched position, with the
    position and order of the match."""
    j, n = match(prompt, query, max_n)
    return [int(t) for t in cache_tok[j][:m]], [np.float32(x) for x in cache_lp[j][:m]], j, n


def small_drafter(prompt, cache_tok, cache_lp, ctx, max_n: int):
    """A small-drafter callable for treegraft_oracle.grow_step: children of
    frontier node v as (tokens, log-probabilities) from the n-gram lookup on
    the prefix at v."""
    def expand(state, v: int, m: int):
        q = node_query(state["parent"], state["token"], v, ctx, max_n)
        tok, lp, _, _ = draft(prompt, cache_tok, cache_lp, q, max_n, m)
        return tok, lp
    return expand
