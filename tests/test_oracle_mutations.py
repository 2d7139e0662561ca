"""The oracle pins catch plausible mistakes in the oracle.

Each case plants one mistake in an in-memory copy of an oracle module: a
dropped term, a wrong index, sign or tie rule, a transposed operand, an
off-by-one.  The case points the pin tests (tests/test_oracle_pins.py,
test_oracle_sample.py, test_oracle_ngram.py) at that copy and runs them with
every parametrisation; the oracle modules built on the mutated one see the
copy too.  At least one pin must fail.  The oracle files are
only read, never modified.  CPU only."""
import inspect
import os
import types

import pytest

from oracle import ngram_oracle, sample_oracle
from tests import test_oracle_ngram, test_oracle_pins, test_oracle_sample

ORACLE_DIR = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle")

PIN_MODULES = (test_oracle_pins, test_oracle_sample, test_oracle_ngram)

# oracle module -> every (module, global name) through which it is used: the
# pin modules and the oracle modules built on it
USES = {
    "treegraft_oracle": ((test_oracle_pins, "O"), (test_oracle_sample, "O"),
                         (test_oracle_ngram, "O"), (sample_oracle, "O"), (ngram_oracle, "T")),
    "sample_oracle": ((test_oracle_sample, "S"),),
    "ngram_oracle": ((test_oracle_ngram, "NG"),),
}

# id: (oracle module, exact text, replacement)
MUTATIONS = {
    # Algorithm 3 mask and depth
    "mask-drops-self": ("treegraft_oracle", "        v = u\n        while v != -1:",
                        "        v = int(parent[u])\n        while v != -1:"),
    "depth-off-by-one": ("treegraft_oracle", "        d[u] = k\n", "        d[u] = k + 1\n"),
    "tree-check-allows-self-parent": ("treegraft_oracle", "if not (0 <= parent[i] < i):",
                                      "if not (0 <= parent[i] <= i):"),
    "attn-lse-base-2": ("treegraft_oracle", "lse[a:e, h] = (m + np.log(l))[:, 0]",
                        "lse[a:e, h] = (m + np.log2(l))[:, 0]"),
    "topk-ignores-row-idx": ("treegraft_oracle",
                             "r = int(row_idx[i]) if row_idx is not None else i", "r = i"),
    "prune-adds-partial-chains": ("treegraft_oracle",
                                  "                if len(K) + len(chain) <= M:\n"
                                  "                    K.update(chain)\n",
                                  "                K.update(chain[:M - len(K)])\n"),
    "grow-middle-lse-of-own-row": ("treegraft_oracle",
                                   "edge[v] = np.float32(row[token[v]] - lse_m[parent[v]])",
                                   "edge[v] = np.float32(row[token[v]] - lse_m[v])"),
    "bf16-decode-no-shift": ("treegraft_oracle",
                             "b = np.ascontiguousarray(bits).view(np.uint16).astype(np.uint32) << 16",
                             "b = np.ascontiguousarray(bits).view(np.uint16).astype(np.uint32)"),
    "argmax-ties-to-higher-token": ("treegraft_oracle",
                                    "np.array([int(np.argmax(_row_values(target_logits, r, bf16))) for r in rows],",
                                    "np.array([len(_row_values(target_logits, r, bf16)) - 1 - int(np.argmax("
                                    "_row_values(target_logits, r, bf16)[::-1])) for r in rows],"),
    # tree attention
    "attn-scale-1/D": ("treegraft_oracle", "scale = 1.0 / np.sqrt(D)", "scale = 1.0 / D"),
    "attn-gqa-modulo": ("treegraft_oracle", "kv = h // G", "kv = h % Hkv"),
    "attn-no-mask": ("treegraft_oracle", "s[~allowed] = NEG_INF", "s[~allowed] = s[~allowed]"),
    "attn-mask-transposed": ("treegraft_oracle", "ancestor_mask(parent[a:e])], axis=1)",
                             "ancestor_mask(parent[a:e]).T], axis=1)"),
    "attn-lse-drops-max": ("treegraft_oracle", "lse[a:e, h] = (m + np.log(l))[:, 0]",
                           "lse[a:e, h] = np.log(l)[:, 0]"),
    "attn-values-from-keys": ("treegraft_oracle", "Vv = v_cache[b, kv, :P + n]",
                              "Vv = k_cache[b, kv, :P + n]"),
    # expand_topk
    "topk-ties-to-higher-token": ("treegraft_oracle",
                                  "order = np.lexsort((np.arange(V), -x))[:k]",
                                  "order = np.lexsort((-np.arange(V), -x))[:k]"),
    "topk-lse-drops-max": ("treegraft_oracle", "lse[i] = m + np.log(np.exp(x - m).sum())",
                           "lse[i] = np.log(np.exp(x - m).sum())"),
    "topk-score-subtracts": ("treegraft_oracle",
                             "sc[i] = (float(np.float32(parent_score[i])) + (x[order] - lse[i]))",
                             "sc[i] = (float(np.float32(parent_score[i])) - (x[order] - lse[i]))"),
    "topk-logprob-sign": ("treegraft_oracle", "lp[i] = (x[order] - lse[i]).astype(np.float32)",
                          "lp[i] = (lse[i] - x[order]).astype(np.float32)"),
    # rescore_select
    "rescore-own-row": ("treegraft_oracle",
                        "strong_lp[a + int(parent[a + v]), int(token[a + v])]",
                        "strong_lp[a + v, int(token[a + v])]"),
    "rescore-visited-inverted": ("treegraft_oracle", "            if visited[a + v]:\n",
                                 "            if not visited[a + v]:\n"),
    "rescore-sum-previous-index": ("treegraft_oracle",
                                   "score[a + v] = np.float32(score[a + int(parent[a + v])])",
                                   "score[a + v] = np.float32(score[a + v - 1])"),
    "rescore-ties-to-higher-id": ("treegraft_oracle",
                                  "cand.sort(key=lambda v: (-float(score[a + v]), v))",
                                  "cand.sort(key=lambda v: (-float(score[a + v]), -v))"),
    "rescore-visited-candidates": ("treegraft_oracle",
                                   "cand = [v for v in range(e - a) if not visited[a + v]]",
                                   "cand = [v for v in range(e - a)]"),
    # accept
    "accept-own-row": ("treegraft_oracle", "int(token[a + w]) == am[int(par[w])]",
                       "int(token[a + w]) == am[w]"),
    "accept-ties-to-higher-id": ("treegraft_oracle", "key = (len(chain) - 1, -v)",
                                 "key = (len(chain) - 1, v)"),
    "accept-bonus-from-root": ("treegraft_oracle", "bonus[b] = am[chain[-1]]",
                               "bonus[b] = am[chain[0]]"),
    "accept-length-counts-root": ("treegraft_oracle", "alen[b] = len(chain) - 1",
                                  "alen[b] = len(chain)"),
    # GlobalPrune
    "prune-ties-deeper-first": ("treegraft_oracle", "key=lambda v: (-s[v], int(d[v]), v))",
                                "key=lambda v: (-s[v], -int(d[v]), v))"),
    "prune-lowest-scores": ("treegraft_oracle", "key=lambda v: (-s[v], int(d[v]), v))",
                            "key=lambda v: (s[v], int(d[v]), v))"),
    "prune-budget-off-by-one": ("treegraft_oracle", "    M = budget + 1\n", "    M = budget\n"),
    "prune-position-one-based": ("treegraft_oracle", "pos_o[b, :k] = [int(d[v]) for v in kept]",
                                 "pos_o[b, :k] = [int(d[v]) + 1 for v in kept]"),
    "prune-paths-to-internal-nodes": ("treegraft_oracle",
                                      "leaves = [i for i in range(k) if i not in has_child]",
                                      "leaves = [i for i in range(k) if i in has_child]"),
    # grow step (Algorithm 2)
    "grow-small-frontier-all-nodes": ("treegraft_oracle", 'C = list(state["new"])',
                                      "C = list(range(n))"),
    "grow-middle-own-row": ("treegraft_oracle",
                            "row = _row_values(middle_logits, parent[v], bf16)",
                            "row = _row_values(middle_logits, v, bf16)"),
    "grow-visited-never-updated": ("treegraft_oracle", "        P.update(C)\n", "        pass\n"),
    "grow-frontier-ties-to-higher-id": ("treegraft_oracle",
                                        "F = sorted(C, key=lambda v: (-float(score[v]), v))[:W]",
                                        "F = sorted(C, key=lambda v: (-float(score[v]), -v))[:W]"),
    "grow-score-subtracts": ("treegraft_oracle", "score.append(np.float32(score[v] + lp))",
                             "score.append(np.float32(score[v] - lp))"),
    "grow-ngram-score-subtracts": ("treegraft_oracle",
                                   "score.append(np.float32(score[v] + np.float32(lp)))",
                                   "score.append(np.float32(score[v] - np.float32(lp)))"),
    # stochastic verification
    "sample-children-descending": ("sample_oracle",
                                   "            for c in children[v]:\n                x = int(token[a + c])",
                                   "            for c in children[v][::-1]:\n                x = int(token[a + c])"),
    "sample-residual-kept": ("sample_oracle", "                R -= p[x]\n",
                             "                pass\n"),
    "sample-accept-inverted": ("sample_oracle", "if lhs < p[x]:", "if lhs > p[x]:"),
    "sample-bonus-keeps-children": ("sample_oracle",
                                    "            resid[int(token[a + c])] = 0.0\n",
                                    "            pass\n"),
    "sample-temperature-multiplies": ("sample_oracle", "e = np.exp((x - m) / T)",
                                      "e = np.exp((x - m) * T)"),
    "sample-bonus-wrong-uniform": ("sample_oracle", "target = float(u[a + v, 1]) * total",
                                   "target = float(u[a + v, 0]) * total"),
    # n-gram small drafter
    "ngram-earliest-occurrence": ("ngram_oracle", "return max(hits), n", "return min(hits), n"),
    "ngram-frequency-ties-to-higher-id": ("ngram_oracle", "best = min(counts, key=lambda t: (-counts[t], t))",
                                          "best = min(counts, key=lambda t: (-counts[t], -t))"),
    "ngram-fallback-earliest-position": ("ngram_oracle",
                                         "return max(j for j, t in enumerate(prompt) if int(t) == best)",
                                         "return min(j for j, t in enumerate(prompt) if int(t) == best)"),
    "ngram-shortest-order-first": ("ngram_oracle", "for n in range(min(max_n, len(query)), 0, -1):",
                                   "for n in range(1, min(max_n, len(query)) + 1):"),
    "ngram-query-repeats-root-token": ("ngram_oracle", "    while w != 0:\n", "    while w != -1:\n"),
    "ngram-path-reversed": ("ngram_oracle", "seq = [int(t) for t in ctx] + path[::-1]",
                            "seq = [int(t) for t in ctx] + path"),
    "ngram-window-from-the-start": ("ngram_oracle", "return seq[-max_n:]", "return seq[:max_n]"),
    "ngram-skips-first-position": ("ngram_oracle", "for j in range(n - 1, len(prompt))",
                                   "for j in range(n, len(prompt))"),
    "ngram-draft-next-row": ("ngram_oracle", "return [int(t) for t in cache_tok[j][:m]], [np.float32(x) for x in cache_lp[j][:m]], j, n",
                             "return [int(t) for t in cache_tok[j - 1][:m]], [np.float32(x) for x in cache_lp[j - 1][:m]], j, n"),
}


def _mutant(module, old, new):
    path = os.path.join(ORACLE_DIR, module + ".py")
    with open(path) as f:
        src = f.read()
    assert src.count(old) == 1, f"mutation text not found exactly once in {module}: {old!r}"
    mod = types.ModuleType(f"oracle.{module}")
    mod.__file__ = path
    exec(compile(src.replace(old, new), path, "exec"), mod.__dict__)
    return mod


def _pin_calls(pins):
    """Every test function of a pin module, once per parametrisation."""
    for name, fn in inspect.getmembers(pins, inspect.isfunction):
        if not name.startswith("test_") or fn.__module__ != pins.__name__:
            continue
        combos = [{}]
        for mark in getattr(fn, "pytestmark", []):
            if mark.name != "parametrize":
                continue
            argnames, values = mark.args[0], mark.args[1]
            names = ([a.strip() for a in argnames.split(",")] if isinstance(argnames, str)
                     else list(argnames))
            grown = []
            for c in combos:
                for v in values:
                    if hasattr(v, "marks") and hasattr(v, "values"):  # pytest.param(...)
                        vals = tuple(v.values)
                    elif len(names) == 1:
                        vals = (v,)
                    else:
                        vals = tuple(v)
                    d = dict(c)
                    d.update(zip(names, vals))
                    grown.append(d)
            combos = grown
        if set(inspect.signature(fn).parameters) != set(combos[0]):
            continue  # takes fixtures other than its parameters
        for kw in combos:
            yield name, fn, kw


def _all_pin_calls():
    for pins in PIN_MODULES:
        yield from _pin_calls(pins)


def test_every_pin_module_has_runnable_pins():
    for pins in PIN_MODULES:
        assert sum(1 for _ in _pin_calls(pins)) >= 8, pins.__name__


def test_unmutated_oracle_passes_every_pin():
    for name, fn, kw in _all_pin_calls():
        fn(**kw)


@pytest.mark.parametrize("case", list(MUTATIONS))
def test_pins_catch_the_mistake(case, monkeypatch):
    module, old, new = MUTATIONS[case]
    mutant = _mutant(module, old, new)
    for user, attr in USES[module]:
        monkeypatch.setattr(user, attr, mutant)
    for name, fn, kw in _all_pin_calls():
        try:
            fn(**kw)
        except (Exception, pytest.fail.Exception):  # a failed check, or any error it causes
            return
    pytest.fail(f"no pin fails with the mistake {case!r}")
