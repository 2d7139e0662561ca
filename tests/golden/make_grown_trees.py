"""Write tests/golden/llama3_8b_grown_trees.json: the draft trees of the
Llama-3-8B-shaped verify workload, grown the way that workload is defined.

Each tree is built by the oracle alone:
  * Algorithm 1 (the all-small schedule of Algorithm 2): D = 6 expansion
    steps with frontier W = 10 and m = 10 children per frontier node, chosen
    by the drafter's top-m tokens and ranked by cumulative log-probability
    (Sec. 3.1, s(u) = s(v) p(u) in log form), from the root alone;
  * then GlobalPrune (Algorithm 3) to a verification budget of B_ver = 59
    non-root nodes, so the verified tree has 60 nodes.
The drafter's next-token logits at node v are row v of a seeded fp32 table
over the 128256-token Llama-3 vocabulary (the stand-in for the drafter's
forward over the tree): N(0, 3^2) plus, in every row, one planted confident
token whose logit is raised by a bump drawn uniformly from [4, 24].  A real
drafter is often sure of its next token; without such rows every top-10
log-probability sits near -3 to -4.5 and GlobalPrune keeps a bushy tree of
depth 2-3 instead of the depth-6 tree the workload names.  synth only draws
those rows; every step of the method runs in oracle/.

    python tests/golden/make_grown_trees.py      # rewrites the JSON file
"""
from __future__ import annotations

import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

from oracle import treegraft_oracle as O  # noqa: E402
from paper_2608_26112_gb300 import synth  # noqa: E402

OUT = os.path.join(HERE, "llama3_8b_grown_trees.json")
STEPS, W, M_CHILD, BUDGET = 6, 10, 10, 59
N_TREES = 16
BUMP = (4.0, 24.0)
TABLE_SEED = 50_000
V = synth.LLAMA3_VOCAB


def grown_tree(i: int):
    rng = synth.make_rng(TABLE_SEED + i)
    # rows of nodes that can be expanded: every node but the last step's children
    rows = 1 + W + (STEPS - 2) * W * M_CHILD
    table = synth.normal_f32(rng, (rows, V), 3.0)
    sure = rng.integers(0, V, size=rows)
    table[np.arange(rows), sure] += rng.uniform(BUMP[0], BUMP[1], size=rows).astype(np.float32)
    parent, token, _, score, _, _ = O.grow_tree([0] * STEPS, W, M_CHILD, table, table)
    kept, n_kept, new_parent, position, _, _, _ = O.global_prune(
        parent, score, np.array([0, len(parent)], np.int32), BUDGET, STEPS + 1)
    k = int(n_kept[0])
    ids = kept[0, :k]
    return dict(index=i, nodes_grown=int(len(parent)), parent=[int(x) for x in new_parent[0, :k]],
                token=[int(token[v]) for v in ids], depth=int(position[0, :k].max()))


def main():
    trees = [grown_tree(i) for i in range(N_TREES)]
    doc = {"source": ("Algorithm 1 (all-small schedule of Algorithm 2: 6 expansion steps, "
                      "W = m = 10, cumulative log-probability, Sec. 3.1) on seeded fp32 drafter "
                      "rows over 128256 tokens, N(0, 3^2) plus one confident token per row "
                      f"raised by U{BUMP} (row v = node v, table seed {TABLE_SEED} + index), "
                      f"then GlobalPrune (Algorithm 3) to B_ver = {BUDGET}. Written by "
                      "tests/golden/make_grown_trees.py with oracle/ only."),
           "trees": trees}
    with open(OUT, "w") as f:
        json.dump(doc, f, separators=(",", ":"))
        f.write("\n")
    print(OUT, [t["depth"] for t in trees], [len(t["parent"]) for t in trees])


if __name__ == "__main__":
    main()
