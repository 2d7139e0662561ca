#!/usr/bin/env python
"""Benchmark of the TreeGraft verify-and-grow step on GB300.

One step = one pass of the whole hot path over one batch of synthetic input
of the Llama-3-8B-shaped verify workload (batch 1, prefix 2048, 60-node tree
of depth 6, GQA 32/8, head_dim 128, vocab 128256, bf16):
  treegraft_tree_attn      target verification attention over prefix + tree
  treegraft_expand_topk    per-node log-softmax + top-10 + path scores (drafter rows)
  treegraft_rescore_select stronger-drafter rescoring + top-10 reselection
  treegraft_accept         greedy longest accepted path on the target rows

Inputs are resident in HBM; eight input sets are rotated so that the bytes
touched between two uses of a set (~280 MB) exceed the 126 MB L2.  Steps
are replayed from CUDA graphs.  Per-kernel durations come from graphs of
that kernel alone, timed with CUDA events on the launching stream.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun (N > 1) every rank runs its own independent sequences (the
verify step of one sequence never needs another's data): weak scaling, no
data-path collective; the barrier and the max-over-ranks time use NCCL.
Rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tree-verify steps/s & tree_attn HBM GB/s (% of peak), Llama-3-8B shape"
WORKLOAD = "llama3-8b-verify"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20000)
    p.add_argument("--warmup", type=int, default=50)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--sets", type=int, default=8)
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-serving", action="store_true", help="skip the batched serving sweep")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


# --------------------------------------------------------------------------- workload

def algorithmic_costs(wl):
    """Bytes each call must move at minimum and the attention FLOPs."""
    sh = wl["shape"]
    n = len(wl["parent"])
    P = int(wl["prefix_len"][0])
    Hq, Hkv, D, V, k, N = sh["Hq"], sh["Hkv"], sh["D"], sh["V"], sh["k"], sh["N"]
    depth = [0] * n
    for v in range(1, n):
        depth[v] = depth[wl["parent"][v]] + 1
    keys = sum(P + d + 1 for d in depth)
    attn_bytes = 2 * (P + n) * Hkv * D * 2 + 2 * n * Hq * D * 2 + n * 4 * 2
    attn_flops = 4 * Hq * D * keys
    expand_bytes = n * V * 2 + n * 4 + n * k * 12
    accept_bytes = n * V * 2 + n * 8 + 4 * 3 + n * 4
    rescore_bytes = n * (4 + 4 + 4 + 4 + 1) + n * 4 + n * 8 + N * 4
    return dict(tree_attn=(attn_bytes, attn_flops), expand_topk=(expand_bytes, 0),
                rescore_select=(rescore_bytes, 0), accept=(accept_bytes, 0))


def build_sets(R, seed, dev):
    import numpy as np
    import torch
    from paper_2608_26112_gb300 import synth

    def bf(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)

    def t(a):
        return torch.from_numpy(np.ascontiguousarray(a)).to(dev)

    sets, host = [], []
    for r in range(R):
        wl = synth.make_workload(WORKLOAD, seed=seed + r, with_strong=(r == 0))
        rng = synth.make_rng(10_000 + seed + r)
        # target rows for accept: a second, independent logit array with its own bumps
        tl = synth.normal_f32(rng, wl["logits"].shape, 3.0)
        synth.plant_child_bump(rng, tl, wl["parent"], wl["token"], np.arange(len(wl["parent"])))
        wl["target_logits"] = synth.f32_to_bf16_bits(tl)
        if r == 0:
            strong = t(wl["strong_lp"])
        d = dict(q=bf(wl["q"]), k=bf(wl["k_cache"]), v=bf(wl["v_cache"]),
                 prefix_len=t(wl["prefix_len"]), parent=t(wl["parent"]), token=t(wl["token"]),
                 node_off=t(wl["node_off"]), logits=bf(wl["logits"]),
                 target=bf(wl["target_logits"]), parent_score=t(wl["parent_score"]),
                 weak_edge=t(wl["weak_edge"]), visited=t(wl["visited"]), strong=strong,
                 u=t(rng.random((len(wl["parent"]), 2)).astype(np.float32)))
        sets.append(d)
        wl.pop("strong_lp", None)
        host.append(wl)
    return sets, host


def alloc_outputs(d, sh, dev):
    import torch
    import paper_2608_26112_gb300 as tg
    n = d["parent"].shape[0]
    k, N = sh["k"], sh["N"]
    return dict(
        o=torch.empty_like(d["q"]),
        tok=torch.empty(n, k, dtype=torch.int32, device=dev),
        lp=torch.empty(n, k, dtype=torch.float32, device=dev),
        sc=torch.empty(n, k, dtype=torch.float32, device=dev),
        edge=torch.empty(n, dtype=torch.float32, device=dev),
        score=torch.empty(n, dtype=torch.float32, device=dev),
        sel=torch.empty(1, N, dtype=torch.int32, device=dev),
        nsel=torch.empty(1, dtype=torch.int32, device=dev),
        path=torch.empty(1, n, dtype=torch.int32, device=dev),
        alen=torch.empty(1, dtype=torch.int32, device=dev),
        bonus=torch.empty(1, dtype=torch.int32, device=dev),
        ws=tg.accept_workspace(1, n, dev),
        sws=tg.accept_sample_workspace(1, n, dev),
        attn_ws=torch.zeros(max(16, tg.tree_attn_workspace_size(
            1, n, d["q"].shape[1], d["k"].shape[1], d["q"].shape[2])), dtype=torch.uint8,
            device=dev))


def call(name, d, o, sh):
    import paper_2608_26112_gb300 as tg
    n = d["parent"].shape[0]
    if name == "tree_attn":
        tg.tree_attn(d["q"], d["k"], d["v"], d["prefix_len"], d["parent"], d["node_off"], n,
                     out=o["o"], ws=o["attn_ws"])
    elif name == "expand_topk":
        tg.expand_topk(d["logits"], d["parent_score"], sh["k"], out=(o["tok"], o["lp"], o["sc"]))
    elif name == "rescore_select":
        tg.rescore_select(d["weak_edge"], d["strong"], d["parent"], d["token"], d["visited"],
                          d["node_off"], n, sh["N"],
                          out=(o["edge"], o["score"], o["sel"], o["nsel"]))
    elif name == "accept":
        tg.accept(d["target"], d["token"], d["parent"], d["node_off"], n, n, o["ws"],
                  out=(o["path"], o["alen"], o["bonus"]))
    elif name == "accept_sample":
        tg.accept_sample(d["target"], d["token"], d["parent"], d["node_off"], n, n, d["u"],
                         SAMPLE_T, o["sws"], out=(o["path"], o["alen"], o["bonus"]))


KERNELS = ["tree_attn", "expand_topk", "rescore_select", "accept"]
REPEATS = 5  # the K-step timed region is run this many times; the median is reported
# timed beside the step: verification at temperature SAMPLE_T instead of 0
BESIDE = ["accept_sample"]
SAMPLE_T = 1.0


def step(d, o, sh):
    for name in KERNELS:
        call(name, d, o, sh)


def capture(fn, stream):
    import torch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    return g


def time_graph(g, reps, stream):
    import torch
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(reps):
            g.replay()
        e1.record(stream)
    e1.synchronize()
    return e0.elapsed_time(e1) / 1e3  # seconds


def prune_timing(R, seed, dev, stream, reps):
    """GlobalPrune (Algorithm 3) timed beside the step, not inside it: the
    pre-pruning tree of the Llama-3-8B-shaped verify step (6 expansion steps
    of frontier 10 and branching 10: 511 nodes) with path-sum scores,
    pruned to a 59-node budget; R input sets, one launch each."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    sets = []
    for r in range(R):
        rng = synth.make_rng(20_000 + seed + r)
        par = synth.expansion_tree(rng, 6, 10, 10)
        sc = synth.path_scores(rng, par)
        sets.append((torch.from_numpy(sc).to(dev), torch.from_numpy(par).to(dev),
                     torch.tensor([0, len(par)], dtype=torch.int32, device=dev), len(par)))
    outs = []
    with torch.cuda.stream(stream):
        for sc, par, off, n in sets:
            outs.append(tg.global_prune(sc, par, off, n, 59, 8, stream=stream))
    stream.synchronize()
    g = capture(lambda: [tg.global_prune(sc, par, off, n, 59, 8, out=o, stream=stream)
                         for (sc, par, off, n), o in zip(sets, outs)], stream)
    g.replay()
    t = time_graph(g, reps, stream) / (reps * R)
    n = sets[0][3]
    return {"us": t * 1e6, "nodes_in": n, "budget": 59, "bytes": n * 8 + 60 * 16,
            "in_step": False, "note": "Algorithm 3 on the pre-pruning tree, latency-bound"}


EXTRA_CONFIGS = ["llama3-70b-verify", "graft-mha", "tiny"]


def config_timing(name, seed, dev, stream, n_sets=2, seconds=0.15):
    """The step's four kernels on another synthetic workload, timed alone
    (not part of the headline step): per-kernel launch time over n_sets
    rotating input sets, attention FLOP/s against the bf16 tensor peak and
    bytes/s against the HBM peak.  For the Llama-3-70B-shaped verify batch
    (4 trees of 128 nodes, prefix 8192, GQA 64/8) the attention is
    tensor-bound (137 GFLOP per launch)."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    def bf(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)

    def t(a):
        return torch.from_numpy(np.ascontiguousarray(a)).to(dev)

    sets = []
    for r in range(n_sets):
        wl = synth.make_workload(name, seed=seed + r)
        sh = wl["shape"]
        rng = synth.make_rng(40_000 + seed + r)
        lg = wl["logits"]
        bf16 = lg.dtype == np.uint16
        tl = synth.normal_f32(rng, lg.shape, 3.0)
        synth.plant_child_bump(rng, tl, wl["parent"], wl["token"], np.arange(len(wl["parent"])))
        target = synth.f32_to_bf16_bits(tl) if bf16 else tl
        node_off = wl["node_off"]
        B = len(node_off) - 1
        mx = int(np.max(np.diff(node_off)))
        n_total = len(wl["parent"])
        d = dict(q=bf(wl["q"]), k=bf(wl["k_cache"]), v=bf(wl["v_cache"]),
                 prefix_len=t(wl["prefix_len"]), parent=t(wl["parent"]), token=t(wl["token"]),
                 node_off=t(node_off), logits=bf(lg) if bf16 else t(lg),
                 target=bf(target) if bf16 else t(target), parent_score=t(wl["parent_score"]),
                 weak_edge=t(wl["weak_edge"]), visited=t(wl["visited"]), strong=t(wl["strong_lp"]))
        k, N = sh["k"], sh["N"]
        o = dict(o=torch.empty_like(d["q"]),
                 tok=torch.empty(n_total, k, dtype=torch.int32, device=dev),
                 lp=torch.empty(n_total, k, dtype=torch.float32, device=dev),
                 sc=torch.empty(n_total, k, dtype=torch.float32, device=dev),
                 edge=torch.empty(n_total, dtype=torch.float32, device=dev),
                 score=torch.empty(n_total, dtype=torch.float32, device=dev),
                 sel=torch.empty(B, N, dtype=torch.int32, device=dev),
                 nsel=torch.empty(B, dtype=torch.int32, device=dev),
                 path=torch.empty(B, mx, dtype=torch.int32, device=dev),
                 alen=torch.empty(B, dtype=torch.int32, device=dev),
                 bonus=torch.empty(B, dtype=torch.int32, device=dev),
                 ws=tg.accept_workspace(B, n_total, dev),
                 attn_ws=torch.zeros(max(16, tg.tree_attn_workspace_size(
                     B, mx, sh["Hq"], sh["Hkv"], sh["D"])), dtype=torch.uint8, device=dev))
        sets.append((wl, d, o, mx))
    wl, _, _, mx = sets[0]
    sh = wl["shape"]

    def run(kname, d, o, mx):
        if kname == "tree_attn":
            tg.tree_attn(d["q"], d["k"], d["v"], d["prefix_len"], d["parent"], d["node_off"], mx,
                         out=o["o"], ws=o["attn_ws"], stream=stream)
        elif kname == "expand_topk":
            tg.expand_topk(d["logits"], d["parent_score"], sh["k"], out=(o["tok"], o["lp"], o["sc"]),
                           stream=stream)
        elif kname == "rescore_select":
            tg.rescore_select(d["weak_edge"], d["strong"], d["parent"], d["token"], d["visited"],
                              d["node_off"], mx, sh["N"],
                              out=(o["edge"], o["score"], o["sel"], o["nsel"]), stream=stream)
        else:
            tg.accept(d["target"], d["token"], d["parent"], d["node_off"], mx, mx, o["ws"],
                      out=(o["path"], o["alen"], o["bonus"]), stream=stream)

    with torch.cuda.stream(stream):
        for _, d, o, m_ in sets:
            for kname in KERNELS:
                run(kname, d, o, m_)
    stream.synchronize()
    assert tg.last_device_status(stream) == 0
    # algorithmic costs of set 0
    parent, node_off = wl["parent"], wl["node_off"]
    B = len(node_off) - 1
    Hq, Hkv, D, V = sh["Hq"], sh["Hkv"], sh["D"], sh["V"]
    elem = 2 if wl["logits"].dtype == np.uint16 else 4
    keys, kv_bytes = 0, 0
    for b in range(B):
        lo, hi = int(node_off[b]), int(node_off[b + 1])
        P = int(wl["prefix_len"][b])
        depth = [0] * (hi - lo)
        for v in range(1, hi - lo):
            depth[v] = depth[parent[lo + v]] + 1
        keys += sum(P + dd + 1 for dd in depth)
        kv_bytes += 2 * (P + hi - lo) * Hkv * D * 2
    n_total = len(parent)
    costs = dict(tree_attn=(kv_bytes + 2 * n_total * Hq * D * 2, 4 * Hq * D * keys),
                 expand_topk=(n_total * V * elem, 0), accept=(n_total * V * elem, 0),
                 rescore_select=(n_total * 17, 0))
    pk, _ = peaks()
    out = {}
    for kname in KERNELS:
        g = capture(lambda kname=kname: [run(kname, d, o, m_) for _, d, o, m_ in sets], stream)
        g.replay()
        t1 = time_graph(g, 3, stream) / (3 * n_sets)
        reps = max(3, min(2000, int(seconds / max(t1 * n_sets, 1e-7))))
        tk = time_graph(g, reps, stream) / (reps * n_sets)
        b_, f_ = costs[kname]
        ent = {"us": tk * 1e6, "bytes": b_, "GBps": b_ / tk / 1e9, "hbm_frac": b_ / tk / 1e9 / pk["hbm_gbs"]}
        if f_:
            ent["TFLOPs"] = f_ / tk / 1e12
            ent["tensor_frac"] = f_ / tk / 1e12 / pk["bf16_tflops"]
            ent["roofline_frac"] = max(b_ / (pk["hbm_gbs"] * 1e9), f_ / (pk["bf16_tflops"] * 1e12)) / tk
        out[kname] = ent
    return {"shape": {k_: v_ for k_, v_ in sh.items() if k_ in ("B", "P", "n", "Hq", "Hkv", "D", "V", "k", "N")},
            "kernels": out, "sets": n_sets}


SERVING_BATCHES = [1, 2, 4, 8, 16, 32, 64]


def _attn_costs(parent, node_off, prefix_len, Hq, Hkv, D):
    """Algorithmic bytes (K/V of prefix and tree, q and o) and FLOPs
    (4 Hq D per visible key of every node) of one tree_attn launch."""
    kv_bytes, keys = 0, 0
    n_total = int(node_off[-1])
    for b in range(len(node_off) - 1):
        lo, hi = int(node_off[b]), int(node_off[b + 1])
        P = int(prefix_len[b])
        depth = [0] * (hi - lo)
        for v in range(1, hi - lo):
            depth[v] = depth[int(parent[lo + v])] + 1
        keys += sum(P + d + 1 for d in depth)
        kv_bytes += 2 * (P + hi - lo) * Hkv * D * 2
    return kv_bytes + 2 * n_total * Hq * D * 2, 4 * Hq * D * keys


def serving_timing(B, dev, stream, seconds=0.12):
    """One point of the batched serving sweep: B trees with prefixes
    log-uniform in [512, 32768], 32-256 nodes, depth 4-10 (synth's serving
    shape, seed 1000 + B), GQA 32/8, head_dim 128, Llama-3 vocabulary, top-10.
    q/k/v ~ N(0, 1) and the drafter and target logits ~ N(0, 3^2) are drawn
    on the device from a generator seeded 1000 + B and rounded to bf16; the
    stronger drafter's fp32 rows likewise.  Per kernel: launch time over
    rotating input sets (enough that a cycle touches more than the L2), GB/s
    and, for the attention, TFLOP/s and the roofline fraction.  A step is
    tree_attn -> expand_topk -> rescore_select -> accept on one input set."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    shape = synth.serving_shape(B, seed=0)
    rng = synth.make_rng(1000 + B)
    parent, token, node_off = synth.make_trees(rng, shape)
    Hq, Hkv, D, V, k, N = 32, 8, 128, synth.LLAMA3_VOCAB, 10, 10
    P = np.asarray(shape["P"], np.int32)
    ns = np.diff(node_off)
    n_total, mx = int(node_off[-1]), int(ns.max())
    S_max = int((P + ns).max())
    set_bytes = (2 * B * Hkv * S_max * D * 2 + 2 * n_total * V * 2 + n_total * V * 4)
    R = int(min(4, max(1, -(-400 * 2 ** 20 // set_bytes))))
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 + B)

    def randn_bf16(shape_, sigma=1.0, rows_per=512):
        out = torch.empty(shape_, dtype=torch.bfloat16, device=dev)
        flat = out.view(shape_[0], -1)
        for r0 in range(0, shape_[0], rows_per):
            r1 = min(shape_[0], r0 + rows_per)
            flat[r0:r1] = torch.randn((r1 - r0, flat.shape[1]), generator=gen, device=dev).mul_(sigma)
        return out

    t32 = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    vis = np.zeros(n_total, np.uint8)
    sets = []
    for _ in range(R):
        kv = [randn_bf16((B * Hkv, S_max, D), rows_per=8).view(B, Hkv, S_max, D) for _ in range(2)]
        strong = torch.empty(n_total, V, dtype=torch.float32, device=dev)
        for r0 in range(0, n_total, 512):
            r1 = min(n_total, r0 + 512)
            strong[r0:r1] = torch.randn((r1 - r0, V), generator=gen, device=dev).mul_(3.0).sub_(
                float(np.log(V)) + 4.5).clamp_(max=0.0)
        d = dict(q=randn_bf16((n_total, Hq, D)), k=kv[0], v=kv[1], prefix_len=t32(P),
                 parent=t32(parent), token=t32(token), node_off=t32(node_off),
                 logits=randn_bf16((n_total, V), 3.0), target=randn_bf16((n_total, V), 3.0),
                 parent_score=torch.zeros(n_total, device=dev),
                 weak_edge=torch.full((n_total,), -12.0, device=dev), visited=t32(vis),
                 strong=strong)
        o = dict(o=torch.empty_like(d["q"]),
                 tok=torch.empty(n_total, k, dtype=torch.int32, device=dev),
                 lp=torch.empty(n_total, k, dtype=torch.float32, device=dev),
                 sc=torch.empty(n_total, k, dtype=torch.float32, device=dev),
                 edge=torch.empty(n_total, dtype=torch.float32, device=dev),
                 score=torch.empty(n_total, dtype=torch.float32, device=dev),
                 sel=torch.empty(B, N, dtype=torch.int32, device=dev),
                 nsel=torch.empty(B, dtype=torch.int32, device=dev),
                 path=torch.empty(B, mx, dtype=torch.int32, device=dev),
                 alen=torch.empty(B, dtype=torch.int32, device=dev),
                 bonus=torch.empty(B, dtype=torch.int32, device=dev),
                 ws=tg.accept_workspace(B, n_total, dev),
                 attn_ws=torch.zeros(max(16, tg.tree_attn_workspace_size(B, mx, Hq, Hkv, D)),
                                     dtype=torch.uint8, device=dev))
        sets.append((d, o))

    def run(kname, d, o):
        if kname == "tree_attn":
            tg.tree_attn(d["q"], d["k"], d["v"], d["prefix_len"], d["parent"], d["node_off"], mx,
                         out=o["o"], ws=o["attn_ws"], stream=stream)
        elif kname == "expand_topk":
            tg.expand_topk(d["logits"], d["parent_score"], k, out=(o["tok"], o["lp"], o["sc"]),
                           stream=stream)
        elif kname == "rescore_select":
            tg.rescore_select(d["weak_edge"], d["strong"], d["parent"], d["token"], d["visited"],
                              d["node_off"], mx, N, out=(o["edge"], o["score"], o["sel"], o["nsel"]),
                              stream=stream)
        else:
            tg.accept(d["target"], d["token"], d["parent"], d["node_off"], mx, mx, o["ws"],
                      out=(o["path"], o["alen"], o["bonus"]), stream=stream)

    with torch.cuda.stream(stream):
        for d, o in sets:
            for kname in KERNELS:
                run(kname, d, o)
    stream.synchronize()
    assert tg.last_device_status(stream) == 0
    pk, _ = peaks()
    ab, af = _attn_costs(parent, node_off, P, Hq, Hkv, D)
    costs = dict(tree_attn=(ab, af), expand_topk=(n_total * V * 2, 0), accept=(n_total * V * 2, 0),
                 rescore_select=(n_total * 17, 0))

    def timed(fn):
        g = capture(lambda: [fn(d, o) for d, o in sets], stream)
        g.replay()
        t1 = time_graph(g, 2, stream) / (2 * R)
        reps = max(3, min(2000, int(seconds / max(t1 * R, 1e-7))))
        return time_graph(g, reps, stream) / (reps * R)

    out = {}
    for kname in KERNELS:
        tk = timed(lambda d, o, kname=kname: run(kname, d, o))
        b_, f_ = costs[kname]
        ent = {"us": tk * 1e6, "bytes": b_, "GBps": b_ / tk / 1e9,
               "hbm_frac": b_ / tk / 1e9 / pk["hbm_gbs"]}
        if f_:
            roof = max(b_ / (pk["hbm_gbs"] * 1e9), f_ / (pk["bf16_tflops"] * 1e12))
            ent.update(TFLOPs=f_ / tk / 1e12, tensor_frac=f_ / tk / 1e12 / pk["bf16_tflops"],
                       roofline_frac=roof / tk,
                       bound="tensor" if f_ / (pk["bf16_tflops"] * 1e12) > b_ / (pk["hbm_gbs"] * 1e9)
                       else "hbm")
        out[kname] = ent
    t_step = timed(lambda d, o: [run(kn, d, o) for kn in KERNELS])
    res = {"B": B, "prefix_min": int(P.min()), "prefix_max": int(P.max()),
           "prefix_mean": float(P.mean()), "nodes": int(n_total), "nodes_max": mx,
           "sets": R, "kernels": out, "step_us": t_step * 1e6, "steps_per_s": 1.0 / t_step,
           "launches_per_step": len(KERNELS)}
    del sets
    torch.cuda.empty_cache()
    return res


def graft_pipeline_timing(seed, dev, stream, seconds=0.15, n_sets=4):
    """The two-drafter grafting step of the MHA drafter shape as one
    CUDA-graph step: the drafter's tree attention over its 64-node tree
    (32 heads, head_dim 128, prefix 1024), rescoring of all 64 nodes from the
    stronger drafter's fp32 log-probs (32000 tokens; weak log-probs +
    N(0, 0.5^2)), reselection of the top 16 grafting positions, expansion of
    each by its top-8 tokens with the children grafted onto the tree (192
    nodes), then greedy acceptance on bf16 target logits of the grafted
    tree.  n_sets rotating input sets; per-kernel launch times beside."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    n, V, N, k = 64, 32000, 16, 8
    cap = n + N * k
    sets = []
    for r in range(n_sets):
        wl = synth.make_workload("graft-mha", seed=seed + r, with_logits=False, with_strong=False)
        sh = wl["shape"]
        rng = synth.make_rng(60_000 + seed + r)
        weak_lp = synth.normal_f32(rng, (n, V), 3.0, -np.log(V) - 4.5)
        strong_lp = (weak_lp + synth.normal_f32(rng, (n, V), 0.5)).astype(np.float32)
        weak_edge = np.zeros(n, np.float32)
        weak_edge[1:] = weak_lp[wl["parent"][1:], wl["token"][1:]]
        tl = synth.f32_to_bf16_bits(synth.normal_f32(rng, (cap, V), 3.0))
        bf = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(dev).view(torch.bfloat16)
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        d = dict(q=bf(wl["q"]), k=bf(wl["k_cache"]), v=bf(wl["v_cache"]),
                 prefix_len=t(wl["prefix_len"]), node_off=t(wl["node_off"]),
                 node_off2=torch.tensor([0, cap], dtype=torch.int32, device=dev),
                 weak_edge=t(weak_edge), strong=t(strong_lp),
                 visited=torch.zeros(n, dtype=torch.uint8, device=dev),
                 target=bf(tl), parent0=t(wl["parent"]), token0=t(wl["token"]))
        o = dict(o=torch.empty_like(d["q"]),
                 parent=torch.zeros(cap, dtype=torch.int32, device=dev),
                 token=torch.zeros(cap, dtype=torch.int32, device=dev),
                 edge=torch.zeros(cap, dtype=torch.float32, device=dev),
                 score=torch.zeros(cap, dtype=torch.float32, device=dev),
                 sel=torch.empty(1, N, dtype=torch.int32, device=dev),
                 nsel=torch.empty(1, dtype=torch.int32, device=dev),
                 path=torch.empty(1, cap, dtype=torch.int32, device=dev),
                 alen=torch.empty(1, dtype=torch.int32, device=dev),
                 bonus=torch.empty(1, dtype=torch.int32, device=dev),
                 ws=tg.accept_workspace(1, cap, dev),
                 attn_ws=torch.zeros(max(16, tg.tree_attn_workspace_size(
                     1, n, sh["Hq"], sh["Hkv"], sh["D"])), dtype=torch.uint8, device=dev))
        o["parent"][:n] = d["parent0"]
        o["token"][:n] = d["token0"]
        sets.append((d, o))

    def stage(name, d, o):
        if name == "tree_attn":
            tg.tree_attn(d["q"], d["k"], d["v"], d["prefix_len"], o["parent"][:n], d["node_off"], n,
                         out=o["o"], ws=o["attn_ws"], stream=stream)
        elif name == "rescore_select":
            tg.rescore_select(d["weak_edge"], d["strong"], o["parent"][:n], o["token"][:n],
                              d["visited"], d["node_off"], n, N,
                              out=(o["edge"][:n], o["score"][:n], o["sel"], o["nsel"]), stream=stream)
        elif name == "graft_expand":
            tg.graft_expand(d["strong"], o["sel"], k, cap, n, o["parent"], o["token"], o["edge"],
                            o["score"], stream=stream)
        else:
            tg.accept(d["target"], o["token"], o["parent"], d["node_off2"], cap, cap, o["ws"],
                      out=(o["path"], o["alen"], o["bonus"]), stream=stream)

    names = ["tree_attn", "rescore_select", "graft_expand", "accept"]
    with torch.cuda.stream(stream):
        for d, o in sets:
            for nm in names:
                stage(nm, d, o)
    stream.synchronize()
    assert tg.last_device_status(stream) == 0

    def timed(fn):
        g = capture(lambda: [fn(d, o) for d, o in sets], stream)
        g.replay()
        t1 = time_graph(g, 2, stream) / (2 * n_sets)
        reps = max(3, min(4000, int(seconds / max(t1 * n_sets, 1e-7))))
        return time_graph(g, reps, stream) / (reps * n_sets)

    t_step = timed(lambda d, o: [stage(nm, d, o) for nm in names])
    per = {nm: timed(lambda d, o, nm=nm: stage(nm, d, o)) * 1e6 for nm in names}
    d0 = sets[0][0]
    ab, af = _attn_costs(sets[0][1]["parent"][:n].cpu().numpy(), [0, n], [1024], 32, 32, 128)
    bytes_ = {"tree_attn": ab, "rescore_select": n * 17 + 64 * 4,
              "graft_expand": N * V * 4 + N * k * 16, "accept": cap * V * 2}
    kern = {nm: {"us": per[nm], "bytes": bytes_[nm], "GBps": bytes_[nm] / per[nm] / 1e3}
            for nm in names}
    kern["tree_attn"]["TFLOPs"] = af / per["tree_attn"] / 1e6
    return {"shape": {"P": 1024, "n": n, "n_grafted": cap, "Hq": 32, "Hkv": 32, "D": 128, "V": V,
                      "N": N, "k": k},
            "step_us": t_step * 1e6, "steps_per_s": 1.0 / t_step, "launches_per_step": len(names),
            "kernels": kern, "sets": n_sets}


GROW_SCHEDULE = [1, 0, 1, 0, 1]


def grow_timing(seed, dev, stream, reps, n_sets=3):
    """The shared-tree construction (Algorithm 2) timed beside the step, not
    inside it: the fixed schedule [1, 0, 1, 0, 1] of the paper's ablation
    (middle, small, middle, small, middle drafter) with frontier W = 10 and
    branching m = 10, on seeded N(0, 3^2) bf16 drafter tables over the
    Llama-3 vocabulary (128256); one tree, grown from its root to 411
    nodes.  Each loop is 5 grow_step calls (15 launches); n_sets table pairs
    rotate so the 85 MB of rows a loop scans come from HBM."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    W = m = 10
    V = 128256
    sizes, n, new_lo, n_vis = [], 1, 0, 0
    for a in GROW_SCHEDULE:
        pool_lo = new_lo if a == 0 else n_vis
        sizes.append((a, n, pool_lo))
        if a == 1:
            n_vis = n
        new_lo, n = n, n + min(W, n - pool_lo) * m
    cap = n
    rows = sum((1 if a == 0 else 0) * min(W, n_ - lo) + (1 if a == 1 else 0) * (n_ - lo)
               for a, n_, lo in sizes)
    sets = []
    for r in range(n_sets):
        rng = synth.make_rng(30_000 + seed + r)
        tabs = [torch.from_numpy(synth.f32_to_bf16_bits(synth.normal_f32(rng, (cap, V), 3.0))
                                 .view(np.int16)).to(dev).view(torch.bfloat16) for _ in range(2)]
        tree = dict(parent=torch.full((1, cap), -1, dtype=torch.int32, device=dev),
                    token=torch.zeros(1, cap, dtype=torch.int32, device=dev),
                    edge=torch.zeros(1, cap, dtype=torch.float32, device=dev),
                    score=torch.zeros(1, cap, dtype=torch.float32, device=dev),
                    lse=torch.zeros(1, cap, dtype=torch.float32, device=dev),
                    fr=torch.empty(1, W, dtype=torch.int32, device=dev),
                    ws=tg.grow_workspace(1, cap, m, dev))
        sets.append((tabs, tree))

    def loop(tabs, t):
        for a, n_, lo in sizes:
            tg.grow_step(a, tabs[a], W, m, t["parent"], t["token"], t["edge"], t["score"], n_, lo,
                         lse_mid=t["lse"], frontier=t["fr"], ws=t["ws"], stream=stream)

    with torch.cuda.stream(stream):
        for tabs, t in sets:
            loop(tabs, t)
    stream.synchronize()
    g = capture(lambda: [loop(tabs, t) for tabs, t in sets], stream)
    g.replay()
    loops = max(5, reps // 10)
    t = time_graph(g, loops, stream) / (loops * n_sets)
    b = rows * V * 2
    return {"us": t * 1e6, "schedule": GROW_SCHEDULE, "W": W, "m": m, "vocab": V,
            "nodes_out": cap, "rows_scanned": rows, "bytes": b, "GBps": b / t / 1e9,
            "launches": 2 * len(GROW_SCHEDULE), "in_step": False,
            "note": "Algorithm 2 grow loop; bytes = drafter-table rows scanned x V x 2"}


NGRAM_PROMPT, NGRAM_MAX_N, NGRAM_M_CACHE = 2048, 4, 10


def ngram_timing(seed, dev, stream, reps, n_sets=3):
    """The n-gram small drafter (the paper's training-free small drafter)
    timed beside the step: its prefill work on a 2048-token prompt (the top-10
    cache over 2048 rows of seeded N(0, 3^2) bf16 prefill logits, 128256
    tokens, next-token bump; the order-1..4 index build), then Algorithm 2
    with its small steps: the schedule [1, 0, 1, 0, 1] with W = m = 10 (the
    middle steps on drafter tables as in the grow loop) and the all-small
    schedule [0, 0, 0, 0, 0] (Algorithm 1 with this drafter), one tree from
    the prompt's last token, n_sets rotating trees and tables."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    W = m = 10
    V, L, max_n, mc = 128256, NGRAM_PROMPT, NGRAM_MAX_N, NGRAM_M_CACHE
    rng = synth.make_rng(40_000 + seed)
    prompt = synth.prompt_stream(rng, L, V)
    gen = torch.Generator(device=dev)
    gen.manual_seed(40_000 + seed)
    lg = torch.randn(L, V, generator=gen, device=dev, dtype=torch.float32).mul_(3.0)
    nxt = torch.from_numpy(prompt[1:].astype(np.int64)).to(dev)
    hit = torch.from_numpy(rng.random(L - 1) < 0.7).to(dev)
    lg[torch.arange(L - 1, device=dev)[hit], nxt[hit]] += 8.0
    lg = lg.to(torch.bfloat16)
    toks = torch.from_numpy(prompt).to(dev)
    seq = torch.tensor([0, L], dtype=torch.int32, device=dev)
    ctok = torch.empty(L, mc, dtype=torch.int32, device=dev)
    clp = torch.empty(L, mc, dtype=torch.float32, device=dev)
    with torch.cuda.stream(stream):
        index = tg.ngram_build(toks, seq, max_n, stream=stream)
        tg.ngram_cache(lg, mc, cache_tok=ctok, cache_lp=clp, stream=stream)
    stream.synchronize()
    g_cache = capture(lambda: tg.ngram_cache(lg, mc, cache_tok=ctok, cache_lp=clp, stream=stream),
                      stream)
    g_build = capture(lambda: tg.ngram_build(toks, seq, max_n, index=index, stream=stream), stream)
    g_cache.replay()
    g_build.replay()
    t_cache = time_graph(g_cache, max(5, reps // 20), stream) / max(5, reps // 20)
    t_build = time_graph(g_build, max(5, reps // 10), stream) / max(5, reps // 10)
    ctx = torch.from_numpy(prompt[-max_n:].reshape(1, max_n).astype(np.int32)).to(dev)
    clen = torch.tensor([max_n], dtype=torch.int32, device=dev)

    def plan(schedule):
        sizes, n, new_lo, n_vis = [], 1, 0, 0
        for a in schedule:
            pool_lo = new_lo if a == 0 else n_vis
            sizes.append((a, n, pool_lo))
            if a == 1:
                n_vis = n
            new_lo, n = n, n + min(W, n - pool_lo) * m
        return sizes, n

    out = {"prompt_tokens": L, "max_n": max_n, "m_cache": mc, "vocab": V,
           "cache_us": t_cache * 1e6, "cache_bytes": L * V * 2,
           "cache_GBps": L * V * 2 / t_cache / 1e9, "build_us": t_build * 1e6,
           "build_launches": 4, "in_step": False}
    for label, schedule in (("grow_mixed", GROW_SCHEDULE), ("grow_small", [0] * 5)):
        sizes, cap = plan(schedule)
        sets = []
        for r in range(n_sets):
            rr = synth.make_rng(41_000 + seed + r)
            mid = None
            if 1 in schedule:
                mid = torch.from_numpy(synth.f32_to_bf16_bits(synth.normal_f32(rr, (cap, V), 3.0))
                                       .view(np.int16)).to(dev).view(torch.bfloat16)
            sets.append((mid, dict(
                parent=torch.full((1, cap), -1, dtype=torch.int32, device=dev),
                token=torch.zeros(1, cap, dtype=torch.int32, device=dev),
                edge=torch.zeros(1, cap, dtype=torch.float32, device=dev),
                score=torch.zeros(1, cap, dtype=torch.float32, device=dev),
                lse=torch.zeros(1, cap, dtype=torch.float32, device=dev),
                fr=torch.empty(1, W, dtype=torch.int32, device=dev),
                ws=tg.grow_workspace(1, cap, m, dev))))

        def loop(mid, t, sizes=sizes):
            for a, n_, lo in sizes:
                if a == 1:
                    tg.grow_step(1, mid, W, m, t["parent"], t["token"], t["edge"], t["score"], n_,
                                 lo, lse_mid=t["lse"], frontier=t["fr"], ws=t["ws"], stream=stream)
                else:
                    tg.ngram_grow_step(index, ctok, clp, ctx, clen, W, m, t["parent"], t["token"],
                                       t["edge"], t["score"], n_, lo, frontier=t["fr"],
                                       stream=stream)

        with torch.cuda.stream(stream):
            for mid, t in sets:
                loop(mid, t)
        stream.synchronize()
        g = capture(lambda: [loop(mid, t) for mid, t in sets], stream)
        g.replay()
        loops = max(5, reps // 10)
        t = time_graph(g, loops, stream) / (loops * n_sets)
        out[label] = {"schedule": schedule, "W": W, "m": m, "nodes_out": cap, "us": t * 1e6,
                      "launches": sum(2 if a == 1 else 1 for a in schedule)}
    return out


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, dev_index):
        self.proc = None
        self.dev_index = dev_index

    def __enter__(self):
        import torch
        sel = str(self.dev_index)
        try:
            u = str(torch.cuda.get_device_properties(self.dev_index).uuid)
            sel = u if u.startswith("GPU-") else "GPU-" + u
        except Exception:
            pass
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50", "-i", sel], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                text=True)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [ln for ln in out.splitlines() if ln.strip()]

    def summary(self):
        rows = []
        for ln in getattr(self, "lines", []):
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append(dict(sm=float(parts[1]), smax=float(parts[2]), power=float(parts[3]),
                                 hw=parts[5], hwt=parts[6], swt=parts[7], swp=parts[8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        load = [r for r in rows if r["power"] > 0] or rows
        reasons = set()
        for r in load:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("swp", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(r["sm"] for r in load),
                "sm_max_mhz": max(r["smax"] for r in load), "reasons": sorted(reasons),
                "samples": len(load), "power_w_max": max(r["power"] for r in load)}


# --------------------------------------------------------------------------- CPU baseline

CPU_SNIPPET = r"""
import json, sys, time
sys.path.insert(0, {root!r})
import numpy as np
from oracle import treegraft_oracle as O
from paper_2608_26112_gb300 import synth
wl = synth.make_workload({workload!r}, seed=0)
sh = wl["shape"]; n = len(wl["parent"])
def one_step():
    O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"], wl["parent"],
                     wl["node_off"], Hkv=sh["Hkv"])
    O.expand_topk(wl["logits"], wl["parent_score"], sh["k"], bf16=True)
    O.rescore_select(wl["weak_edge"], wl["strong_lp"], wl["parent"], wl["token"], wl["visited"],
                     wl["node_off"], sh["N"])
    O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], n, bf16=True)
for _ in range({warmup}):
    one_step()
t0 = time.perf_counter(); k = 0
while True:
    one_step(); k += 1
    el = time.perf_counter() - t0
    if (k >= {steps} and el >= {min_s}) or el >= {max_s}:
        break
print(json.dumps(dict(steps=k, seconds=el)))
"""


def run_cpu_oracle_all_cores(min_s, max_s, procs=None, steps=1, warmup=1):
    """The oracle on every host core at once: one single-threaded oracle
    process per core, each running at least `steps` whole steps and at least
    min_s seconds (at most max_s) after `warmup` untimed ones; the figure is
    the sum of their steps/s."""
    procs = procs or (os.cpu_count() or 1)
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = "1"
    env["CUDA_VISIBLE_DEVICES"] = ""
    code = CPU_SNIPPET.format(root=ROOT, workload=WORKLOAD, steps=steps, warmup=warmup,
                              min_s=min_s, max_s=max_s)
    ps = [subprocess.Popen([sys.executable, "-c", code], stdout=subprocess.PIPE,
                           stderr=subprocess.PIPE, text=True, env=env) for _ in range(procs)]
    total, steps = 0.0, 0
    for p_ in ps:
        out, err = p_.communicate(timeout=max_s * 3 + 300)
        if p_.returncode != 0:
            raise RuntimeError("CPU oracle failed: " + err[-2000:])
        d = json.loads(out.strip().splitlines()[-1])
        total += d["steps"] / d["seconds"]
        steps += d["steps"]
    return total, procs, steps


def run_cpu_oracle(steps, warmup, min_s, max_s):
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = "1"
    env["CUDA_VISIBLE_DEVICES"] = ""
    code = CPU_SNIPPET.format(root=ROOT, workload=WORKLOAD, steps=steps, warmup=warmup,
                              min_s=min_s, max_s=max_s)
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env,
                       timeout=max_s * 3 + 300)
    if r.returncode != 0:
        raise RuntimeError("CPU oracle failed: " + r.stderr[-2000:])
    d = json.loads(r.stdout.strip().splitlines()[-1])
    return d["steps"], d["seconds"]


# --------------------------------------------------------------------------- traffic record

def traffic_record(kernel):
    """dram read+write bytes per launch from the committed ncu summary, or
    None if any source the kernel is built from changed since those counters
    were taken."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        rec = json.load(f).get(kernel)
    if not rec:
        return None
    return rec["bytes_per_launch"] if sources_hash(rec["sources"]) == rec.get("sources_sha256_16") else None


def sources_hash(names):
    h = hashlib.sha256()
    for name in names:
        path = os.path.join(ROOT, "paper_2608_26112_gb300", "csrc", name)
        if not os.path.exists(path):
            return None
        with open(path, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


# --------------------------------------------------------------------------- arms

def dist_setup(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return world, rank, local


def rank_seed(seed, rank):
    """Each rank draws its own sequences: the ranks share no input and the
    step has no exchange between them."""
    return seed + 1000 * rank


def max_over_ranks(x, world):
    """Slowest rank's time (the job's time): an all-reduce of one float on
    the host side of the timing, never inside the timed step."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world, steps, t_max):
    """Whole-job steps/s: every rank runs `steps` steps of its own sequences."""
    return world * steps / t_max


def barrier(world):
    import torch
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    if torch.cuda.is_available():
        torch.cuda.synchronize()


def reference_arm(args):
    """The reference arm of this build: the oracle (plain fp64 numpy, the
    paper's definitions) on the host cores, one single-threaded process per
    core running whole steps of the workload at once.  The K timed steps are
    shared out over the processes (ceil(K / cores) each, after up to 3
    warm-up steps each); a process stops early once its timed steps pass
    120 s, so large K stays bounded, and the line then counts the steps that
    ran."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    K, W = max(1, args.steps), max(0, args.warmup)
    procs = os.cpu_count() or 1
    per = -(-K // procs)
    warm = min(W, 3)
    v, n_proc, steps = run_cpu_oracle_all_cores(0.0, 120.0, procs=procs, steps=per, warmup=warm)
    timed = min(K, steps)
    note = "" if steps >= K else f" (stopped at 120 s per process: {steps} of {K} steps)"
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "steps/s",
            "n_gpus": args.gpus, "steps": timed, "warmup": warm,
            "ms_per_step": 1e3 / v, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "note": "oracle (plain fp64 numpy) on host cores"},
            "cpu_baseline": {"value": v, "unit": "steps/s", "cores": n_proc, "kind": "oracle",
                             "sample": f"{steps} full steps of {WORKLOAD} ({per} per process): "
                                       f"{n_proc} single-threaded oracle processes at once, "
                                       f"{warm} warm-up steps each{note}"},
            "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def ours_arm(args):
    import numpy as np
    import torch

    world, rank, local = dist_setup(args)
    from paper_2608_26112_gb300 import build as _b
    if rank == 0:
        _b.build()
    if world > 1:
        barrier(world)
    import paper_2608_26112_gb300 as tg
    from paper_2608_26112_gb300 import synth

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    R = args.sets
    sets, host = build_sets(R, rank_seed(args.seed, rank), dev)
    sh = host[0]["shape"]
    outs = [alloc_outputs(d, sh, dev) for d in sets]
    stream = torch.cuda.Stream(device=dev)

    # warm-up through the plain API (also initialises the library's caches)
    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            step(sets[i % R], outs[i % R], sh)
    stream.synchronize()
    assert tg.last_device_status(stream) == 0

    cycle = capture(lambda: [step(sets[r], outs[r], sh) for r in range(R)], stream)
    singles = [capture(lambda r=r: step(sets[r], outs[r], sh), stream) for r in range(R)]
    per_kernel_graphs = {name: capture(lambda name=name: [call(name, sets[r], outs[r], sh)
                                                         for r in range(R)], stream)
                         for name in KERNELS + BESIDE}
    for _ in range(3):
        cycle.replay()
    torch.cuda.synchronize()

    K, W = args.steps, args.warmup
    q, rem = divmod(K, R)
    clocks = ClockSampler(dev.index)
    with clocks:
        # ---- timed region: exactly K steps, repeated REPEATS times; the
        #      median repeat is the reported time, the spread is kept
        reps_t = []
        for _ in range(REPEATS):
            barrier(world)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                e0.record(stream)
                for _ in range(q):
                    cycle.replay()
                for r in range(rem):
                    singles[r].replay()
                e1.record(stream)
            e1.synchronize()
            barrier(world)
            reps_t.append(e0.elapsed_time(e1) / 1e3)
        t_steps = statistics.median(reps_t)
        # ---- per-kernel launch durations (each graph = R launches over the R sets)
        kreps = max(20, min(2000, int(0.25 / max(1e-6, t_steps / max(1, K)) / R)))
        kt = {}
        for name, g in per_kernel_graphs.items():
            g.replay()
            kt[name] = time_graph(g, kreps, stream) / (kreps * R)
        prune = prune_timing(R, rank_seed(args.seed, rank), dev, stream, kreps)
        grow = grow_timing(rank_seed(args.seed, rank), dev, stream, kreps)
        ngram = ngram_timing(rank_seed(args.seed, rank), dev, stream, kreps)
        extra = {nm: config_timing(nm, rank_seed(args.seed, rank), dev, stream)
                 for nm in EXTRA_CONFIGS}
        extra["graft-mha-pipeline"] = graft_pipeline_timing(rank_seed(args.seed, rank), dev, stream)
        if not args.no_serving:
            extra["serving-sweep"] = [serving_timing(B, dev, stream) for B in SERVING_BATCHES]
    assert tg.last_device_status(stream) == 0
    t_max = max_over_ranks(t_steps, world)
    steps_per_s = job_throughput(world, K, t_max)
    spread = [job_throughput(world, K, max_over_ranks(t, world)) for t in (max(reps_t), min(reps_t))]

    pk, pk_src = peaks()
    hbm = pk["hbm_gbs"]
    costs = algorithmic_costs(host[0])
    kernels = {}
    for name in KERNELS:
        b, f = costs[name]
        kernels[name] = {"us": kt[name] * 1e6, "bytes": b, "GBps": b / kt[name] / 1e9,
                         "hbm_frac": b / kt[name] / 1e9 / hbm}
        if f:
            kernels[name]["TFLOPs"] = f / kt[name] / 1e12
    b = costs["accept"][0]
    kernels["accept_sample"] = {"us": kt["accept_sample"] * 1e6, "bytes": b,
                                "GBps": b / kt["accept_sample"] / 1e9,
                                "hbm_frac": b / kt["accept_sample"] / 1e9 / hbm,
                                "temperature": SAMPLE_T, "launches": 1, "in_step": False,
                                "note": "verification at T > 0: every node row once"}
    kernels["global_prune"] = prune
    kernels["grow_loop"] = grow
    kernels["ngram_drafter"] = ngram
    dom = max(KERNELS, key=lambda n: kt[n])
    b, f = costs[dom]
    achieved = b / kt[dom] / 1e9
    roofline = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "traffic": traffic_record(dom),
                "peak_source": f"{pk_src} hbm_gbs (burst copy)",
                "algorithmic_bytes_per_launch": b}
    attn_b, attn_f = costs["tree_attn"]
    t_attn = kt["tree_attn"]
    roof_t = max(attn_b / (hbm * 1e9), attn_f / (pk["bf16_tflops"] * 1e12))
    kernels["tree_attn"]["roofline_frac"] = roof_t / t_attn
    kernels["tree_attn"]["roofline_frac_8TBps_nominal"] = max(attn_b / 8e12, attn_f / (pk["bf16_tflops"] * 1e12)) / t_attn

    # ---- end to end through the public API with host buffers
    e2e = end_to_end(host, sh, dev, stream, reps=max(20, min(200, K // 10 or 20)))

    line = {"metric": METRIC, "value": steps_per_s, "unit": "steps/s", "n_gpus": world,
            "steps": K, "warmup": W, "ms_per_step": 1e3 * t_max / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "batch": 1, "prefix": int(host[0]["prefix_len"][0]),
                       "tree_nodes": len(host[0]["parent"]), "tree_depth": sh["depth"],
                       "heads_q_kv": f"{sh['Hq']}/{sh['Hkv']}", "head_dim": sh["D"],
                       "vocab": sh["V"], "topk": sh["k"], "reselect_N": sh["N"],
                       "l2": f"{R} rotating input sets, ~{R * 40} MB touched per cycle "
                             + ("> 126 MB L2" if R * 40 > 126 else "(fits in L2)"),
                       "parallelism": f"independent sequences per GPU x{world}"},
            "roofline": roofline, "kernels": kernels, "other_workloads": extra, "e2e": e2e,
            "gpu_launches": K * len(KERNELS), "clocks": clocks.summary(),
            "repeats": {"count": REPEATS, "statistic": "median", "steps_per_s_min": spread[0],
                        "steps_per_s_max": spread[1]}}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        steps_c, sec = run_cpu_oracle(3, 1, 10.0, 30.0)
        v_all, n_proc, steps_all = run_cpu_oracle_all_cores(10.0, 30.0)
        line["cpu_baseline"] = {"value": v_all, "unit": "steps/s", "cores": n_proc,
                                "kind": "oracle",
                                "sample": f"{steps_all} full steps of {WORKLOAD}: {n_proc} "
                                          "single-threaded oracle processes at once, 10-30 s each",
                                "single_core": {"value": steps_c / sec, "unit": "steps/s",
                                                "cores": 1, "sample": f"{steps_c} full steps"}}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def end_to_end(host, sh, dev, stream, reps):
    """Steps/s through the public API with inputs copied from pinned host
    memory every step and the step's results read back.  Served as a
    pipeline: two device input buffers, the copies for step i+1 spread over
    four copy streams while step i computes; every step still moves all of
    its inputs host->device and its results device->host."""
    import numpy as np
    import torch
    import paper_2608_26112_gb300 as tg

    wl = host[0]

    def pin(a, dtype=None):
        t = torch.from_numpy(np.ascontiguousarray(a))
        if dtype is not None:
            t = t.view(dtype)
        return t.pin_memory()

    hs = dict(q=pin(wl["q"].view(np.int16), torch.bfloat16),
              k=pin(wl["k_cache"].view(np.int16), torch.bfloat16),
              v=pin(wl["v_cache"].view(np.int16), torch.bfloat16),
              prefix_len=pin(wl["prefix_len"]), parent=pin(wl["parent"]), token=pin(wl["token"]),
              node_off=pin(wl["node_off"]), logits=pin(wl["logits"].view(np.int16), torch.bfloat16),
              target=pin(wl["target_logits"].view(np.int16), torch.bfloat16),
              parent_score=pin(wl["parent_score"]), weak_edge=pin(wl["weak_edge"]),
              visited=pin(wl["visited"]))
    from paper_2608_26112_gb300 import synth
    hs["strong"] = pin(synth.make_workload(WORKLOAD, seed=0, with_logits=False)["strong_lp"])
    nbuf, ncopy = 2, 4
    d = [{k: torch.empty(v.shape, dtype=v.dtype, device=dev) for k, v in hs.items()}
         for _ in range(nbuf)]
    o = [alloc_outputs(d[i], sh, dev) for i in range(nbuf)]
    res_names = ["o", "tok", "lp", "sc", "edge", "score", "sel", "nsel", "path", "alen", "bonus"]
    res_h = [{k: torch.empty(o[0][k].shape, dtype=o[0][k].dtype).pin_memory() for k in res_names}
             for _ in range(nbuf)]
    h2d = sum(v.numel() * v.element_size() for v in hs.values())
    d2h = sum(v.numel() * v.element_size() for v in res_h[0].values())
    # spread the tensors over the copy streams by size (largest first)
    lanes = [[] for _ in range(ncopy)]
    load = [0] * ncopy
    for k_, v in sorted(hs.items(), key=lambda kv: -kv[1].numel() * kv[1].element_size()):
        j = load.index(min(load))
        lanes[j].append(k_)
        load[j] += v.numel() * v.element_size()
    cstreams = [torch.cuda.Stream(device=dev) for _ in range(ncopy)]
    freed = [torch.cuda.Event() for _ in range(nbuf)]      # buffer i no longer read
    copied = [[torch.cuda.Event() for _ in range(ncopy)] for _ in range(nbuf)]

    def copy_in(i):
        for j, cs in enumerate(cstreams):
            cs.wait_event(freed[i])
            with torch.cuda.stream(cs):
                for k_ in lanes[j]:
                    d[i][k_].copy_(hs[k_], non_blocking=True)
            copied[i][j].record(cs)

    def compute(i):
        for j in range(ncopy):
            stream.wait_event(copied[i][j])
        with torch.cuda.stream(stream):
            step(d[i], o[i], sh)
            for k_ in res_names:
                res_h[i][k_].copy_(o[i][k_], non_blocking=True)
        freed[i].record(stream)

    def run(n):
        for i in range(nbuf):
            freed[i].record(stream)
        copy_in(0)
        for s_ in range(n):
            if s_ + 1 < n:
                copy_in((s_ + 1) % nbuf)
            compute(s_ % nbuf)

    run(4)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for cs in cstreams:
        cs.wait_event(e0)
    run(reps)
    e1.record(stream)
    e1.synchronize()
    t = e0.elapsed_time(e1) / 1e3
    return {"value": reps / t, "unit": "steps/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": reps,
            "pipeline": f"{nbuf} input buffers, {ncopy} copy streams, copies of step i+1 "
                        "overlap step i"}


def main():
    args = parse()
    if args.impl == "reference":
        reference_arm(args)
    else:
        ours_arm(args)


if __name__ == "__main__":
    main()
