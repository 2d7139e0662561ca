"""Parity of the CUDA path (through the C ABI) with the CPU oracle on seeded
synthetic inputs.  Bars: top-k indices, reselected sets and accepted paths
bit-exact (ties to the lower token / node id); attention max-abs 2e-2 and
mean-abs 2e-3 on bf16 outputs; path scores 1e-4 relative."""
import numpy as np
import pytest
import torch

import paper_2608_26112_gb300 as tg
from oracle import treegraft_oracle as O
from paper_2608_26112_gb300 import synth
from tests import _dev

pytestmark = pytest.mark.gpu

ATT_MAX_ABS, ATT_MEAN_ABS, LSE_ABS = 2e-2, 2e-3, 2e-3
SCORE_RTOL = 1e-4


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26112_gb300 import build
    build.build()
    return torch.device("cuda:0")


def _status_clean():
    assert tg.last_device_status() == 0


# ------------------------------------------------------------------ tree attention

def _attn_shape(B, P, n, depth, Hq, Hkv, D, cap=None):
    return dict(B=B, P=P, n=n, depth=depth, cap=cap, rank_bias=0.3, Hq=Hq, Hkv=Hkv, D=D, V=64,
                logit_dtype="f32", k=4, N=4)


ATTN_CASES = {
    "tiny": "tiny",
    "graft-mha": "graft-mha",
    "llama3-8b-verify": "llama3-8b-verify",
    "g1-d64-p1-n2": _attn_shape(1, 1, 2, 1, 4, 4, 64),
    "g2-d128-p127-n33": _attn_shape(1, 127, 33, 5, 8, 4, 128),
    "g8-d128-p129-n255": _attn_shape(1, 129, 255, 9, 64, 8, 128, cap=16),
    "g4-d64-p0-n256": _attn_shape(1, 0, 256, 8, 16, 4, 64),
    "g4-d128-n1": _attn_shape(2, [300, 17], [1, 1], 1, 32, 8, 128),
    "ragged-b3": _attn_shape(3, [5, 300, 1000], [2, 64, 128], [1, 6, 8], 32, 8, 128, cap=10),
    "n31-n32": _attn_shape(2, [128, 256], [31, 32], [3, 4], 16, 8, 64),
    "g8-d64-b2": _attn_shape(2, [64, 200], [40, 50], [5, 6], 64, 8, 64, cap=10),
    # head size 64 with the keys split over CTAs: cooperative (GQA) and cluster (MHA) paths
    "split-d64-gqa": _attn_shape(1, 4000, 60, 6, 32, 8, 64),
    "split-coop-d64": _attn_shape(1, 8000, 60, 6, 32, 8, 64),
    "split-cluster-d64-mha": _attn_shape(1, 1500, 64, 7, 32, 32, 64),
    # one split over four query tiles of 128 rows: the 33-, 64- and 1-node
    # trees leave tiles with no rows, the 33-node tree one with four
    "ragged-b4-empty-tiles": _attn_shape(4, [300, 17, 1000, 5], [33, 100, 64, 1], [5, 7, 6, 1], 32, 8,
                                128, cap=10),
}


def _run_attn(wl, dev):
    sh = wl["shape"]
    q = _dev.bf16(wl["q"], dev)
    k = _dev.bf16(wl["k_cache"], dev)
    v = _dev.bf16(wl["v_cache"], dev)
    lse = torch.full((q.shape[0], q.shape[1]), float("nan"), device=dev)
    out, _ = tg.tree_attn(q, k, v, _dev.i32(wl["prefix_len"], dev), _dev.i32(wl["parent"], dev),
                          _dev.i32(wl["node_off"], dev), _dev.max_nodes(wl), lse_out=lse)
    _status_clean()
    return _dev.bf16_to_np(out), lse.cpu().numpy().astype(np.float64)


def _check_attn(wl, o, lse, oracle_o, oracle_lse):
    err = np.abs(o - oracle_o)
    assert np.isfinite(o).all()
    assert err.max() <= ATT_MAX_ABS, err.max()
    assert err.mean() <= ATT_MEAN_ABS, err.mean()
    np.testing.assert_allclose(lse, oracle_lse, atol=LSE_ABS, rtol=0)


@pytest.mark.parametrize("case", list(ATTN_CASES))
def test_tree_attn_matches_oracle(dev, case):
    wl = synth.make_workload(ATTN_CASES[case], seed=1, with_logits=False, with_strong=False)
    o, lse = _run_attn(wl, dev)
    ref_o, ref_lse = O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"],
                                      wl["parent"], wl["node_off"], Hkv=wl["shape"]["Hkv"])
    _check_attn(wl, o, lse, ref_o, ref_lse)


def test_tree_attn_ignores_nan_past_the_sequence(dev):
    wl = synth.make_workload(_attn_shape(2, [100, 61], [20, 67], [3, 5], 16, 4, 128), seed=2,
                             kv_tail="nan", with_logits=False, with_strong=False, S_max=300)
    o, lse = _run_attn(wl, dev)
    ref_o, ref_lse = O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"],
                                      wl["parent"], wl["node_off"], Hkv=4)
    _check_attn(wl, o, lse, ref_o, ref_lse)


def test_tree_attn_split_kernel_nan_one_row_into_the_last_tile(dev):
    # one tree, keys 1000 + 25 = 1025: the last key tile holds one real row,
    # so 127 V rows past the end (NaN here) are zeroed before its PV product,
    # in a launch whose keys are split over several CTAs
    wl = synth.make_workload(_attn_shape(1, 1000, 25, 5, 32, 8, 128), seed=5, kv_tail="nan",
                             with_logits=False, with_strong=False, S_max=1200)
    o, lse = _run_attn(wl, dev)
    ref_o, ref_lse = O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"],
                                      wl["parent"], wl["node_off"], Hkv=8)
    _check_attn(wl, o, lse, ref_o, ref_lse)


def test_tree_attn_whole_units_ignore_nan_past_the_sequence(dev):
    # 2 trees x 8 kv-heads x 10 row tiles of 128 (G 8, 160 nodes) fill a wave
    # of 152 SMs, so the whole-unit kernel runs; KV rows past each sequence
    # hold NaN, and each sequence ends inside a key tile
    wl = synth.make_workload(_attn_shape(2, [300, 517], [160, 100], [7, 6], 64, 8, 128, cap=16),
                             seed=4, kv_tail="nan", with_logits=False, with_strong=False, S_max=800)
    o, lse = _run_attn(wl, dev)
    ref_o, ref_lse = O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"],
                                      wl["parent"], wl["node_off"], Hkv=8)
    _check_attn(wl, o, lse, ref_o, ref_lse)


def test_tree_attn_chain_equals_causal(dev):
    # chain tree: the kernel's result must equal causal attention (oracle pin)
    shape = _attn_shape(1, 200, 40, 39, 32, 8, 128)
    wl = synth.make_workload(shape, seed=3, with_logits=False, with_strong=False)
    wl["parent"] = np.arange(-1, 39, dtype=np.int32)
    o, lse = _run_attn(wl, dev)
    ref_o, ref_lse = O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"],
                                      wl["parent"], wl["node_off"], Hkv=8)
    _check_attn(wl, o, lse, ref_o, ref_lse)


def test_tree_attn_llama70b_shape_sampled(dev):
    # full 4 x (8192 + 128) Llama-3-70B-shaped launch; oracle on trees 0 and 3
    wl = synth.make_workload("llama3-70b-verify", seed=0, with_logits=False, with_strong=False)
    o, lse = _run_attn(wl, dev)
    off = wl["node_off"]
    for b in (0, 3):
        a, e = int(off[b]), int(off[b + 1])
        ref_o, ref_lse = O.tree_attention(wl["q"][a:e], wl["k_cache"][b:b + 1],
                                          wl["v_cache"][b:b + 1], wl["prefix_len"][b:b + 1],
                                          wl["parent"][a:e], [0, e - a], Hkv=8)
        _check_attn(wl, o[a:e], lse[a:e], ref_o, ref_lse)


@pytest.mark.parametrize("name", ["llama3-8b-verify", "llama3-70b-verify"])
def test_tree_attn_rows_outside_every_tree_set_status(dev, name):
    """node_off whose last entry falls short of n_total (rows in no tree) sets
    TG_ERR_DEVICE_TREE, in the split kernel (one tree) and in the whole-unit
    kernel (a batch), and the next well-formed call is exact."""
    wl = synth.make_workload(name, seed=12, with_logits=False, with_strong=False)
    short = wl["node_off"].copy()
    short[-1] -= 3
    q = _dev.bf16(wl["q"], dev)
    k, v = _dev.bf16(wl["k_cache"], dev), _dev.bf16(wl["v_cache"], dev)
    tg.tree_attn(q, k, v, _dev.i32(wl["prefix_len"], dev), _dev.i32(wl["parent"], dev),
                 _dev.i32(short, dev), _dev.max_nodes(wl))
    assert tg.last_device_status() & 4
    o, lse = _run_attn(wl, dev)
    off = wl["node_off"]
    b = len(off) - 2                      # the last tree, the one the short extent cut
    a, e = int(off[b]), int(off[b + 1])
    ref_o, ref_lse = O.tree_attention(wl["q"][a:e], wl["k_cache"][b:b + 1], wl["v_cache"][b:b + 1],
                                      wl["prefix_len"][b:b + 1], wl["parent"][a:e], [0, e - a],
                                      Hkv=wl["shape"]["Hkv"])
    _check_attn(wl, o[a:e], lse[a:e], ref_o, ref_lse)


def test_tree_attn_malformed_tree_sets_status(dev):
    wl = synth.make_workload(_attn_shape(1, 16, 8, 3, 8, 8, 64), seed=4, with_logits=False,
                             with_strong=False)
    bad = wl["parent"].copy()
    bad[5] = 6                                           # parent after child
    q = _dev.bf16(wl["q"], dev)
    out = torch.zeros_like(q)
    tg.tree_attn(q, _dev.bf16(wl["k_cache"], dev), _dev.bf16(wl["v_cache"], dev),
                 _dev.i32(wl["prefix_len"], dev), _dev.i32(bad, dev),
                 _dev.i32(wl["node_off"], dev), 8, out=out)
    assert tg.last_device_status() & 4
    assert tg.last_device_status() == 0                  # cleared by the read


def test_tree_attn_split_wait_runs_out_and_recovers(dev):
    """The split barrier of tree_attn is a bounded wait on other thread
    blocks, on counters in the caller's workspace.  A workspace whose first
    counter holds a value the splits can never bring up to their count (as a
    corrupted workspace would) makes every split of that unit give up after
    a short budget: the call returns, TG_ERR_TIMEOUT is set, the unit's two
    counters are back at zero and the next call on the same workspace is
    exact.  Nothing waits without a bound, so no GPU hang is involved."""
    wl = synth.make_workload("llama3-8b-verify", seed=5, with_logits=False, with_strong=False)
    sh = wl["shape"]
    q = _dev.bf16(wl["q"], dev)
    k, v = _dev.bf16(wl["k_cache"], dev), _dev.bf16(wl["v_cache"], dev)
    pl, par, off = (_dev.i32(wl["prefix_len"], dev), _dev.i32(wl["parent"], dev),
                    _dev.i32(wl["node_off"], dev))
    n = len(wl["parent"])
    nbytes = tg.tree_attn_workspace_size(1, n, sh["Hq"], sh["Hkv"], sh["D"])
    assert nbytes > 0                                    # this shape runs a split plan
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    ws.view(torch.int32)[0] = -1000                      # unit 0's arrival counter
    tg.set_wait_budget(20_000)                           # ~10 us at the GB300's clock
    try:
        tg.tree_attn(q, k, v, pl, par, off, n, ws=ws)
        torch.cuda.synchronize()
        st = tg.last_device_status()
    finally:
        tg.set_wait_budget(0)
    assert st & 8, st                                    # TG_ERR_TIMEOUT
    assert ws.view(torch.int32)[:2].tolist() == [0, 0]   # counters returned to zero
    lse = torch.empty(n, sh["Hq"], device=dev)
    o, _ = tg.tree_attn(q, k, v, pl, par, off, n, ws=ws, lse_out=lse)
    _status_clean()
    ref_o, ref_lse = O.tree_attention(wl["q"], wl["k_cache"], wl["v_cache"], wl["prefix_len"],
                                      wl["parent"], wl["node_off"], Hkv=sh["Hkv"])
    _check_attn(wl, _dev.bf16_to_np(o), lse.cpu().numpy().astype(np.float64), ref_o, ref_lse)


# ------------------------------------------------------------------ expand_topk

def _run_expand(lg_dev, ps, k, dev, row_idx=None, V=None):
    rows = len(ps)
    lse = torch.empty(rows, device=dev)
    tok, lp, sc, _ = tg.expand_topk(lg_dev, _dev.f32(ps, dev), k,
                                    row_idx=None if row_idx is None else _dev.i32(row_idx, dev),
                                    V=V, lse_out=lse)
    _status_clean()
    return tok.cpu().numpy(), lp.cpu().numpy(), sc.cpu().numpy(), lse.cpu().numpy()


def _check_expand(got, ref):
    tok, lp, sc, lse = got
    rtok, rlp, rsc, rlse = ref
    np.testing.assert_array_equal(tok, rtok)
    np.testing.assert_allclose(lp, rlp, rtol=SCORE_RTOL, atol=1e-5)
    np.testing.assert_allclose(sc, rsc, rtol=SCORE_RTOL, atol=1e-5)
    np.testing.assert_allclose(lse, rlse, rtol=1e-5, atol=1e-5)


@pytest.mark.parametrize("name", ["tiny", "llama3-8b-verify", "graft-mha"])
def test_expand_topk_workloads(dev, name):
    wl = synth.make_workload(name, seed=0, with_strong=False)
    bf = wl["logits"].dtype == np.uint16
    k = wl["shape"]["k"]
    got = _run_expand(_dev.logits(wl, dev), wl["parent_score"], k, dev)
    ref = O.expand_topk(wl["logits"], wl["parent_score"], k, bf16=bf)
    _check_expand(got, ref)


@pytest.mark.parametrize("V,ld,dtype,k", [(1023, 1024, "f32", 5), (32001, 32001, "bf16", 10),
                                          (32001, 32008, "bf16", 32), (777, 801, "f32", 1),
                                          (100, 100, "bf16", 32), (262144, 262144, "bf16", 16)])
def test_expand_topk_ragged_vocab(dev, V, ld, dtype, k):
    rng = synth.make_rng(V + k)
    rows = 7
    x = synth.normal_f32(rng, (rows, ld), 3.0)
    ps = synth.normal_f32(rng, (rows,), 2.0)
    if dtype == "bf16":
        bits = synth.f32_to_bf16_bits(x)
        got = _run_expand(_dev.bf16(bits, dev), ps, k, dev, V=V)
        ref = O.expand_topk(bits[:, :V], ps, k, bf16=True)
    else:
        got = _run_expand(_dev.f32(x, dev), ps, k, dev, V=V)
        ref = O.expand_topk(x[:, :V], ps, k)
    _check_expand(got, ref)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_expand_topk_ties_inf_and_row_idx(dev, dtype):
    # heavy ties overflow the candidate buffer and take the exact-key fallback
    rng = synth.make_rng(5)
    V = 5000 if dtype == "f32" else 40000
    x = rng.integers(-1, 2, size=(6, V)).astype(np.float32)     # heavy ties
    x[2] = -np.inf                                              # all -inf row
    x[3, ::3] = -np.inf
    x[4] = 0.0
    x[5, :] = -0.0
    x[5, 17] = 0.0
    x[4, V - 1] = 0.5
    ps = np.array([0, -1, -2, -3, -4, -5, -6, -7], np.float32)
    row_idx = np.array([5, 4, 3, 0, 1, 0, 2, 2], np.int32)
    if dtype == "f32":
        got = _run_expand(_dev.f32(x, dev), ps, 12, dev, row_idx=row_idx)
        ref = O.expand_topk(x, ps, 12, row_idx=row_idx)
    else:
        bits = synth.f32_to_bf16_bits(x)
        got = _run_expand(_dev.bf16(bits, dev), ps, 12, dev, row_idx=row_idx)
        ref = O.expand_topk(bits, ps, 12, row_idx=row_idx, bf16=True)
    np.testing.assert_array_equal(got[0], ref[0])
    for g, r in zip(got[1:], ref[1:]):
        np.testing.assert_array_equal(np.isneginf(g), np.isneginf(r))
        fin = np.isfinite(r)
        np.testing.assert_allclose(g[fin], r[fin], rtol=1e-5, atol=1e-5)


def test_expand_topk_bad_row_idx_sets_status(dev):
    x = torch.zeros(4, 64, device=dev)
    tg.expand_topk(x, torch.zeros(2, device=dev), 3, row_idx=_dev.i32([1, 9], dev))
    assert tg.last_device_status() & 16


# ------------------------------------------------------------------ rescore_select

def _run_rescore(wl, N, dev, visited=None):
    vis = wl["visited"] if visited is None else visited
    e, s, sel, ns = tg.rescore_select(_dev.f32(wl["weak_edge"], dev), _dev.f32(wl["strong_lp"], dev),
                                      _dev.i32(wl["parent"], dev), _dev.i32(wl["token"], dev),
                                      _dev.u8(vis, dev), _dev.i32(wl["node_off"], dev),
                                      _dev.max_nodes(wl), N)
    _status_clean()
    return e.cpu().numpy(), s.cpu().numpy(), sel.cpu().numpy(), ns.cpu().numpy()


@pytest.mark.parametrize("name,visited", [("tiny", None), ("llama3-8b-verify", None),
                                          ("graft-mha", "none"), ("graft-mha", "all"),
                                          ("llama3-70b-verify", None)])
def test_rescore_select_bit_exact(dev, name, visited):
    wl = synth.make_workload(name, seed=0, with_logits=False)
    vis = {None: wl["visited"], "none": np.zeros_like(wl["visited"]),
           "all": np.ones_like(wl["visited"])}[visited]
    N = wl["shape"]["N"]
    got = _run_rescore(wl, N, dev, vis)
    ref = O.rescore_select(wl["weak_edge"], wl["strong_lp"], wl["parent"], wl["token"], vis,
                           wl["node_off"], N)
    for g, r in zip(got, ref):
        np.testing.assert_array_equal(g, r)


@pytest.mark.parametrize("name", ["llama3-8b-verify", "llama3-70b-verify"])
def test_rescore_select_rows_outside_every_tree_set_status(dev, name):
    """node_off that leaves rows in no tree (node_off[B] < n_total) sets
    TG_ERR_DEVICE_TREE (the trees within their own extents are still
    computed), and the next well-formed call is exact."""
    wl = synth.make_workload(name, seed=5, with_logits=False)
    N = wl["shape"]["N"]
    short = wl["node_off"].copy()
    short[-1] -= 2
    e, s, sel, ns = tg.rescore_select(_dev.f32(wl["weak_edge"], dev), _dev.f32(wl["strong_lp"], dev),
                                      _dev.i32(wl["parent"], dev), _dev.i32(wl["token"], dev),
                                      _dev.u8(wl["visited"], dev), _dev.i32(short, dev),
                                      _dev.max_nodes(wl), N)
    assert tg.last_device_status() & 4
    got = _run_rescore(wl, N, dev)
    ref = O.rescore_select(wl["weak_edge"], wl["strong_lp"], wl["parent"], wl["token"],
                           wl["visited"], wl["node_off"], N)
    for g, r in zip(got, ref):
        np.testing.assert_array_equal(g, r)


# ------------------------------------------------------------------ accept

def _run_accept(wl, dev, path_cap, lg=None):
    B = len(wl["node_off"]) - 1
    ws = tg.accept_workspace(B, len(wl["parent"]), dev)
    lg = _dev.logits(wl, dev) if lg is None else lg
    path, alen, bonus = tg.accept(lg, _dev.i32(wl["token"], dev), _dev.i32(wl["parent"], dev),
                                  _dev.i32(wl["node_off"], dev), _dev.max_nodes(wl), path_cap, ws)
    _status_clean()
    return path.cpu().numpy(), alen.cpu().numpy(), bonus.cpu().numpy(), ws


@pytest.mark.parametrize("name,bump", [("tiny", 8.0), ("tiny", 40.0), ("llama3-8b-verify", 8.0),
                                       ("llama3-8b-verify", 40.0), ("llama3-70b-verify", 40.0),
                                       ("graft-mha", 40.0)])
def test_accept_bit_exact(dev, name, bump):
    wl = synth.make_workload(name, seed=7, with_strong=False)
    if bump != 8.0:
        # re-plant with a larger bump so that long accepted paths occur
        wl = synth.make_workload(name, seed=7, with_strong=False, with_logits=False)
        rng = synth.make_rng(99)
        lg = synth.normal_f32(rng, (len(wl["parent"]), wl["shape"]["V"]), 3.0)
        off = wl["node_off"]
        for b in range(len(off) - 1):
            a, e = int(off[b]), int(off[b + 1])
            synth.plant_child_bump(rng, lg, wl["parent"][a:e], wl["token"][a:e], np.arange(a, e),
                                   prob=0.9, bump=bump)
        wl["logits"] = lg if wl["shape"]["logit_dtype"] == "f32" else synth.f32_to_bf16_bits(lg)
    bf = wl["logits"].dtype == np.uint16
    cap = _dev.max_nodes(wl)
    got = _run_accept(wl, dev, cap)
    ref = O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], cap, bf16=bf)
    for g, r in zip(got[:3], ref):
        np.testing.assert_array_equal(g, r)
    if bump == 40.0:
        assert ref[1].max() >= 1        # a planted child was accepted
    # the workspace is ready for a second call: same answer
    got2 = _run_accept(wl, dev, cap)
    for g, r in zip(got2[:3], ref):
        np.testing.assert_array_equal(g, r)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_accept_tied_logits(dev, dtype):
    # quantised target logits: every row's argmax is decided by the lowest-token rule
    wl = synth.make_workload("llama3-8b-verify", seed=11, with_logits=False, with_strong=False)
    rng = synth.make_rng(12)
    V = 50000
    x = rng.integers(-1, 2, size=(len(wl["parent"]), V)).astype(np.float32)
    x[:, :3] = -1.0
    wl["logits"] = x if dtype == "f32" else synth.f32_to_bf16_bits(x)
    cap = _dev.max_nodes(wl)
    got = _run_accept(wl, dev, cap)
    ref = O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], cap,
                   bf16=(dtype == "bf16"))
    for g, r in zip(got[:3], ref):
        np.testing.assert_array_equal(g, r)


def test_accept_path_cap_too_small_sets_status(dev):
    n, V = 6, 50
    parent = np.arange(-1, n - 1, dtype=np.int32)
    token = np.arange(n, dtype=np.int32) + 3
    x = np.zeros((n, V), np.float32)
    for v in range(n - 1):
        x[v, token[v + 1]] = 5.0
    wl = dict(parent=parent, token=token, node_off=np.array([0, n], np.int32), logits=x)
    ws = tg.accept_workspace(1, n, dev)
    tg.accept(_dev.f32(x, dev), _dev.i32(token, dev), _dev.i32(parent, dev),
              _dev.i32(wl["node_off"], dev), n, 3, ws)
    assert tg.last_device_status() & 16
    path, A, bonus, _ = _run_accept(wl, dev, n)
    assert A[0] == n - 1 and list(path[0]) == list(range(n))


@pytest.mark.parametrize("where", ["short-end", "late-start"])
def test_accept_rows_outside_every_tree_set_status(dev, where):
    """node_off that does not cover [0, n_total): the uncovered rows belong to
    no tree, raise TG_ERR_DEVICE_TREE and draw no ticket, so the workspace
    counters stay clean and the next well-formed call is exact."""
    wl = synth.make_workload("llama3-70b-verify", seed=21,
                             with_strong=False)
    off = wl["node_off"].copy()
    bad = off.copy()
    if where == "short-end":
        bad[-1] -= 3          # the last three rows are in no tree
    else:
        bad[0] = 2            # rows 0 and 1 are in no tree
    lg = _dev.logits(wl, dev)
    B, n_total = len(off) - 1, len(wl["parent"])
    ws = tg.accept_workspace(B, n_total, dev)
    tok, par = _dev.i32(wl["token"], dev), _dev.i32(wl["parent"], dev)
    cap = _dev.max_nodes(wl)
    tg.accept(lg, tok, par, _dev.i32(bad, dev), cap, cap, ws)
    assert tg.last_device_status() & 4
    got = tg.accept(lg, tok, par, _dev.i32(off, dev), cap, cap, ws)
    _status_clean()
    ref = O.accept(wl["logits"], wl["token"], wl["parent"], off, cap, bf16=True)
    for g, r in zip(got, ref):
        np.testing.assert_array_equal(g.cpu().numpy(), r)


def test_accept_one_workspace_serves_any_shape(dev):
    """The walk returns every ticket and argmax slot of a well-formed call to
    zero, even when the tree's path does not fit path_cap, so one workspace
    sized for the largest call serves later calls of other B and n_total
    (their tickets then sit where an earlier call kept argmax slots)."""
    big = synth.make_workload("llama3-70b-verify", seed=31, with_strong=False)
    ws = tg.accept_workspace(len(big["node_off"]) - 1, len(big["parent"]), dev)
    for name, seed, cap in (("llama3-70b-verify", 31, None), ("tiny", 32, 2),
                            ("llama3-8b-verify", 33, None), ("tiny", 34, None)):
        wl = synth.make_workload(name, seed=seed, with_strong=False)
        bf = wl["logits"].dtype == np.uint16
        full = _dev.max_nodes(wl)
        got = tg.accept(_dev.logits(wl, dev), _dev.i32(wl["token"], dev),
                        _dev.i32(wl["parent"], dev), _dev.i32(wl["node_off"], dev), full,
                        cap or full, ws)
        st = tg.last_device_status()
        assert not torch.any(ws != 0)
        if cap is None:
            assert st == 0
            ref = O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], full, bf16=bf)
            for g, r in zip(got, ref):
                np.testing.assert_array_equal(g.cpu().numpy(), r)
        else:
            ref = O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], full, bf16=bf)
            assert (st & 16) == (16 if ref[1].max() + 1 > cap else 0)


def test_accept_grafting_examples(dev):
    import json, os
    with open(os.path.join(os.path.dirname(__file__), "golden", "grafting_examples.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        parent = np.array(case["parent"], np.int32)
        n, V = len(parent), case["vocab"]
        x = np.zeros((n, V), np.float32)
        x[np.arange(n), case["target_argmax"]] = 3.0
        wl = dict(parent=parent, token=np.array(case["token"], np.int32),
                  node_off=np.array([0, n], np.int32), logits=x)
        path, A, bonus, _ = _run_accept(wl, dev, n)
        exp = case["accepted_path"]
        assert list(path[0, :len(exp)]) == exp and A[0] == len(exp) - 1
        assert bonus[0] == case["bonus"]


# ------------------------------------------------------------------ graft step pipeline

def test_graft_step_pipeline(dev):
    """Two-drafter grafting step: rescore all 64 weak-tree nodes, reselect 16
    grafting positions, expand each by top-8 from the stronger drafter's
    rows, graft the 128 children non-destructively (append), accept on the
    192-node tree.  Every stage gets identical inputs on both sides."""
    wl = synth.make_workload("graft-mha", seed=0, with_logits=False, with_strong=False)
    rng = synth.make_rng(123)
    n, V, N, k = 64, 32000, 16, 8
    weak_lp = synth.normal_f32(rng, (n, V), 3.0, -np.log(V) - 4.5)
    strong_lp = (weak_lp + synth.normal_f32(rng, (n, V), 0.5)).astype(np.float32)
    weak_edge = np.zeros(n, np.float32)
    for v in range(1, n):
        weak_edge[v] = weak_lp[wl["parent"][v], wl["token"][v]]
    visited = np.zeros(n, np.uint8)
    # stage 1: rescore + reselect
    e_g, s_g, sel_g, ns_g = tg.rescore_select(
        _dev.f32(weak_edge, dev), _dev.f32(strong_lp, dev), _dev.i32(wl["parent"], dev),
        _dev.i32(wl["token"], dev), _dev.u8(visited, dev), _dev.i32(wl["node_off"], dev), n, N)
    e_o, s_o, sel_o, ns_o = O.rescore_select(weak_edge, strong_lp, wl["parent"], wl["token"],
                                             visited, wl["node_off"], N)
    np.testing.assert_array_equal(sel_g.cpu().numpy(), sel_o)
    np.testing.assert_array_equal(s_g.cpu().numpy(), s_o)
    sel = sel_o[0]
    # stage 2: expand the selected nodes from the stronger drafter's rows
    tok_g, lp_g, sc_g, _ = tg.expand_topk(_dev.f32(strong_lp, dev), s_g[torch.from_numpy(sel).long().to(dev)].contiguous(), k,
                                          row_idx=_dev.i32(sel, dev))
    tok_o, lp_o, sc_o, _ = O.expand_topk(strong_lp, s_o[sel], k, row_idx=sel)
    np.testing.assert_array_equal(tok_g.cpu().numpy(), tok_o)
    np.testing.assert_allclose(sc_g.cpu().numpy(), sc_o, rtol=SCORE_RTOL, atol=1e-5)
    # stage 3: non-destructive graft (append children), then accept
    parent = np.concatenate([wl["parent"], np.repeat(sel, k)]).astype(np.int32)
    token = np.concatenate([wl["token"], tok_o.reshape(-1)]).astype(np.int32)
    n2 = len(parent)
    assert n2 == 192
    tl = synth.normal_f32(rng, (n2, V), 3.0)
    synth.plant_child_bump(rng, tl, parent, token, np.arange(n2), prob=0.9, bump=40.0)
    tl_bits = synth.f32_to_bf16_bits(tl)
    g = dict(parent=parent, token=token, node_off=np.array([0, n2], np.int32), logits=tl_bits)
    path, A, bonus, _ = _run_accept(g, dev, n2)
    rp, rA, rb = O.accept(tl_bits, token, parent, g["node_off"], n2, bf16=True)
    np.testing.assert_array_equal(path, rp)
    assert A[0] == rA[0] and bonus[0] == rb[0]


def test_graft_expand_on_device(dev):
    """The same two-drafter step with the graft on the device
    (treegraft_graft_expand, capacity layout): rescore + reselect, then the
    16 selected positions expanded by top-8 from the stronger drafter's rows
    and their children appended at rows 64.. of the 192-node tree.  Tokens
    and parents bit-exact, edge and path scores within 1e-4 relative of the
    oracle's expand_topk of the same rows; then accept on the grafted
    device arrays equals the oracle's accept."""
    wl = synth.make_workload("graft-mha", seed=4, with_logits=False, with_strong=False)
    rng = synth.make_rng(321)
    n, V, N, k, cap = 64, 32000, 16, 8, 192
    weak_lp = synth.normal_f32(rng, (n, V), 3.0, -np.log(V) - 4.5)
    strong_lp = (weak_lp + synth.normal_f32(rng, (n, V), 0.5)).astype(np.float32)
    weak_edge = np.zeros(n, np.float32)
    for v in range(1, n):
        weak_edge[v] = weak_lp[wl["parent"][v], wl["token"][v]]
    visited = (np.arange(n) < 5).astype(np.uint8)
    par = torch.full((cap,), -7, dtype=torch.int32, device=dev)
    tok = torch.full((cap,), -7, dtype=torch.int32, device=dev)
    edge = torch.zeros(cap, dtype=torch.float32, device=dev)
    score = torch.zeros(cap, dtype=torch.float32, device=dev)
    par[:n] = _dev.i32(wl["parent"], dev)
    tok[:n] = _dev.i32(wl["token"], dev)
    sel = torch.empty(1, N, dtype=torch.int32, device=dev)
    nsel = torch.empty(1, dtype=torch.int32, device=dev)
    strong = _dev.f32(strong_lp, dev)
    tg.rescore_select(_dev.f32(weak_edge, dev), strong, par[:n], tok[:n], _dev.u8(visited, dev),
                      _dev.i32(wl["node_off"], dev), n, N,
                      out=(edge[:n], score[:n], sel, nsel))
    tg.graft_expand(strong, sel, k, cap, n, par, tok, edge, score)
    _status_clean()
    e_o, s_o, sel_o, ns_o = O.rescore_select(weak_edge, strong_lp, wl["parent"], wl["token"],
                                             visited, wl["node_off"], N)
    assert int(nsel[0]) == N and int(ns_o[0]) == N
    np.testing.assert_array_equal(sel.cpu().numpy(), sel_o)
    tok_o, lp_o, sc_o, _ = O.expand_topk(strong_lp, s_o[sel_o[0]], k, row_idx=sel_o[0])
    np.testing.assert_array_equal(par.cpu().numpy()[n:], np.repeat(sel_o[0], k))
    np.testing.assert_array_equal(tok.cpu().numpy()[n:], tok_o.reshape(-1))
    np.testing.assert_allclose(edge.cpu().numpy()[n:], lp_o.reshape(-1), rtol=SCORE_RTOL, atol=1e-5)
    np.testing.assert_allclose(score.cpu().numpy()[n:], sc_o.reshape(-1), rtol=SCORE_RTOL, atol=1e-5)
    np.testing.assert_array_equal(score.cpu().numpy()[:n], s_o)
    # accept on the grafted device tree
    parent_h = np.concatenate([wl["parent"], np.repeat(sel_o[0], k)]).astype(np.int32)
    token_h = np.concatenate([wl["token"], tok_o.reshape(-1)]).astype(np.int32)
    tl = synth.normal_f32(rng, (cap, V), 3.0)
    synth.plant_child_bump(rng, tl, parent_h, token_h, np.arange(cap), prob=0.9, bump=40.0)
    tl_bits = synth.f32_to_bf16_bits(tl)
    ws = tg.accept_workspace(1, cap, dev)
    path, A, bonus = tg.accept(_dev.bf16(tl_bits, dev), tok, par,
                               torch.tensor([0, cap], dtype=torch.int32, device=dev), cap, cap, ws)
    _status_clean()
    rp, rA, rb = O.accept(tl_bits, token_h, parent_h, np.array([0, cap], np.int32), cap, bf16=True)
    np.testing.assert_array_equal(path.cpu().numpy(), rp)
    assert int(A[0]) == int(rA[0]) and int(bonus[0]) == int(rb[0])


def test_graft_expand_bad_selected_sets_status(dev):
    n, V, N, k, cap = 8, 64, 2, 2, 16
    lg = torch.zeros(n, V, device=dev)
    sel = torch.tensor([[3, 9]], dtype=torch.int32, device=dev)   # 9 is not a node
    par = torch.zeros(cap, dtype=torch.int32, device=dev)
    tok = torch.zeros(cap, dtype=torch.int32, device=dev)
    edge = torch.zeros(cap, device=dev)
    score = torch.zeros(cap, device=dev)
    tg.graft_expand(lg, sel, k, cap, n, par, tok, edge, score)
    assert tg.last_device_status() & 16
    assert par.cpu().numpy()[n:n + k].tolist() == [3, 3]            # the valid slot is grafted


# ------------------------------------------------------------------ serving sweep

def _serving_kv(wl, dev):
    """Device K/V caches of a serving workload built with kv_trees: the
    drawn trees' rows scattered into zero caches."""
    sh = wl["shape"]
    B, Hkv, D = sh["B"], sh["Hkv"], sh["D"]
    k = torch.zeros((B, Hkv, wl["S_max"], D), dtype=torch.bfloat16, device=dev)
    v = torch.zeros_like(k)
    for i, b in enumerate(wl["kv_trees"]):
        k[b] = _dev.bf16(wl["k_cache"][i], dev)
        v[b] = _dev.bf16(wl["v_cache"][i], dev)
    return k, v


@pytest.mark.parametrize("B", [4, 16, 64])
def test_tree_attn_serving_sweep(dev, B):
    """Ragged serving batch: prefixes log-uniform in 512-32768, trees of
    32-256 nodes, depth 4-10, GQA 32/8.  Three trees carry random K/V and
    are checked against the oracle; every other tree has all-zero K/V, so
    its outputs are exactly 0 and its lse is ln(P + depth(u) + 1) - the
    number of keys the Algorithm 3 mask lets node u see."""
    sh = synth.serving_shape(B, seed=0)
    drawn = sorted({0, B // 2, B - 1})
    wl = synth.make_workload(sh, seed=B, with_logits=False, with_strong=False, kv_trees=drawn)
    k, v = _serving_kv(wl, dev)
    q = _dev.bf16(wl["q"], dev)
    lse = torch.full((q.shape[0], q.shape[1]), float("nan"), device=dev)
    out, _ = tg.tree_attn(q, k, v, _dev.i32(wl["prefix_len"], dev), _dev.i32(wl["parent"], dev),
                          _dev.i32(wl["node_off"], dev), _dev.max_nodes(wl), lse_out=lse)
    _status_clean()
    o = _dev.bf16_to_np(out)
    lse = lse.cpu().numpy().astype(np.float64)
    off = wl["node_off"]
    for i, b in enumerate(drawn):
        a, e = int(off[b]), int(off[b + 1])
        ref_o, ref_lse = O.tree_attention(wl["q"][a:e], wl["k_cache"][i:i + 1],
                                          wl["v_cache"][i:i + 1], wl["prefix_len"][b:b + 1],
                                          wl["parent"][a:e], [0, e - a], Hkv=sh["Hkv"])
        _check_attn(wl, o[a:e], lse[a:e], ref_o, ref_lse)
    for b in range(B):
        if b in drawn:
            continue
        a, e = int(off[b]), int(off[b + 1])
        assert np.all(o[a:e] == 0.0)
        count = int(wl["prefix_len"][b]) + O.node_depth(wl["parent"][a:e]) + 1
        np.testing.assert_allclose(lse[a:e], np.log(count)[:, None] * np.ones((1, sh["Hq"])),
                                   atol=LSE_ABS, rtol=0)


@pytest.mark.parametrize("p_long", [8000, 20000])
def test_tree_attn_long_tree_cut_into_key_chunks(dev, p_long):
    """One long tree among short ones: the batch runs as whole units dealt
    longest first, and the long tree's units are cut into key chunks (about
    one resident CTA's share of the batch each) whose last one to finish
    merges them (about 7 chunks for the 8000-token prefix, 11 for 20000: the
    merge then takes its chunks' statistics in two batches).  The long tree
    and a short one carry random K/V and are checked against the oracle; the
    others have all-zero K/V (outputs exactly 0, lse = ln of the number of
    keys each node sees).  Two calls in a row on the same workspace: the
    chunk tickets are back at zero after each."""
    P = [p_long, 300, 500, 700, 900, 1100, 1300, 1500, 1700]
    n = [64, 40, 48, 56, 64, 72, 80, 88, 96]
    shape = _attn_shape(len(P), P, n, [6] * len(P), 32, 8, 128, cap=10)
    drawn = [0, 4]
    wl = synth.make_workload(shape, seed=31, with_logits=False, with_strong=False, kv_trees=drawn)
    k, v = _serving_kv(wl, dev)
    q = _dev.bf16(wl["q"], dev)
    sh = wl["shape"]
    B = len(P)
    ws = torch.zeros(tg.tree_attn_workspace_size(B, _dev.max_nodes(wl), 32, 8, 128),
                     dtype=torch.uint8, device=dev)
    off = wl["node_off"]
    refs = {}
    for i, b in enumerate(drawn):
        a, e = int(off[b]), int(off[b + 1])
        refs[b] = O.tree_attention(wl["q"][a:e], wl["k_cache"][i:i + 1], wl["v_cache"][i:i + 1],
                                   wl["prefix_len"][b:b + 1], wl["parent"][a:e], [0, e - a], Hkv=8)
    for _ in range(2):
        lse = torch.full((q.shape[0], q.shape[1]), float("nan"), device=dev)
        out, _ = tg.tree_attn(q, k, v, _dev.i32(wl["prefix_len"], dev), _dev.i32(wl["parent"], dev),
                              _dev.i32(wl["node_off"], dev), _dev.max_nodes(wl), lse_out=lse, ws=ws)
        _status_clean()
        o = _dev.bf16_to_np(out)
        lse = lse.cpu().numpy().astype(np.float64)
        for b in drawn:
            a, e = int(off[b]), int(off[b + 1])
            _check_attn(wl, o[a:e], lse[a:e], *refs[b])
        for b in range(B):
            if b in drawn:
                continue
            a, e = int(off[b]), int(off[b + 1])
            assert np.all(o[a:e] == 0.0)
            count = int(wl["prefix_len"][b]) + O.node_depth(wl["parent"][a:e]) + 1
            np.testing.assert_allclose(lse[a:e], np.log(count)[:, None] * np.ones((1, 32)),
                                       atol=LSE_ABS, rtol=0)


@pytest.mark.parametrize("D,Hq,Hkv", [(64, 32, 8), (128, 8, 8), (128, 64, 8)])
def test_tree_attn_whole_units_head_dims_and_groups(dev, D, Hq, Hkv):
    """Batches that fill the GPU with whole units, at head size 64 and at
    GQA groups of 1 and 8 (the serving tests use 128 and 4): units of one and
    of two query tiles, and one long tree whose units are cut into key chunks.
    Two trees carry random K/V and are checked against the oracle; the others
    have all-zero K/V (outputs exactly 0, lse = ln of the keys each node
    sees)."""
    P = [12000, 700, 1500, 300, 900, 2100, 60, 1200, 500, 1800, 1000, 400]
    n = [90, 120, 64, 200, 33, 150, 100, 128, 17, 180, 75, 140]
    shape = _attn_shape(len(P), P, n, [6] * len(P), Hq, Hkv, D, cap=10)
    drawn = [1, 2]
    wl = synth.make_workload(shape, seed=41, with_logits=False, with_strong=False, kv_trees=drawn)
    k, v = _serving_kv(wl, dev)
    q = _dev.bf16(wl["q"], dev)
    B = len(P)
    ws = torch.zeros(tg.tree_attn_workspace_size(B, _dev.max_nodes(wl), Hq, Hkv, D),
                     dtype=torch.uint8, device=dev)
    lse = torch.full((q.shape[0], q.shape[1]), float("nan"), device=dev)
    out, _ = tg.tree_attn(q, k, v, _dev.i32(wl["prefix_len"], dev), _dev.i32(wl["parent"], dev),
                          _dev.i32(wl["node_off"], dev), _dev.max_nodes(wl), lse_out=lse, ws=ws)
    _status_clean()
    o = _dev.bf16_to_np(out)
    lse = lse.cpu().numpy().astype(np.float64)
    off = wl["node_off"]
    for i, b in enumerate(drawn):
        a, e = int(off[b]), int(off[b + 1])
        ref_o, ref_lse = O.tree_attention(wl["q"][a:e], wl["k_cache"][i:i + 1], wl["v_cache"][i:i + 1],
                                          wl["prefix_len"][b:b + 1], wl["parent"][a:e], [0, e - a],
                                          Hkv=Hkv)
        _check_attn(wl, o[a:e], lse[a:e], ref_o, ref_lse)
    for b in range(B):
        if b in drawn:
            continue
        a, e = int(off[b]), int(off[b + 1])
        assert np.all(o[a:e] == 0.0)
        count = int(wl["prefix_len"][b]) + O.node_depth(wl["parent"][a:e]) + 1
        np.testing.assert_allclose(lse[a:e], np.log(count)[:, None] * np.ones((1, Hq)),
                                   atol=LSE_ABS, rtol=0)


def test_accept_serving_sweep(dev):
    """accept on an 8-tree ragged serving batch (n 32-256, depth 4-10) with
    bf16 target logits over 128256 tokens, bumps planted at +40 so that long
    paths occur; bit-exact against the oracle."""
    sh = synth.serving_shape(8, seed=1)
    wl = synth.make_workload(sh, seed=8, with_strong=False, with_logits=False, kv_trees=[])
    rng = synth.make_rng(88)
    lg = synth.normal_f32(rng, (len(wl["parent"]), sh["V"]), 3.0)
    off = wl["node_off"]
    for b in range(sh["B"]):
        a, e = int(off[b]), int(off[b + 1])
        synth.plant_child_bump(rng, lg, wl["parent"][a:e], wl["token"][a:e], np.arange(a, e),
                               prob=0.9, bump=40.0)
    wl["logits"] = synth.f32_to_bf16_bits(lg)
    cap = 16
    got = _run_accept(wl, dev, cap)
    ref = O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], cap, bf16=True)
    for g, r in zip(got[:3], ref):
        np.testing.assert_array_equal(g, r)
    assert ref[1].max() >= 2


def test_expand_topk_many_rows_llama_vocab(dev):
    """336 bf16 rows over 128256 tokens picked by row_idx from 400 (k = 10):
    two rows or more per SM, so whole rows are streamed by one CTA each (8
    batches per row)."""
    rng = synth.make_rng(21)
    lg = synth.f32_to_bf16_bits(synth.normal_f32(rng, (400, 128256), 3.0))
    rows = synth.make_rng(22).permutation(400)[:336].astype(np.int32)
    ps = -np.abs(synth.normal_f32(rng, (336,), 4.0))
    got = _run_expand(_dev.bf16(lg, dev), ps, 10, dev, row_idx=rows)
    ref = O.expand_topk(lg, ps, 10, row_idx=rows, bf16=True)
    _check_expand(got, ref)


@pytest.mark.parametrize("V,ld,dtype,k", [(32001, 32008, "bf16", 32), (1023, 1024, "f32", 5),
                                          (40000, 40000, "f32", 16)])
def test_expand_topk_many_rows_ragged_vocab(dev, V, ld, dtype, k):
    """320 rows, ragged vocabularies and row strides, both dtypes: the
    streamed rows end inside a batch (or are shorter than one)."""
    rng = synth.make_rng(V + 3 * k)
    rows = 320
    x = synth.normal_f32(rng, (rows, ld), 3.0)
    ps = synth.normal_f32(rng, (rows,), 2.0)
    if dtype == "bf16":
        bits = synth.f32_to_bf16_bits(x)
        got = _run_expand(_dev.bf16(bits, dev), ps, k, dev, V=V)
        ref = O.expand_topk(bits[:, :V], ps, k, bf16=True)
    else:
        got = _run_expand(_dev.f32(x, dev), ps, k, dev, V=V)
        ref = O.expand_topk(x[:, :V], ps, k)
    _check_expand(got, ref)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_expand_topk_many_rows_ties_and_inf(dev, dtype):
    """320 streamed rows of heavy ties (the candidate buffer overflows and the
    exact-key fallback ranks the row), all -inf and signed-zero rows."""
    rng = synth.make_rng(31)
    rows, V = 320, 9000
    x = rng.integers(-1, 2, size=(rows, V)).astype(np.float32)
    x[7] = -np.inf
    x[8, ::3] = -np.inf
    x[9] = 0.0
    x[10, :] = -0.0
    x[10, 17] = 0.0
    x[11, V - 1] = 0.5
    x[100:200] = synth.normal_f32(rng, (100, V), 3.0)    # ordinary rows between
    ps = synth.normal_f32(rng, (rows,), 1.0)
    if dtype == "f32":
        got = _run_expand(_dev.f32(x, dev), ps, 12, dev)
        ref = O.expand_topk(x, ps, 12)
    else:
        bits = synth.f32_to_bf16_bits(x)
        got = _run_expand(_dev.bf16(bits, dev), ps, 12, dev)
        ref = O.expand_topk(bits, ps, 12, bf16=True)
    np.testing.assert_array_equal(got[0], ref[0])
    for g, r in zip(got[1:], ref[1:]):
        np.testing.assert_array_equal(np.isneginf(g), np.isneginf(r))
        fin = np.isfinite(r)
        np.testing.assert_allclose(g[fin], r[fin], rtol=1e-5, atol=1e-5)


def test_expand_topk_serving_rows(dev):
    """expand_topk over 128 frontier rows picked by row_idx from 512 bf16
    logit rows over 128256 tokens (k = 10), as a serving step expands the
    frontier of every tree in the batch."""
    sh = synth.serving_shape(8, seed=2)
    rng = synth.make_rng(9)
    lg = synth.f32_to_bf16_bits(synth.normal_f32(rng, (512, sh["V"]), 3.0))
    rows = np.sort(synth.make_rng(77).choice(512, size=128, replace=False)).astype(np.int32)
    ps = -np.abs(synth.normal_f32(rng, (128,), 4.0))
    got = _run_expand(_dev.bf16(lg, dev), ps, sh["k"], dev, row_idx=rows)
    ref = O.expand_topk(lg, ps, sh["k"], row_idx=rows, bf16=True)
    _check_expand(got, ref)



# ------------------------------------------------------------------ GlobalPrune (Algorithm 3)

def _mask_words(mask_bool):
    """bool [B, Mo, Mo] -> uint32 words [B, Mo, ceil(Mo / 32)], bit j of word j // 32."""
    B, Mo, _ = mask_bool.shape
    W = (Mo + 31) // 32
    out = np.zeros((B, Mo, W), dtype=np.uint32)
    for j in range(Mo):
        out[:, :, j // 32] |= mask_bool[:, :, j].astype(np.uint32) << np.uint32(j % 32)
    return out


def _run_prune(parents, scores, budget, path_cap, dev):
    off = np.concatenate([[0], np.cumsum([len(p) for p in parents])]).astype(np.int32)
    par, sc = np.concatenate(parents).astype(np.int32), np.concatenate(scores).astype(np.float32)
    maxn = max(len(p) for p in parents)
    got = tg.global_prune(_dev.f32(sc, dev), _dev.i32(par, dev), _dev.i32(off, dev), maxn, budget,
                          path_cap)
    _status_clean()
    got = [t.cpu().numpy() for t in got]
    got[4] = got[4].view(np.uint32)
    ref = O.global_prune(par, sc, off, budget, path_cap)
    return got, ref


def _check_prune(got, ref):
    kept, n_kept, new_par, pos, mask, paths, n_paths = got
    rk, rn, rp, rpos, rmask, rpaths, rnp = ref
    np.testing.assert_array_equal(n_kept, rn)
    np.testing.assert_array_equal(kept, rk)
    np.testing.assert_array_equal(new_par, rp)
    np.testing.assert_array_equal(pos, rpos)
    np.testing.assert_array_equal(mask, _mask_words(rmask))
    np.testing.assert_array_equal(n_paths, rnp)
    np.testing.assert_array_equal(paths, rpaths)


@pytest.mark.parametrize("monotone", [True, False])
def test_global_prune_expansion_trees(dev, monotone):
    """Trees with the shape of 6 expansion steps of frontier 10 and branching
    10 (511 nodes) and of smaller growths, pruned to a 59-node budget:
    path-sum scores (the realistic case) and random scores (long chains)."""
    rng = synth.make_rng(300 + monotone)
    parents = [synth.expansion_tree(rng, 6, 10, 10), synth.expansion_tree(rng, 4, 3, 4),
               synth.expansion_tree(rng, 3, 5, 8), synth.sample_tree(rng, 40, 5)]
    scores = [synth.path_scores(rng, p) if monotone else synth.normal_f32(rng, (len(p),), 3.0)
              for p in parents]
    got, ref = _run_prune(parents, scores, 59, 12, dev)
    _check_prune(got, ref)


def test_global_prune_largest_trees_and_budgets(dev):
    rng = synth.make_rng(310)
    parents = [synth.sample_tree(rng, 1024, 9, 16), synth.sample_tree(rng, 700, 12),
               np.array([-1], np.int32), synth.expansion_tree(rng, 5, 8, 8)]
    scores = [synth.path_scores(rng, parents[0]), synth.normal_f32(rng, (700,), 2.0),
              np.zeros(1, np.float32), np.round(synth.normal_f32(rng, (len(parents[3]),), 1.0))]
    for budget in (1, 63, 255):
        got, ref = _run_prune(parents, scores, budget, 16, dev)
        _check_prune(got, ref)


def test_global_prune_rows_outside_every_tree_set_status(dev):
    """node_off[B] < n_total leaves rows in no tree: TG_ERR_DEVICE_TREE, and
    the trees within their extents are still pruned exactly."""
    rng = synth.make_rng(77)
    pars = [synth.expansion_tree(rng, 4, 5, 5) for _ in range(2)]
    parent = np.concatenate(pars).astype(np.int32)
    score = np.concatenate([synth.path_scores(rng, p) for p in pars]).astype(np.float32)
    off = np.array([0, len(pars[0]), len(parent)], np.int32)
    short = off.copy()
    short[-1] -= 2                      # tree 1 loses its last two nodes (still a valid tree)
    got = tg.global_prune(_dev.f32(score, dev), _dev.i32(parent, dev), _dev.i32(short, dev),
                          int(np.max(np.diff(off))), 12, 8)
    assert tg.last_device_status() & 4
    ref = O.global_prune(parent, score, short, 12, 8)
    for g, r in zip(got[:2], ref[:2]):  # kept nodes and their counts, both trees
        np.testing.assert_array_equal(g.cpu().numpy(), r)


def test_global_prune_malformed_tree_sets_status(dev):
    par = np.array([-1, 0, 3, 1], np.int32)            # parent after child
    tg.global_prune(_dev.f32(np.zeros(4), dev), _dev.i32(par, dev), _dev.i32([0, 4], dev), 4, 2,
                    4)
    assert tg.last_device_status() & 4
