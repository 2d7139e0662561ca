"""treegraft_accept_noalloc, the accept entry point for callers that cannot
allocate device memory (for example a plugin that an inference engine hands
only its inputs and outputs): it must give exactly what treegraft_accept
gives with a caller-provided workspace, on two calls in a row (the second
call starts from whatever the first left in the library's fixed scratch
array).  Called through the C ABI with raw device pointers.

This file is collected last on purpose, and it passes both on its own in a
fresh process and after the rest of the suite."""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _inputs(name, seed, dev):
    from paper_2608_26112_gb300 import synth
    wl = synth.make_workload(name, seed=seed, with_strong=False)
    lg = wl["logits"]
    if lg.dtype == np.uint16:
        logits = torch.from_numpy(lg.view(np.int16)).to(dev).view(torch.bfloat16)
    else:
        logits = torch.from_numpy(lg).to(dev)
    as_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)
    n_total = len(wl["parent"])
    B = len(wl["node_off"]) - 1
    max_nodes = int(np.max(np.diff(wl["node_off"])))
    return (logits, as_dev(wl["token"]), as_dev(wl["parent"]), as_dev(wl["node_off"]), B,
            max_nodes, n_total)


def _noalloc_call(lib, logits, token, parent, node_off, B, max_nodes, n_total, path_cap):
    dev = logits.device
    path = torch.full((B, path_cap), -7, dtype=torch.int32, device=dev)
    alen = torch.full((B,), -7, dtype=torch.int32, device=dev)
    bonus = torch.full((B,), -7, dtype=torch.int32, device=dev)
    dtype = 0 if logits.dtype == torch.bfloat16 else 1
    st = lib.treegraft_accept_noalloc(
        ctypes.c_void_p(logits.data_ptr()), dtype, logits.shape[1], logits.stride(0),
        ctypes.c_void_p(token.data_ptr()), ctypes.c_void_p(parent.data_ptr()),
        ctypes.c_void_p(node_off.data_ptr()), B, max_nodes, n_total, path_cap,
        ctypes.c_void_p(path.data_ptr()), ctypes.c_void_p(alen.data_ptr()),
        ctypes.c_void_p(bonus.data_ptr()), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0
    return path, alen, bonus


def test_accept_noalloc_matches_accept_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26112_gb300 import build
    build.build()
    import paper_2608_26112_gb300 as tg
    lib = tg.lib()
    dev = torch.device("cuda:0")
    # two calls in a row, different shapes: a 4-tree bf16 batch, then a 1-tree fp32 one
    for name, seed in (("llama3-70b-verify", 3), ("tiny", 5)):
        logits, token, parent, node_off, B, max_nodes, n_total = _inputs(name, seed, dev)
        cap = max_nodes
        got = _noalloc_call(lib, logits, token, parent, node_off, B, max_nodes, n_total, cap)
        ws = tg.accept_workspace(B, n_total, dev)
        ref = tg.accept(logits, token, parent, node_off, max_nodes, cap, ws)
        assert tg.last_device_status() == 0
        for g, r in zip(got, ref):
            assert torch.equal(g, r)        # integer outputs: exact
        # and directly against the CPU oracle
        from oracle import treegraft_oracle as O
        from paper_2608_26112_gb300 import synth
        wl = synth.make_workload(name, seed=seed, with_strong=False)
        want = O.accept(wl["logits"], wl["token"], wl["parent"], wl["node_off"], cap,
                        bf16=wl["logits"].dtype == np.uint16)
        for g, r in zip(got, want):
            np.testing.assert_array_equal(g.cpu().numpy(), r)


def test_accept_noalloc_rows_outside_every_tree():
    """A node_off whose last entry falls short of n_total leaves rows in no
    tree: they raise TG_ERR_DEVICE_TREE instead of drawing a ticket of the
    last tree, and the next call is exact again."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_26112_gb300 import build
    build.build()
    import paper_2608_26112_gb300 as tg
    lib = tg.lib()
    dev = torch.device("cuda:0")
    logits, token, parent, node_off, B, max_nodes, n_total = _inputs("llama3-70b-verify", 9, dev)
    short = node_off.clone()
    short[-1] -= 3
    _noalloc_call(lib, logits, token, parent, short, B, max_nodes, n_total, max_nodes)
    assert tg.last_device_status() & 4
    got = _noalloc_call(lib, logits, token, parent, node_off, B, max_nodes, n_total, max_nodes)
    ws = tg.accept_workspace(B, n_total, dev)
    ref = tg.accept(logits, token, parent, node_off, max_nodes, max_nodes, ws)
    assert tg.last_device_status() == 0
    for g, r in zip(got, ref):
        assert torch.equal(g, r)


def test_accept_noalloc_rejects_sizes_beyond_its_array():
    from paper_2608_26112_gb300 import build
    build.build()
    import paper_2608_26112_gb300 as tg
    fake = ctypes.c_void_p(0x1000)
    # more nodes than the fixed scratch holds: refused on the host, nothing launched
    st = tg.lib().treegraft_accept_noalloc(fake, 0, 100, 100, fake, fake, fake, 300, 256,
                                           70000, 8, fake, fake, fake, None)
    assert st == 2
