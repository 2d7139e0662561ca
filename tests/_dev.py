"""Helpers for GPU tests: move the generator's numpy arrays onto the device
in the layouts the C ABI expects (no arithmetic)."""
import numpy as np
import torch


def bf16(bits, dev):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)


def f32(a, dev):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)


def i32(a, dev):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)


def u8(a, dev):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint8)).to(dev)


def logits(wl, dev):
    lg = wl["logits"]
    return bf16(lg, dev) if lg.dtype == np.uint16 else f32(lg, dev)


def bf16_to_np(t):
    """bf16 device tensor -> float64 numpy (exact)."""
    bits = t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def max_nodes(wl):
    off = wl["node_off"]
    return int(np.max(np.diff(off)))
