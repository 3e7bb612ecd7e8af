"""Shared helpers of the GPU parity tests: device buffers through torch (memory
plumbing only), oracle set-up from the seeded generators, tolerances."""
from __future__ import annotations

import numpy as np

import synth
from oracle import model as M
from oracle import quant

# Tolerances of the parity bar: max |gpu - ref| <= tau * max |ref| per tensor,
# 2e-2 on bf16 / int8 weight paths, 5e-2 on int4 weight paths (GPTQ4 is int4).
TAU = {0: 2e-2, 1: 2e-2, 2: 5e-2, 3: 5e-2}


def torch_mod():
    import torch

    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch


# Every device buffer a test makes stays referenced until the test ends, so a
# pointer taken from a temporary (ptr(dev(x))) cannot be recycled by torch's
# caching allocator before the kernel reading it has run.
KEEP = []


def dev(a: np.ndarray):
    """Host numpy array -> device tensor with the same bytes."""
    torch = torch_mod()
    a = np.ascontiguousarray(a)
    view = {np.dtype(np.uint16): np.int16, np.dtype(np.uint32): np.int32}.get(a.dtype)
    t = torch.from_numpy(a.view(view) if view else a).to("cuda")
    KEEP.append(t)
    return t


def host(t, dtype):
    torch = torch_mod()
    torch.cuda.synchronize()
    a = t.detach().cpu().numpy()
    return a.view(dtype)


def empty(n_bytes_or_shape, dtype=np.uint8):
    torch = torch_mod()
    tmap = {np.dtype(np.uint8): torch.uint8, np.dtype(np.int8): torch.int8, np.dtype(np.uint16): torch.int16,
            np.dtype(np.int16): torch.int16, np.dtype(np.int32): torch.int32, np.dtype(np.float32): torch.float32}
    shape = n_bytes_or_shape if isinstance(n_bytes_or_shape, tuple) else (n_bytes_or_shape,)
    t = torch.zeros(shape, dtype=tmap[np.dtype(dtype)], device="cuda")
    KEEP.append(t)
    return t


def ptr(t):
    return t.data_ptr() if t is not None else None


def rel_err(gpu, ref):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.max(np.abs(gpu - ref)) / max(np.max(np.abs(ref)), 1e-30))


# ---------------------------------------------------------------- weights
def arch_dict(a: M.Arch):
    return dict(n_layers=a.n_layers, hidden=a.hidden, n_heads=a.n_heads, n_kv_heads=a.n_kv_heads,
                head_dim=a.head_dim, ffn=a.ffn, vocab=a.vocab, rms_eps=a.rms_eps, rope_base=a.rope_base)


def weight_getter(seed, gains="random", scale=1.0):
    """bf16 tensors for both sides: seeded N(0, 0.02)-like matrices (times
    ``scale``) and random gains in [0.5, 1.5) so a dropped gain shows."""

    def get(layer, t, shape):
        if len(shape) == 1:
            if gains == "ones":
                return synth.f32_to_bf16_bits(np.ones(shape, np.float32))
            return synth.uniform_bf16(seed, 900 + 16 * (layer + 1) + t, shape, 0.5, 1.5)
        w = synth.weight_bf16(seed, layer, t, shape)
        if scale != 1.0:
            w = synth.f32_to_bf16_bits(quant.bf16_to_f32(w) * np.float32(scale))
        return w

    return get


def upload_weights(fp, h, arch: M.Arch, get):
    for t in range(3):
        fp.fp_set_weight(h, -1, t, get(-1, t, M.tensor_shape(arch, -1, t)).reshape(-1))
    for l in range(arch.n_layers):
        for t in range(9):
            fp.fp_set_weight(h, l, t, get(l, t, M.tensor_shape(arch, l, t)).reshape(-1))
