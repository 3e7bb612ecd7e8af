"""Seeded synthetic inputs for the fingerprint forward pass.

This module serves the tests, ``bench.py`` and the oracle alike.  It holds
none of the method's arithmetic: only counter-based random draws and their
mapping to bf16 weight values and prompt token ids.

Generator (the same definition is implemented independently on the device
in ``paper_2501_13111_gb300/csrc/fp_quant.cu`` and ``common.cuh``):

* SplitMix64 (Steele, Lea and Flood, OOPSLA 2014): the state advances by the
  golden-ratio increment ``GAMMA`` and each output is the state passed
  through the ``mix64`` finaliser.  It is counter-based: output ``i`` of a
  stream is ``mix64(key + (i + 1) * GAMMA)``, so any element can be drawn
  without drawing the ones before it.
* A stream's ``key`` is ``mix64(seed + (stream + 1) * GAMMA)``.
* Weights: the four 16-bit lanes of one 64-bit draw are summed (Irwin-Hall
  with n = 4, an approximate normal), centred, scaled to standard deviation
  ``sigma`` by one fp64 multiplication, rounded to fp32 and then to bf16
  (both round-to-nearest-even).  Every step is exact or correctly rounded,
  so host and device produce bit-identical weights.
* Token ids: Lemire's multiply-shift maps the high 32 bits of a draw onto
  ``[0, vocab)``.
* Act orders (the input-channel permutation of a GPTQ-format matrix): the
  Fisher-Yates shuffle in Durstenfeld's form over the identity, for
  ``i = K-1 .. 1`` swapping entry ``i`` with entry ``j``, ``j`` the
  multiply-shift of draw ``K-1-i`` onto ``[0, i]``.  The runtime draws the
  same permutation on the host (``csrc/fp_runtime.cu``).
"""
from __future__ import annotations

import os

import numpy as np

GAMMA = 0x9E3779B97F4A7C15
_M1 = 0xBF58476D1CE4E5B9
_M2 = 0x94D049BB133111EB
_MASK = (1 << 64) - 1

# sigma / std(sum of four uniform 16-bit integers) for sigma = 0.02:
# 0.02 / sqrt(4 * (65536**2 - 1) / 12), written as an exact fp64 literal.
WEIGHT_SCALE_002 = float.fromhex("0x1.1bc779ef9b324p-21")
IRWIN_HALL_MEAN = 2 * 65535  # mean of the sum of four lanes, times 2 / 2

# Stream numbering: one stream per weight tensor, (layer + 1) * 16 + tensor.
# layer = -1 holds the embedding (0), the final norm gain (1) and the LM head (2).
TOKEN_STREAM = 1 << 20


def weight_stream(layer: int, tensor: int) -> int:
    return (layer + 1) * 16 + tensor


def perm_stream(layer: int, mat: int) -> int:
    """Stream of the act order of fused matrix ``mat`` (0 QKV, 1 O, 2 gate+up,
    3 down) of block ``layer``: slots 9..12 of the layer's 16 streams."""
    return (layer + 1) * 16 + 9 + mat


def _mix64_int(z: int) -> int:
    z &= _MASK
    z = ((z ^ (z >> 30)) * _M1) & _MASK
    z = ((z ^ (z >> 27)) * _M2) & _MASK
    return z ^ (z >> 31)


def mix64(z: np.ndarray) -> np.ndarray:
    z = z.astype(np.uint64, copy=True)
    z ^= z >> np.uint64(30)
    z *= np.uint64(_M1)
    z ^= z >> np.uint64(27)
    z *= np.uint64(_M2)
    z ^= z >> np.uint64(31)
    return z


def stream_key(seed: int, stream: int) -> int:
    return _mix64_int((seed + (stream + 1) * GAMMA) & _MASK)


def draws(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """Outputs ``start .. start+count-1`` of the SplitMix64 stream (uint64)."""
    key = np.uint64(stream_key(seed, stream))
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        state = key + idx * np.uint64(GAMMA)
    return mix64(state)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest, ties to even); returns the uint16 bit pattern."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _irwin_hall_sum(u: np.ndarray) -> np.ndarray:
    m = np.uint64(0xFFFF)
    s = (u & m) + ((u >> np.uint64(16)) & m) + ((u >> np.uint64(32)) & m) + (u >> np.uint64(48))
    return s.astype(np.int64)


def normal_bf16(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """bf16 bit patterns of approximately N(0, 0.02) weights (see module doc)."""
    out = np.empty(count, dtype=np.uint16)
    step = 1 << 20  # chunks that stay in cache

    def chunk(lo):
        n = min(step, count - lo)
        s = _irwin_hall_sum(draws(seed, stream, start + lo, n))
        v = (s - IRWIN_HALL_MEAN).astype(np.float64) * WEIGHT_SCALE_002
        out[lo:lo + n] = f32_to_bf16_bits(v.astype(np.float32))

    starts = range(0, count, step)
    if count >= 8 * step:  # counter-based draws: chunks are independent, numpy releases the GIL
        from concurrent.futures import ThreadPoolExecutor

        with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
            list(ex.map(chunk, starts))
    else:
        for lo in starts:
            chunk(lo)
    return out


def weight_bf16(seed: int, layer: int, tensor: int, shape) -> np.ndarray:
    """A whole weight tensor, row-major, as bf16 bit patterns."""
    n = int(np.prod(shape))
    return normal_bf16(seed, weight_stream(layer, tensor), 0, n).reshape(shape)


def weight_rows_bf16(seed: int, layer: int, tensor: int, rows, ncols: int) -> np.ndarray:
    """Selected rows of a row-major weight tensor (random access by counter)."""
    out = [normal_bf16(seed, weight_stream(layer, tensor), int(r) * ncols, ncols) for r in rows]
    return np.stack(out) if out else np.zeros((0, ncols), np.uint16)


def tokens(seed: int, count: int, vocab: int, stream: int = TOKEN_STREAM) -> np.ndarray:
    """Uniform token ids in [0, vocab) by multiply-shift of the high 32 bits."""
    hi = draws(seed, stream, 0, count) >> np.uint64(32)
    return ((hi * np.uint64(vocab)) >> np.uint64(32)).astype(np.int32)


def uniform_bf16(seed: int, stream: int, shape, lo: float, hi: float) -> np.ndarray:
    """bf16 bit patterns uniform in [lo, hi) (test inputs: gains, activations)."""
    n = int(np.prod(shape))
    u = (draws(seed, stream, 0, n) >> np.uint64(11)).astype(np.float64) * (1.0 / (1 << 53))
    return f32_to_bf16_bits((lo + (hi - lo) * u).astype(np.float32)).reshape(shape)


def uniform_f32(seed: int, stream: int, shape, lo: float, hi: float) -> np.ndarray:
    n = int(np.prod(shape))
    u = (draws(seed, stream, 0, n) >> np.uint64(11)).astype(np.float64) * (1.0 / (1 << 53))
    return (lo + (hi - lo) * u).astype(np.float32).reshape(shape)


def act_order(seed: int, layer: int, mat: int, k: int) -> np.ndarray:
    """The seeded act order of one matrix: a permutation of 0 .. k-1 (int32)."""
    p = np.arange(k, dtype=np.int64)
    if k < 2:
        return p.astype(np.int32)
    hi = draws(seed, perm_stream(layer, mat), 0, k - 1) >> np.uint64(32)
    for t in range(k - 1):
        i = k - 1 - t
        j = int((int(hi[t]) * (i + 1)) >> 32)
        p[i], p[j] = p[j], p[i]
    return p.astype(np.int32)
