"""Weight-only and KV-cache quantisers of the oracle (test infrastructure only).

The paper lists INT8 and INT4 weight-only quantisation and an INT8 KV cache
among its deployment configurations (Sec. 2 "LLM deployment configuration
parameters"; Sec. 3.2; Table "Models and configurations") and states their
memory effect (-50 % / -75 %, Sec. 3.2), but not their arithmetic.  The
readings implemented here:

int8 weights, per output channel (row n of W[N, K]):
    a   = max_k |W[n, k]|                      (exact: bf16 inputs)
    s_n = bf16 round-toward-+inf of fp32(a / 127)
    q   = clamp(rint(fp32(W / s_n)), -127, 127)   rint = ties to even
    dequantised weight = q * s_n;  a zero row gives s = 0, q = 0.

int4 weights, asymmetric, groups of 128 along K (row n, group g):
    mn = min(0, min w), mx = max(0, max w)
    s  = bf16 round-toward-+inf of fp32(fp32(mx - mn) / 15)
    z  = clamp(rint(fp32(-mn / s)), 0, 15)     (stored as bf16, exact)
    q  = clamp(rint(fp32(w / s)) + z, 0, 15)
    dequantised weight = (q - z) * s;  a zero range gives s = z = q = 0.
    Packing: bytes [N][K/2].  Each little-endian 32-bit word holds 8
    consecutive elements e0..e7 of a row; nibble i (bits 4i .. 4i+3) holds
    element NIBBLE_ORDER[i] = (0, 2, 4, 6, 1, 3, 5, 7).  So the nibble pair
    (i, i + 4) -- the pair a mask of 0x000F000F selects -- is (e_2i, e_2i+1).

GPTQ-format int4 with act order (GPTQ4 in the table "Models and
configurations"; Sec. 3.2), read as int4 group-128 over groups formed in an
act order: a permutation perm of the K input channels; group g holds the
channels perm[128 g .. 128 g + 127], i.e. channel k is in group
g_idx[k] = (position of k in perm) // 128.  No calibration data exists here,
so the codes are rounded to nearest with the int4 rule above applied to each
group's values (GPTQ's error feedback needs calibration activations).
    dequantised weight W[n, k] = (q[n, k] - z[n, g_idx[k]]) * s[n, g_idx[k]]
    Storage: codes in act order (column j of the packed matrix is channel
    perm[j]), packed as int4 above; scales and zeros [N, K/128] per group.

int8 KV cache, per token and per KV head, separately for K (after RoPE) and V:
    s = fp32(max |x| / 127) (stored as fp32), q = clamp(rint(fp32(x / s)), -127, 127)
    dequantised value = q * s;  s = 0 gives q = 0.

Every division and rounding decision is taken in IEEE fp32, as the device
does, so codes, packing and scales can be compared bit for bit.
"""
from __future__ import annotations

import numpy as np

GROUP = 128
NIBBLE_ORDER = (0, 2, 4, 6, 1, 3, 5, 7)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) to their exact fp32 values."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def f32_to_bf16_rne(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bits, round to nearest, ties to even (finite inputs)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    b = b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))
    return (b >> np.uint64(16)).astype(np.uint16)


def f32_to_bf16_ceil(x: np.ndarray) -> np.ndarray:
    """Non-negative fp32 -> bf16 bits, rounded toward +inf (smallest bf16 >= x)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    up = (b & np.uint64(0xFFFF)) != 0
    hi = b >> np.uint64(16)
    return (hi + up.astype(np.uint64)).astype(np.uint16)


# ---------------------------------------------------------------- int8 weights
def quantize_int8_rows(w_bits: np.ndarray):
    """int8 per-output-channel absmax quantiser.

    w_bits: bf16 bit patterns [N, K].  Returns (codes int8 [N, K],
    scale bf16 bits uint16 [N]).
    """
    w = bf16_to_f32(w_bits)
    amax = np.max(np.abs(w), axis=1)
    s = bf16_to_f32(f32_to_bf16_ceil(amax / np.float32(127.0)))
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(s[:, None] > 0, w / s[:, None], np.float32(0.0)).astype(np.float32)
    q = np.clip(np.rint(r), -127, 127).astype(np.int8)
    return q, f32_to_bf16_ceil(s)  # s is already a bf16 value: ceil is the identity


def dequant_int8(codes: np.ndarray, scale_bits: np.ndarray) -> np.ndarray:
    return codes.astype(np.float64) * bf16_to_f32(scale_bits).astype(np.float64)[:, None]


# ---------------------------------------------------------------- int4 weights
def quantize_int4_g128(w_bits: np.ndarray):
    """int4 asymmetric group-128 quantiser.

    w_bits: bf16 bit patterns [N, K], K % 128 == 0.  Returns (packed uint8
    [N, K/2], scale bf16 bits [N, K/128], zero bf16 bits [N, K/128]).
    """
    n, k = w_bits.shape
    assert k % GROUP == 0
    w = bf16_to_f32(w_bits).reshape(n, k // GROUP, GROUP)
    mn = np.minimum(np.float32(0.0), w.min(axis=2))
    mx = np.maximum(np.float32(0.0), w.max(axis=2))
    d = (mx - mn).astype(np.float32)
    s = bf16_to_f32(f32_to_bf16_ceil((d / np.float32(15.0)).astype(np.float32)))
    pos = s > 0
    with np.errstate(divide="ignore", invalid="ignore"):
        zr = np.where(pos, (-mn) / s, np.float32(0.0)).astype(np.float32)
        r = np.where(pos[..., None], w / s[..., None], np.float32(0.0)).astype(np.float32)
    # the zero point is an integer in [0, 15]; "+ 0" turns rint(-0.0) into +0
    z = np.clip(np.rint(zr), 0, 15) + np.float32(0.0)
    q = np.clip(np.rint(r) + z[..., None], 0, 15).astype(np.uint8).reshape(n, k)
    return pack_int4(q), f32_to_bf16_rne(s), f32_to_bf16_rne(z.astype(np.float32))


def pack_int4(q: np.ndarray) -> np.ndarray:
    """[N, K] codes 0..15 -> [N, K/2] bytes in the nibble order above."""
    n, k = q.shape
    nib = q.reshape(n, k // 8, 8)[..., list(NIBBLE_ORDER)]       # nibble i <- element ORDER[i]
    return (nib[..., 0::2] | (nib[..., 1::2] << np.uint8(4))).astype(np.uint8).reshape(n, k // 2)


def unpack_int4(packed: np.ndarray) -> np.ndarray:
    """[N, K/2] bytes -> [N, K] codes 0..15 (inverse of pack_int4)."""
    n, kh = packed.shape
    b = packed.reshape(n, kh // 4, 4)
    nib = np.empty((n, kh // 4, 8), dtype=np.uint8)
    nib[..., 0::2] = b & np.uint8(0x0F)
    nib[..., 1::2] = b >> np.uint8(4)
    q = np.empty_like(nib)
    q[..., list(NIBBLE_ORDER)] = nib
    return q.reshape(n, kh * 2)


def dequant_int4(packed, scale_bits, zero_bits) -> np.ndarray:
    q = unpack_int4(packed).astype(np.float64)
    n, k = q.shape
    s = bf16_to_f32(scale_bits).astype(np.float64)
    z = bf16_to_f32(zero_bits).astype(np.float64)
    q = q.reshape(n, k // GROUP, GROUP)
    return ((q - z[..., None]) * s[..., None]).reshape(n, k)


# ---------------------------------------------------------------- GPTQ4 (act order)
def g_idx_of(perm: np.ndarray) -> np.ndarray:
    """Group of every input channel: g_idx[perm[j]] = j // 128."""
    perm = np.asarray(perm, dtype=np.int64)
    g = np.empty(perm.shape[0], dtype=np.int64)
    g[perm] = np.arange(perm.shape[0]) // GROUP
    return g


def quantize_gptq4(w_bits: np.ndarray, perm: np.ndarray):
    """int4 over act-order groups.  w_bits: bf16 bits [N, K], perm: a
    permutation of range(K).  Returns (packed codes in act order [N, K/2],
    scale bits [N, K/128], zero bits [N, K/128]): the int4 rule on each
    group's values w[:, perm[128 g:128 g + 128]]."""
    perm = np.asarray(perm, dtype=np.int64)
    assert sorted(perm.tolist()) == list(range(w_bits.shape[1]))
    return quantize_int4_g128(np.ascontiguousarray(w_bits[:, perm]))


def codes_gptq4(packed: np.ndarray, perm: np.ndarray) -> np.ndarray:
    """Codes q[n, k] in channel order from the act-order storage."""
    qa = unpack_int4(packed)
    q = np.empty_like(qa)
    q[:, np.asarray(perm, dtype=np.int64)] = qa
    return q


def dequant_gptq4(packed, scale_bits, zero_bits, perm) -> np.ndarray:
    """W[n, k] = (q[n, k] - z[n, g_idx[k]]) * s[n, g_idx[k]] (channel order)."""
    q = codes_gptq4(packed, perm).astype(np.float64)
    g = g_idx_of(perm)
    s = bf16_to_f32(scale_bits).astype(np.float64)[:, g]
    z = bf16_to_f32(zero_bits).astype(np.float64)[:, g]
    return (q - z) * s


# ---------------------------------------------------------------- int8 KV cache
def quantize_kv_int8(x_bits: np.ndarray):
    """Per-row (token, KV head) absmax int8 quantiser over the last axis.

    x_bits: bf16 bit patterns [..., hd].  Returns (codes int8 [..., hd],
    scale fp32 [...]).
    """
    x = bf16_to_f32(x_bits)
    s = (np.max(np.abs(x), axis=-1) / np.float32(127.0)).astype(np.float32)
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(s[..., None] > 0, x / s[..., None], np.float32(0.0)).astype(np.float32)
    q = np.clip(np.rint(r), -127, 127).astype(np.int8)
    return q, s


def dequant_kv_int8(codes: np.ndarray, scales: np.ndarray) -> np.ndarray:
    return codes.astype(np.float64) * scales.astype(np.float64)[..., None]


# ---------------------------------------------------------------- one entry point
def quantize_weight(w_bits: np.ndarray, wquant: int, perm=None):
    """wquant 0 = bf16 (no codes), 1 = int8 per channel, 2 = int4 group 128,
    3 = GPTQ4 (int4 over the act order perm).

    Returns (payload dict, dequantised fp64 matrix).
    """
    if wquant == 3:
        p, s, z = quantize_gptq4(w_bits, perm)
        return {"codes": p, "scales": s, "zeros": z, "perm": np.asarray(perm, dtype=np.int32)}, \
            dequant_gptq4(p, s, z, perm)
    if wquant == 0:
        return {"w": w_bits}, bf16_to_f32(w_bits).astype(np.float64)
    if wquant == 1:
        q, s = quantize_int8_rows(w_bits)
        return {"codes": q, "scales": s}, dequant_int8(q, s)
    if wquant == 2:
        p, s, z = quantize_int4_g128(w_bits)
        return {"codes": p, "scales": s, "zeros": z}, dequant_int4(p, s, z)
    raise ValueError(wquant)
