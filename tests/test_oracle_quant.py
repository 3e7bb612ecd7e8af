"""Pins of the oracle's quantisers (CPU only).

The paper names the formats (INT8 / INT4 weight-only, INT8 KV cache; Sec. 3.2,
table "Models and configurations") and their memory effect, not their
arithmetic; the readings are stated in oracle/quant.py.  These tests pin the
oracle to them with hand-derived fixtures, exact error bounds and brute force
over every code, independent of how the oracle computes.
"""
import json
import os

import numpy as np
import pytest

import synth
from oracle import quant
from tests.conftest import GOLDEN


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _weights(n, k, seed=3):
    w = synth.weight_bf16(seed, 0, 1, (n, k))
    # special rows: all zero, a single outlier, constant, all negative
    w[0] = 0
    w[1, :] = 0
    w[1, 5] = synth.f32_to_bf16_bits(np.array([0.75], np.float32))[0]
    w[2, :] = synth.f32_to_bf16_bits(np.array([-0.125], np.float32))[0]
    w[3] = synth.f32_to_bf16_bits(-np.abs(quant.bf16_to_f32(w[3])))
    return w


def _exact(x):
    return np.asarray(x, dtype=np.float64)


# ---------------------------------------------------------------- int8
def test_int8_hand_example():
    g = _golden("int8_row_example.json")
    w = np.array([g["w_bits"]], dtype=np.uint16)
    q, s = quant.quantize_int8_rows(w)
    assert int(s[0]) == g["scale_bits"]
    assert float(quant.bf16_to_f32(s)[0]) == g["scale_value"]
    assert q[0].tolist() == g["codes"]


def test_int8_scale_is_smallest_bf16_covering_range():
    w = _weights(16, 256)
    q, s_bits = quant.quantize_int8_rows(w)
    s = _exact(quant.bf16_to_f32(s_bits))
    amax = np.max(np.abs(_exact(quant.bf16_to_f32(w))), axis=1)
    # s * 127 >= amax (no clamping needed); the next bf16 below s is too small
    # for fp32(amax / 127).
    assert np.all(s * 127 >= amax)
    t32 = (amax.astype(np.float32) / np.float32(127)).astype(np.float64)
    below = _exact(quant.bf16_to_f32((s_bits.astype(np.int32) - 1).clip(0).astype(np.uint16)))
    nz = amax > 0
    assert np.all(below[nz] < t32[nz])
    assert s[0] == 0 and np.all(q[0] == 0)


def test_int8_codes_are_nearest_by_brute_force():
    w = _weights(8, 128)
    q, s_bits = quant.quantize_int8_rows(w)
    wf = _exact(quant.bf16_to_f32(w))
    s = _exact(quant.bf16_to_f32(s_bits))
    cand = np.arange(-127, 128, dtype=np.float64)
    for n in range(w.shape[0]):
        err = np.abs(wf[n][:, None] - cand[None, :] * s[n])
        best = err.min(axis=1)
        mine = np.abs(wf[n] - q[n] * s[n])
        # fp32 division can move a value sitting on a half-code boundary by one ulp
        assert np.all(mine <= best + 2.0 ** -22 * max(s[n], 1e-30) * 128)
        assert np.all(mine <= s[n] / 2 * (1 + 2.0 ** -20))
    assert q.min() >= -127 and q.max() <= 127


def test_int8_dequant_error_bound_large():
    w = synth.weight_bf16(11, 1, 6, (64, 4096))
    q, s_bits = quant.quantize_int8_rows(w)
    err = np.abs(quant.dequant_int8(q, s_bits) - _exact(quant.bf16_to_f32(w)))
    s = _exact(quant.bf16_to_f32(s_bits))
    assert np.all(err <= s[:, None] / 2 * (1 + 2.0 ** -20))


# ---------------------------------------------------------------- int4
def test_int4_hand_example():
    g = _golden("int4_group_example.json")
    w = np.zeros((1, g["k"]), dtype=np.uint16)
    for i, b in g["w_nonzero"].items():
        w[0, int(i)] = b
    p, s, z = quant.quantize_int4_g128(w)
    assert int(s[0, 0]) == g["scale_bits"]
    assert int(z[0, 0]) == g["zero_bits"]
    assert p[0, :4].tolist() == g["first_bytes"]
    assert np.all(p[0, 4:] == 0x55)
    deq = quant.dequant_int4(p, s, z)
    assert deq[0, :4].tolist() == g["dequant_first"]


def test_int4_codes_nearest_and_bounded():
    w = _weights(8, 512)
    p, s_bits, z_bits = quant.quantize_int4_g128(w)
    q = quant.unpack_int4(p).astype(np.float64)
    s = _exact(quant.bf16_to_f32(s_bits))
    z = _exact(quant.bf16_to_f32(z_bits))
    assert np.all(z == np.round(z)) and z.min() >= 0 and z.max() <= 15
    wf = _exact(quant.bf16_to_f32(w))
    cand = np.arange(16, dtype=np.float64)
    for n in range(w.shape[0]):
        for g in range(w.shape[1] // 128):
            seg = wf[n, g * 128:(g + 1) * 128]
            sg, zg = s[n, g], z[n, g]
            mine = np.abs(seg - (q[n, g * 128:(g + 1) * 128] - zg) * sg)
            best = np.abs(seg[:, None] - (cand[None, :] - zg) * sg).min(axis=1)
            assert np.all(mine <= best + 2.0 ** -22 * max(sg, 1e-30) * 16)
            assert np.all(mine <= sg / 2 * (1 + 2.0 ** -20))
    # zero row -> s = z = q = 0; the stored zero point is +0 (an integer, no sign)
    assert np.all(s[0] == 0) and np.all(z[0] == 0) and np.all(q[0] == 0)
    assert np.all(z_bits >> 15 == 0)


def test_int4_packing_order_and_roundtrip():
    rng = np.random.default_rng(0)
    q = rng.integers(0, 16, size=(3, 256), dtype=np.uint8)
    packed = quant.pack_int4(q)
    assert packed.shape == (3, 128)
    assert np.array_equal(quant.unpack_int4(packed), q)
    # word w of a row holds elements 8w .. 8w+7; nibble i holds element (0,2,4,6,1,3,5,7)[i]
    word = packed[1, 4:8].astype(np.uint32)
    word = int(word[0] | (word[1] << 8) | (word[2] << 16) | (word[3] << 24))
    for i, e in enumerate((0, 2, 4, 6, 1, 3, 5, 7)):
        assert (word >> (4 * i)) & 0xF == q[1, 8 + e]
    # the 0x000F000F mask of the word shifted by 4s picks elements 2s and 2s+1
    for s_ in range(4):
        pair = (word >> (4 * s_)) & 0x000F000F
        assert (pair & 0xF, pair >> 16) == (q[1, 8 + 2 * s_], q[1, 8 + 2 * s_ + 1])


def test_int4_scale_covers_range():
    w = synth.weight_bf16(5, 0, 7, (32, 1024))
    p, s_bits, z_bits = quant.quantize_int4_g128(w)
    wf = _exact(quant.bf16_to_f32(w)).reshape(32, 8, 128)
    mn = np.minimum(0, wf.min(axis=2))
    mx = np.maximum(0, wf.max(axis=2))
    s = _exact(quant.bf16_to_f32(s_bits))
    # s >= (mx - mn) / 15 up to one fp32 rounding of the difference
    assert np.all(s * 15 >= (mx - mn) * (1 - 2.0 ** -23))
    err = np.abs(quant.dequant_int4(p, s_bits, z_bits).reshape(32, 8, 128) - wf)
    assert np.all(err <= s[..., None] / 2 * (1 + 2.0 ** -20))


# ---------------------------------------------------------------- int8 KV
def test_kv_int8_nearest_and_bound():
    x = synth.uniform_bf16(7, 3, (5, 4, 64), -3.0, 3.0)
    x[0, 0] = 0
    q, s = quant.quantize_kv_int8(x)
    xf = _exact(quant.bf16_to_f32(x))
    amax = np.abs(xf).max(axis=-1)
    assert np.array_equal(s, (amax.astype(np.float32) / np.float32(127)).astype(np.float32))
    s64 = s.astype(np.float64)
    mine = np.abs(xf - q * s64[..., None])
    cand = np.arange(-127, 128, dtype=np.float64)
    best = np.abs(xf[..., None] - cand * s64[..., None, None]).min(axis=-1)
    assert np.all(mine <= best + 2.0 ** -22 * s64[..., None] * 128)
    assert np.all(mine <= s64[..., None] / 2 * (1 + 2.0 ** -20) + 1e-300)
    assert s[0, 0] == 0 and np.all(q[0, 0] == 0)


@pytest.mark.parametrize("wq", [0, 1, 2])
def test_quantize_weight_dispatch(wq):
    w = synth.weight_bf16(1, 0, 1, (4, 256))
    payload, deq = quant.quantize_weight(w, wq)
    ref = _exact(quant.bf16_to_f32(w))
    tol = {0: 0.0, 1: 0.02 / 127 * 4, 2: 0.02 / 15 * 8}[wq]
    assert np.max(np.abs(deq - ref)) <= tol


# ---------------------------------------------------------------- GPTQ4 (act order)
def _fixture_gptq4():
    g = _golden("gptq4_act_order_example.json")
    w = np.zeros((1, g["k"]), dtype=np.uint16)
    for k, v in g["w_nonzero"].items():
        w[0, int(k)] = v
    perm = np.concatenate([np.arange(1, g["k"], 2), np.arange(0, g["k"], 2)]).astype(np.int32)
    return g, w, perm


def test_gptq4_hand_example():
    """The act-order groups, their scale / zero, the act-order packing and the
    channel-order dequantisation of the hand-worked fixture."""
    g, w, perm = _fixture_gptq4()
    p, s, z = quant.quantize_gptq4(w, perm)
    assert s[0].tolist() == g["scale_bits"] and z[0].tolist() == g["zero_bits"]
    for i, b in g["bytes_at"].items():
        assert int(p[0, int(i)]) == b, i
    d = quant.dequant_gptq4(p, s, z, perm)
    for i, v in g["dequant_at"].items():
        assert d[0, int(i)] == v, i
    gi = quant.g_idx_of(perm)
    assert np.all(gi[1::2] == 0) and np.all(gi[0::2] == 1)


def test_gptq4_identity_order_is_int4():
    """With the identity act order GPTQ4 is the int4 group-128 format, bit for bit."""
    w = _weights(12, 512)
    ident = np.arange(512, dtype=np.int32)
    for a, b in zip(quant.quantize_gptq4(w, ident), quant.quantize_int4_g128(w)):
        assert np.array_equal(a, b)
    assert np.array_equal(quant.dequant_gptq4(*quant.quantize_gptq4(w, ident), ident),
                          quant.dequant_int4(*quant.quantize_int4_g128(w)))


def test_gptq4_groups_follow_the_act_order():
    """Every group holds 128 channels, g_idx[perm[j]] = j // 128, and each
    channel's error is at most half its own group's scale."""
    k = 768
    perm = synth.act_order(5, 1, 2, k)
    gi = quant.g_idx_of(perm)
    assert np.array_equal(np.bincount(gi), np.full(k // 128, 128))
    assert np.array_equal(gi[perm], np.arange(k) // 128)
    w = _weights(9, k)
    p, s, z = quant.quantize_gptq4(w, perm)
    err = np.abs(quant.dequant_gptq4(p, s, z, perm) - _exact(quant.bf16_to_f32(w)))
    half = _exact(quant.bf16_to_f32(s))[:, gi] / 2
    assert np.all(err <= half * (1 + 2 ** -20) + 1e-30)
    q = quant.codes_gptq4(p, perm)
    assert q.min() >= 0 and q.max() <= 15


def test_gptq4_product_equals_reordered_int4_product():
    """x W^T with W dequantised in channel order equals x[:, perm] W_a^T, W_a
    the act-order storage read as plain int4: the identity the device uses.
    A perm / inverse mix-up or a group taken in channel order fails it."""
    k = 512
    perm = synth.act_order(3, 0, 1, k)
    assert not np.array_equal(perm[perm], np.arange(k))  # not an involution
    w = _weights(6, k)
    p, s, z = quant.quantize_gptq4(w, perm)
    x = quant.bf16_to_f32(synth.uniform_bf16(4, 9, (5, k), -1.0, 1.0)).astype(np.float64)
    y = x @ quant.dequant_gptq4(p, s, z, perm).T
    ya = x[:, perm] @ quant.dequant_int4(p, s, z).T
    assert np.allclose(y, ya, rtol=0, atol=1e-12)
    # taking the groups in channel order instead gives different weights
    assert not np.allclose(quant.dequant_gptq4(p, s, z, perm), quant.dequant_int4(p, s, z))
