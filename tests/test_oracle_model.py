"""Pins of the oracle's forward pass (CPU only).

Each test fixes a piece of the fingerprint block against a hand-derived value,
a closed form or an invariant that a plausible mistake (a dropped term, a
swapped operand, a wrong index or sign) would break.  The paper fixes the
fingerprint's components (Sec. 1 "Our work"; Sec. 5.1) and the KV-cache
property that decode costs the same per token (Sec. 5.3, before Eq. 1); the
block details are the Llama-2 reading stated in oracle/model.py.
"""
import json
import os

import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import quant
from tests.conftest import GOLDEN

with open(os.path.join(GOLDEN, "components_example.json")) as _f:
    G = json.load(_f)


# ---------------------------------------------------------------- components
def test_rmsnorm_hand_example_and_unit_rms():
    g = G["rmsnorm"]
    y = M.rmsnorm(np.array(g["x"]), np.array(g["g"]), 0.0)
    assert np.allclose(y, g["y"], rtol=1e-15, atol=0)
    x = np.random.default_rng(0).normal(size=(7, 64)) * 5
    y = M.rmsnorm(x, np.ones(64), 0.0)
    assert np.allclose(np.sqrt(np.mean(y * y, axis=-1)), 1.0, rtol=1e-14)
    # eps enters inside the root: x = 0 stays 0, tiny x is damped
    assert np.all(M.rmsnorm(np.zeros((1, 8)), np.ones(8), 1e-5) == 0)


def test_silu_hand_values_and_limits():
    g = G["silu"]
    assert np.allclose(M.silu(np.array(g["x"])), g["y"], rtol=1e-15, atol=0)
    assert abs(M.silu(np.array(60.0)) - 60.0) < 1e-20
    assert abs(M.silu(np.array(-60.0))) < 1e-24


def test_rope_hand_examples():
    g = G["rope"]
    for c in g["cases"]:
        x = np.array(c["x"], dtype=np.float64).reshape(1, 1, g["hd"])
        y = M.rope(x, np.array([c["pos"]]), g["base"]).reshape(-1)
        assert np.allclose(y, c["y"], rtol=0, atol=1e-15)


def test_rope_identity_norm_and_relative_position():
    rng = np.random.default_rng(1)
    hd = 128
    x = rng.normal(size=(1, 1, hd))
    assert np.array_equal(M.rope(x, np.array([0]), 1e4), x)
    y = M.rope(x, np.array([37]), 1e4)
    pair = lambda v: v[..., : hd // 2] ** 2 + v[..., hd // 2:] ** 2
    assert np.allclose(pair(y), pair(x), rtol=1e-13)
    q, k = rng.normal(size=(2, 1, 1, hd))
    dots = [np.sum(M.rope(q, np.array([p + 5]), 1e4) * M.rope(k, np.array([p]), 1e4)) for p in (0, 9, 300)]
    assert np.allclose(dots, dots[0], rtol=1e-12)


def test_attention_two_keys_hand_example():
    g = G["attention_two_keys"]
    q = np.array(g["q"], float).reshape(1, 1, 4)
    k = np.array(g["k"], float).reshape(2, 1, 4)
    v = np.array(g["v"], float).reshape(2, 1, 4)
    o = M.attention(q, np.array([1]), k, v).reshape(-1)
    assert np.allclose(o, g["o"], rtol=1e-15, atol=1e-16)


def test_attention_invariants():
    rng = np.random.default_rng(2)
    hd = 64
    # one key returns V exactly
    v = rng.normal(size=(1, 2, hd))
    o = M.attention(rng.normal(size=(1, 4, hd)), np.array([0]), rng.normal(size=(1, 2, hd)), v)
    assert np.array_equal(o[0, 0], v[0, 0]) and np.array_equal(o[0, 3], v[0, 1])
    # equal keys return the mean of V
    k = np.repeat(rng.normal(size=(1, 1, hd)), 9, axis=0)
    v = rng.normal(size=(9, 1, hd))
    o = M.attention(rng.normal(size=(1, 1, hd)), np.array([8]), k, v)
    assert np.allclose(o[0, 0], v[:, 0].mean(axis=0), rtol=1e-13)
    # softmax rows sum to 1
    s = M.softmax(rng.normal(size=(5, 33)) * 10)
    assert np.allclose(s.sum(-1), 1.0, rtol=0, atol=1e-12)
    # causal: the query at position 0 sees key 0 only
    k = rng.normal(size=(6, 1, hd))
    v = rng.normal(size=(6, 1, hd))
    o = M.attention(rng.normal(size=(2, 1, hd)), np.array([0, 5]), k, v)
    assert np.array_equal(o[0, 0], v[0, 0])


def test_attention_gqa_head_mapping():
    """Query head j reads KV head j // (H / Hkv): with H = 4, Hkv = 2 and a
    constant V per KV head, heads 0-1 return 1 and heads 2-3 return 2."""
    hd = 8
    rng = np.random.default_rng(3)
    k = rng.normal(size=(5, 2, hd))
    v = np.zeros((5, 2, hd))
    v[:, 0] = 1.0
    v[:, 1] = 2.0
    o = M.attention(rng.normal(size=(1, 4, hd)), np.array([4]), k, v)
    assert np.allclose(o[0, :, 0], [1, 1, 2, 2], rtol=1e-14)
    # G = 1 (MHA) equals running each head alone
    q = rng.normal(size=(3, 2, hd))
    vv = rng.normal(size=(5, 2, hd))
    o = M.attention(q, np.array([2, 3, 4]), k, vv)
    for j in range(2):
        oj = M.attention(q[:, j:j + 1], np.array([2, 3, 4]), k[:, j:j + 1], vv[:, j:j + 1])
        assert np.array_equal(oj[:, 0], o[:, j])


def test_argmax_ties_lowest_id():
    x = np.array([[0.0, 3.0, 3.0, 1.0], [-1.0, -1.0, -2.0, -1.0]])
    assert M.argmax(x).tolist() == [1, 0]


# ---------------------------------------------------------------- whole block
def _tiny_arch(**kw):
    base = dict(n_layers=1, hidden=64, n_heads=4, n_kv_heads=2, head_dim=16, ffn=96, vocab=50)
    base.update(kw)
    return M.Arch(**base)


def _weights(arch, wq, seed=0, gains="random"):
    def get(layer, t, shape):
        if len(shape) == 1:
            if gains == "ones":
                return synth.f32_to_bf16_bits(np.ones(shape, np.float32))
            return synth.uniform_bf16(seed, 500 + 16 * (layer + 1) + t, shape, 0.5, 1.5)
        # larger than N(0, 0.02) so the tiny model has non-trivial attention
        return synth.f32_to_bf16_bits(quant.bf16_to_f32(synth.weight_bf16(seed, layer, t, shape)) * np.float32(8))
    return M.build_weights(arch, wq, get)


def test_ffn_block_hand_example():
    """d = 2, f = 1, zero attention: h -> [1 + silu(y0) * y1, 2]."""
    g = G["ffn_block"]
    arch = M.Arch(n_layers=1, hidden=2, n_heads=1, n_kv_heads=1, head_dim=2, ffn=1, vocab=3, rms_eps=0.0)
    w = {(0, "attn_norm"): np.ones(2), (0, "ffn_norm"): np.ones(2),
         (0, "wqkv"): np.zeros((6, 2)), (0, "wo"): np.ones((2, 2)),
         (0, "wgu"): np.array([[1.0, 0.0], [0.0, 1.0]]), (0, "wdown"): np.array([[1.0], [0.0]])}
    fp = M.Fingerprint(arch, w, M.KV_BF16, 1, 4)
    h = fp._block(0, np.array(g["h"]).reshape(1, 1, 2), 0)
    assert np.allclose(h.reshape(-1), g["h_out"], rtol=1e-15)


@pytest.mark.parametrize("wq,kvq", [(0, 0), (1, 1), (2, 0)])
def test_decode_equals_prefill_row(wq, kvq):
    """KV-cache equivalence: prefill of S+1 tokens and prefill of S tokens then
    one decode step give the same last-position logits."""
    arch = _tiny_arch(n_layers=2, hidden=128, head_dim=32, ffn=256)
    w, _ = _weights(arch, wq)
    toks = synth.tokens(9, 2 * 7, arch.vocab).reshape(2, 7)
    a = M.Fingerprint(arch, w, kvq, 2, 16)
    full = a.prefill(toks)
    b = M.Fingerprint(arch, w, kvq, 2, 16)
    b.prefill(toks[:, :6])
    step = b.decode(toks[:, 6])
    assert np.allclose(step["logits"], full["logits"], rtol=1e-11, atol=1e-12)
    for hf, hs in zip(full["hidden"], step["hidden"]):
        assert np.allclose(hs[:, 0], hf[:, -1], rtol=1e-11, atol=1e-12)


def test_zero_sublayers_leave_embedding():
    arch = _tiny_arch()
    w, _ = _weights(arch, 0)
    w[(0, "wo")] = np.zeros_like(w[(0, "wo")])
    w[(0, "wdown")] = np.zeros_like(w[(0, "wdown")])
    toks = np.array([[3, 7, 1]])
    out = M.Fingerprint(arch, w, 0, 1, 8).prefill(toks)
    assert np.array_equal(out["hidden"][0][0], w["embed"][toks[0]])


def test_lm_head_reads_final_norm():
    arch = _tiny_arch(vocab=64)
    w, _ = _weights(arch, 0)
    w["lm_head"] = np.eye(64)
    out = M.Fingerprint(arch, w, 0, 1, 8).prefill(np.array([[5, 6]]))
    h = out["hidden"][-1][0, -1]
    assert np.allclose(out["logits"][0], M.rmsnorm(h, w["final_norm"], arch.rms_eps), rtol=1e-15)


def test_batch_rows_independent():
    arch = _tiny_arch()
    w, _ = _weights(arch, 1)
    toks = synth.tokens(4, 3 * 5, arch.vocab).reshape(3, 5)
    a = M.Fingerprint(arch, w, 1, 3, 8).prefill(toks)
    b = M.Fingerprint(arch, w, 1, 3, 8).prefill(toks[::-1])
    assert np.allclose(a["logits"][::-1], b["logits"], rtol=1e-13, atol=1e-15)


def test_store_kv_modes():
    rng = np.random.default_rng(5)
    x = rng.normal(size=(3, 2, 16))
    r = M.store_kv(x, M.KV_BF16)
    assert np.all(np.abs(r - x) <= np.abs(x) * 2.0 ** -8)
    r8 = M.store_kv(x, M.KV_INT8)
    s = np.abs(r).max(axis=-1, keepdims=True) / 127
    assert np.all(np.abs(r8 - r) <= s / 2 * (1 + 1e-6))


# ---------------------------------------------------------------- a whole block, brute force
def _bf16_scalar(x):
    """fp64 -> fp32 -> bf16, round to nearest even, on one scalar (bit arithmetic)."""
    import struct

    b = struct.unpack("<I", struct.pack("<f", float(np.float32(x))))[0]
    b = (b + 0x7FFF + ((b >> 16) & 1)) >> 16
    return struct.unpack("<f", struct.pack("<I", (b << 16) & 0xFFFFFFFF))[0]


def _block_by_loops(a, w, h):
    """One decoder block over h [T][d] at positions 0 .. T-1, every sum an
    explicit scalar loop from the definitions (pre-norm RMSNorm, fused
    [q | k | v] rows, rotate-half RoPE on q and k, bf16-rounded cache,
    causal GQA softmax attention, O projection, SwiGLU over [gate | up]
    rows, down projection, two residual adds)."""
    import math

    T, d = len(h), a.hidden
    H, G, hd, f = a.n_heads, a.n_kv_heads, a.head_dim, a.ffn

    def rms(x, g):
        ms = sum(v * v for v in x) / len(x)
        return [x[i] / math.sqrt(ms + a.rms_eps) * g[i] for i in range(len(x))]

    def mat_row(W, r, x):
        return sum(W[r][k] * x[k] for k in range(len(x)))

    def rot(x, p):
        out = list(x)
        for i in range(hd // 2):
            th = p * a.rope_base ** (-2.0 * i / hd)
            c, s = math.cos(th), math.sin(th)
            out[i] = x[i] * c - x[i + hd // 2] * s
            out[i + hd // 2] = x[i + hd // 2] * c + x[i] * s
        return out

    Wqkv, Wo, Wgu, Wd = w[(0, "wqkv")], w[(0, "wo")], w[(0, "wgu")], w[(0, "wdown")]
    q, k, v = [], [], []
    for t in range(T):
        y = rms(h[t], w[(0, "attn_norm")])
        q.append([rot([mat_row(Wqkv, j * hd + i, y) for i in range(hd)], t) for j in range(H)])
        k.append([[_bf16_scalar(e) for e in rot([mat_row(Wqkv, H * hd + j * hd + i, y) for i in range(hd)], t)]
                  for j in range(G)])
        v.append([[_bf16_scalar(mat_row(Wqkv, (H + G) * hd + j * hd + i, y)) for i in range(hd)] for j in range(G)])
    out = []
    for t in range(T):
        o = []
        for j in range(H):
            kv = j // (H // G)
            sc = [sum(q[t][j][i] * k[u][kv][i] for i in range(hd)) / math.sqrt(hd) for u in range(t + 1)]
            m = max(sc)
            e = [math.exp(s - m) for s in sc]
            z = sum(e)
            o += [sum(e[u] / z * v[u][kv][i] for u in range(t + 1)) for i in range(hd)]
        h1 = [h[t][r] + mat_row(Wo, r, o) for r in range(d)]
        y2 = rms(h1, w[(0, "ffn_norm")])
        act = []
        for c in range(f):
            gt, up = mat_row(Wgu, c, y2), mat_row(Wgu, f + c, y2)
            act.append(gt / (1.0 + math.exp(-gt)) * up)
        out.append([h1[r] + mat_row(Wd, r, act) for r in range(d)])
    return out


def test_block_matches_brute_force_loops():
    """The oracle's vectorised block against the same block written out as
    scalar loops on a tiny GQA shape (H 4, Hkv 2, hd 4, d 8, f 6, T 5): a
    transposed weight, a wrong q/k/v or gate/up row range, RoPE on v or a
    wrong head mapping all change the result by O(1)."""
    rng = np.random.default_rng(11)
    a = M.Arch(n_layers=1, hidden=8, n_heads=4, n_kv_heads=2, head_dim=4, ffn=6, vocab=7, rms_eps=1e-5)
    w = {(0, "attn_norm"): rng.uniform(0.5, 1.5, 8), (0, "ffn_norm"): rng.uniform(0.5, 1.5, 8),
         (0, "wqkv"): rng.normal(0, 0.5, ((4 + 2 * 2) * 4, 8)), (0, "wo"): rng.normal(0, 0.5, (8, 16)),
         (0, "wgu"): rng.normal(0, 0.5, (12, 8)), (0, "wdown"): rng.normal(0, 0.5, (8, 6))}
    h = rng.normal(0, 1, (5, 8))
    fp = M.Fingerprint(a, w, M.KV_BF16, 1, 8)
    got = fp._block(0, h[None], 0)[0]
    ref = np.array(_block_by_loops(a, w, h.tolist()))
    assert np.allclose(got, ref, rtol=1e-10, atol=1e-12), np.max(np.abs(got - ref))
