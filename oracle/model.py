"""Fingerprint forward pass of the oracle, in fp64 (test infrastructure only).

The fingerprint is the LLM rebuilt with the same components but one or two
hidden layers (Sec. 1, "Our work"; Sec. 5.1).  The block is read as the
Llama-2 decoder block, which the paper does not spell out:

    h0[b, s]  = E[tok[b, s]]                                   embedding
    for each block:
        y       = RMSNorm(h; g_attn)                           x / sqrt(mean x^2 + eps) * g
        q, k, v = y Wq^T, y Wk^T, y Wv^T
        q, k    = RoPE(q, p), RoPE(k, p)                       rotate-half, theta_i = base^(-2i/hd)
        cache  <- k, v at position p                           stored as the KV config says
        o       = softmax(q K^T / sqrt(hd) + causal) V         query head j reads KV head j // (H / Hkv)
        h       = h + o Wo^T
        y       = RMSNorm(h; g_ffn)
        h       = h + (silu(y Wg^T) * (y Wu^T)) Wd^T
    logits = RMSNorm(h_last; g_final) W_head^T,   token = argmax (lowest id on ties)

Decode appends one position per sequence and attends over every cached
position including itself: the KV cache removes recomputation so each new
token costs the same (Sec. 5.3, before Eq. 1).  Both prefill and decode
attention read K and V back from the cache, so with a bf16 cache they see
bf16-rounded values and with an int8 cache the dequantised codes.

Nothing is rounded between steps except the cache store (fp64 -> fp32 ->
bf16, both round-to-nearest-even) and the int8 KV quantiser of ``quant``.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

from . import quant

KV_BF16, KV_INT8 = 0, 1


@dataclass(frozen=True)
class Arch:
    n_layers: int
    hidden: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rms_eps: float = 1e-5
    rope_base: float = 10000.0

    @property
    def q_dim(self):
        return self.n_heads * self.head_dim

    @property
    def kv_dim(self):
        return self.n_kv_heads * self.head_dim


# ------------------------------------------------------------------ components
def rmsnorm(x, g, eps):
    """RMSNorm over the last axis: x / sqrt(mean(x^2) + eps) * g."""
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def rope_inv_freq(hd, base):
    """theta_i = base^(-2 i / hd), i = 0 .. hd/2 - 1."""
    return np.power(float(base), -2.0 * np.arange(hd // 2, dtype=np.float64) / hd)


def rope(x, pos, base):
    """Rotate-half RoPE: pair (i, i + hd/2) is rotated by angle pos * theta_i.

    x: [..., T, nh, hd]; pos: broadcastable to [..., T].
    """
    hd = x.shape[-1]
    ang = np.asarray(pos, dtype=np.float64)[..., None] * rope_inv_freq(hd, base)
    c = np.cos(ang)[..., None, :]
    s = np.sin(ang)[..., None, :]
    x1, x2 = x[..., : hd // 2], x[..., hd // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x):
    return x / (1.0 + np.exp(-x))


def softmax(s, axis=-1):
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def attention(q, qpos, k, v):
    """Causal grouped-query attention for one sequence.

    q: [Tq, H, hd] at absolute positions qpos [Tq]; k, v: [Tk, Hkv, hd] at
    positions 0 .. Tk-1.  Query head j reads KV head j // (H / Hkv).
    Returns [Tq, H, hd].
    """
    tq, nh, hd = q.shape
    tk, nkv, _ = k.shape
    g = nh // nkv
    mask = np.arange(tk)[None, :] > np.asarray(qpos)[:, None]
    out = np.empty((tq, nh, hd), dtype=np.float64)
    for j in range(nh):
        sc = q[:, j, :] @ k[:, j // g, :].T / np.sqrt(hd)
        sc = np.where(mask, -np.inf, sc)
        out[:, j, :] = softmax(sc) @ v[:, j // g, :]
    return out


def round_bf16(x):
    """fp64 -> fp32 -> bf16 (both round to nearest even), returned as fp64."""
    return quant.bf16_to_f32(quant.f32_to_bf16_rne(np.asarray(x, np.float64).astype(np.float32))).astype(np.float64)


def store_kv(x, kvquant):
    """Value the cache holds for x [..., hd]: bf16-rounded, or int8 codes of the bf16 value."""
    if kvquant == KV_BF16:
        return round_bf16(x)
    bits = quant.f32_to_bf16_rne(np.asarray(x, np.float64).astype(np.float32))
    codes, scales = quant.quantize_kv_int8(bits)
    return quant.dequant_kv_int8(codes, scales)


# ------------------------------------------------------------------ weights
LAYER_TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "wgate", "wup", "wdown")
GLOBAL_TENSORS = ("embed", "final_norm", "lm_head")


def tensor_shape(arch: Arch, layer: int, tensor: int):
    d, f = arch.hidden, arch.ffn
    if layer < 0:
        return [(arch.vocab, d), (d,), (arch.vocab, d)][tensor]
    return [(d,), (arch.q_dim, d), (arch.kv_dim, d), (arch.kv_dim, d), (d, arch.q_dim),
            (d,), (f, d), (f, d), (d, f)][tensor]


def build_weights(arch: Arch, wquant: int, get_bf16, map_fn=map, act_order=None):
    """Quantise bf16 weights the way the configuration says.

    get_bf16(layer, tensor, shape) -> bf16 bit patterns.  Linear layers of
    the blocks are quantised per ``wquant`` as the fused matrices
    Wqkv = [Wq; Wk; Wv] and Wgu = [Wgate; Wup] (row-wise quantisers, so
    fusing changes no code).  Embedding, norm gains and the LM head stay
    bf16.  Returns (fp64 weights for the forward pass, quantised payloads).
    ``map_fn`` applies the quantiser to the matrices (a thread pool's map
    spreads the large ones over cores; the result does not depend on it).
    GPTQ4 (wquant 3) takes each fused matrix's act order from
    ``act_order(layer, matrix, K)``, matrix 0..3 = Wqkv, Wo, Wgu, Wdown.
    """
    w, payload = {}, {}
    f64 = lambda b: quant.bf16_to_f32(b).astype(np.float64)
    for t, name in enumerate(GLOBAL_TENSORS):
        w[name] = f64(get_bf16(-1, t, tensor_shape(arch, -1, t)))
    jobs = []
    for l in range(arch.n_layers):
        raw = {name: get_bf16(l, t, tensor_shape(arch, l, t)) for t, name in enumerate(LAYER_TENSORS)}
        w[(l, "attn_norm")] = f64(raw["attn_norm"])
        w[(l, "ffn_norm")] = f64(raw["ffn_norm"])
        mats = {"wqkv": np.concatenate([raw["wq"], raw["wk"], raw["wv"]]),
                "wo": raw["wo"],
                "wgu": np.concatenate([raw["wgate"], raw["wup"]]),
                "wdown": raw["wdown"]}
        jobs += [((l, name), bits, act_order(l, m, bits.shape[1]) if wquant == 3 else None)
                 for m, (name, bits) in enumerate(mats.items())]
    for (key, _, _), res in zip(jobs, map_fn(lambda j: quant.quantize_weight(j[1], wquant, j[2]), jobs)):
        payload[key], w[key] = res
    return w, payload


# ------------------------------------------------------------------ the model
class Fingerprint:
    """Greedy generation with a KV cache, one batch of equal-length sequences."""

    def __init__(self, arch: Arch, weights, kvquant: int, batch: int, max_context: int):
        self.a, self.w, self.kvq, self.B, self.T = arch, weights, kvquant, batch, max_context
        shape = (arch.n_layers, batch, max_context, arch.n_kv_heads, arch.head_dim)
        self.k_cache = np.zeros(shape)
        self.v_cache = np.zeros(shape)
        self.length = 0

    def _block(self, l, h, pos):
        """One decoder block over h [B, T, d] at positions pos .. pos+T-1."""
        a, w = self.a, self.w
        B, T, _ = h.shape
        p = np.arange(pos, pos + T)
        y = rmsnorm(h, w[(l, "attn_norm")], a.rms_eps)
        qkv = y @ w[(l, "wqkv")].T
        q = qkv[..., : a.q_dim].reshape(B, T, a.n_heads, a.head_dim)
        k = qkv[..., a.q_dim: a.q_dim + a.kv_dim].reshape(B, T, a.n_kv_heads, a.head_dim)
        v = qkv[..., a.q_dim + a.kv_dim:].reshape(B, T, a.n_kv_heads, a.head_dim)
        q = rope(q, p, a.rope_base)
        k = rope(k, p, a.rope_base)
        self.k_cache[l, :, pos: pos + T] = store_kv(k, self.kvq)
        self.v_cache[l, :, pos: pos + T] = store_kv(v, self.kvq)
        o = np.stack([attention(q[b], p, self.k_cache[l, b, : pos + T], self.v_cache[l, b, : pos + T])
                      for b in range(B)])
        h = h + o.reshape(B, T, a.q_dim) @ w[(l, "wo")].T
        y = rmsnorm(h, w[(l, "ffn_norm")], a.rms_eps)
        gu = y @ w[(l, "wgu")].T
        act = silu(gu[..., : a.ffn]) * gu[..., a.ffn:]
        return h + act @ w[(l, "wdown")].T

    def _forward(self, tokens):
        tokens = np.asarray(tokens, dtype=np.int64)
        assert tokens.shape[0] == self.B and self.length + tokens.shape[1] <= self.T
        h = self.w["embed"][tokens]
        hidden = []
        for l in range(self.a.n_layers):
            h = self._block(l, h, self.length)
            hidden.append(h)
        self.length += tokens.shape[1]
        last = rmsnorm(h[:, -1, :], self.w["final_norm"], self.a.rms_eps)
        logits = last @ self.w["lm_head"].T
        return {"logits": logits, "hidden": hidden, "tokens": argmax(logits)}

    def prefill(self, tokens):
        """tokens [B, S] from an empty cache -> logits of the last position."""
        self.length = 0
        return self._forward(tokens)

    def decode(self, tokens):
        """tokens [B] (the previous outputs) -> logits of the new position."""
        return self._forward(np.asarray(tokens).reshape(self.B, 1))


def argmax(logits):
    """Greedy choice per row; ties go to the lowest token id."""
    return np.argmax(logits, axis=-1).astype(np.int32)
