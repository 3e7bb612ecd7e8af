"""Kernel-level parity: each entry point of fp_ops.h against the oracle on the
same seeded inputs.  Codes, packing, ids and generated weights are compared
bit for bit; floating-point outputs within max|d| <= tau * max|ref|."""
import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import quant
from tests.gpu_helpers import TAU, dev, empty, host, ptr, rel_err, torch_mod

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


def _special_weights(n, k, seed):
    w = synth.weight_bf16(seed, 2, 1, (n, k))
    w[0] = 0
    w[1] = 0
    w[1, 3] = synth.f32_to_bf16_bits(np.array([0.75], np.float32))[0]
    w[2] = synth.f32_to_bf16_bits(np.array([-0.125], np.float32))[0]
    w[3] = synth.f32_to_bf16_bits(-np.abs(quant.bf16_to_f32(w[3])))
    return w


# ---------------------------------------------------------------- weights
@pytest.mark.parametrize("seed,stream,start,n", [(0, 17, 0, 1000), (7, 3, 123456789, 4099), (2 ** 63 + 5, 99, 5, 77)])
def test_device_generator_matches_host(fp, seed, stream, start, n):
    w = empty(n, np.uint16)
    fp.fp_op_init_weights(ptr(w), n, seed, stream, start)
    assert np.array_equal(host(w, np.uint16), synth.normal_bf16(seed, stream, start, n))


@pytest.mark.parametrize("wq,n,k", [(1, 37, 1376), (1, 256, 4096), (2, 37, 1408), (2, 130, 4096)])
def test_quantize_bit_exact(fp, wq, n, k):
    w = _special_weights(n, k, 5 + wq)
    codes = empty(n * k if wq == 1 else n * k // 2)
    scales = empty(n if wq == 1 else n * (k // 128), np.uint16)
    zeros = empty(n * (k // 128), np.uint16)
    fp.fp_op_quantize(wq, ptr(dev(w)), n, k, ptr(codes), ptr(scales), ptr(zeros))
    payload, _ = quant.quantize_weight(w, wq)
    if wq == 1:
        assert np.array_equal(host(codes, np.int8).reshape(n, k), payload["codes"])
        assert np.array_equal(host(scales, np.uint16), payload["scales"])
    else:
        assert np.array_equal(host(codes, np.uint8).reshape(n, k // 2), payload["codes"])
        assert np.array_equal(host(scales, np.uint16).reshape(n, -1), payload["scales"])
        assert np.array_equal(host(zeros, np.uint16).reshape(n, -1), payload["zeros"])


# ---------------------------------------------------------------- linear
def _quantized_on_device(fp, wq, w):
    n, k = w.shape
    if wq == 0:
        return dev(w), None, None
    codes = empty(n * k if wq == 1 else n * k // 2)
    scales = empty(n if wq == 1 else n * (k // 128), np.uint16)
    zeros = empty(max(1, n * (k // 128)), np.uint16)
    fp.fp_op_quantize(wq, ptr(dev(w)), n, k, ptr(codes), ptr(scales), ptr(zeros))
    return codes, scales, zeros


@pytest.mark.parametrize("wq", [0, 1, 2])
@pytest.mark.parametrize("m", [1, 3, 8, 13, 64, 130])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_linear_matches_oracle(fp, wq, m, epi):
    k, n = (384, 200) if wq != 2 else (512, 200)
    w = synth.weight_bf16(11 + wq, 0, 1, (n, k))
    x = synth.uniform_bf16(12, m, (m, k), -2.0, 2.0)
    r = synth.uniform_bf16(13, m, (m, n), -1.0, 1.0)
    codes, scales, zeros = _quantized_on_device(fp, wq, w)
    _, wd = quant.quantize_weight(w, wq)
    xf = quant.bf16_to_f32(x).astype(np.float64)
    yref = xf @ wd.T
    nout = n // 2 if epi == 2 else n
    out = empty(m * nout * (4 if epi == 3 else 2))
    rd = dev(r)
    ws_b = fp.fp_op_linear_workspace_bytes(wq, m, n, k)
    ws = empty(max(ws_b, 16))
    fp.fp_op_linear(wq, epi, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), ptr(rd), ptr(out),
                    ptr(ws), ws_b)
    if epi == 0:
        got, ref = host(out, np.uint16), yref
        got = quant.bf16_to_f32(got).reshape(m, n)
    elif epi == 1:
        got = quant.bf16_to_f32(host(out, np.uint16)).reshape(m, n)
        ref = quant.bf16_to_f32(r).astype(np.float64) + yref
    elif epi == 2:
        got = quant.bf16_to_f32(host(out, np.uint16)).reshape(m, nout)
        ref = M.silu(yref[:, :nout]) * yref[:, nout:]
    else:
        got = host(out, np.float32).reshape(m, n)
        ref = yref
    assert rel_err(got, ref) <= TAU[wq] / 4, (wq, m, epi, rel_err(got, ref))


@pytest.mark.parametrize("wq", [0, 1, 2])
@pytest.mark.parametrize("m,n,k", [(8, 272, 4096), (16, 200, 5120), (32, 136, 11008), (2, 4104, 1408)])
def test_linear_long_k(fp, wq, m, n, k):
    """Long K ranges per CTA (the weight pipeline wraps many times) and ragged row tiles."""
    w = synth.weight_bf16(31 + wq, 0, 1, (n, k))
    x = synth.uniform_bf16(32, m, (m, k), -2.0, 2.0)
    codes, scales, zeros = _quantized_on_device(fp, wq, w)
    _, wd = quant.quantize_weight(w, wq)
    ref = quant.bf16_to_f32(x).astype(np.float64) @ wd.T
    out = empty(m * n * 4)
    ws_b = fp.fp_op_linear_workspace_bytes(wq, m, n, k)
    ws = empty(max(ws_b, 16))
    fp.fp_op_linear(wq, 3, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), None, ptr(out), ptr(ws), ws_b)
    got = host(out, np.float32).reshape(m, n)
    assert rel_err(got, ref) <= TAU[wq] / 4, (wq, m, n, k, rel_err(got, ref))


@pytest.mark.parametrize("m,n,k,epi", [
    (9, 200, 1024, 3), (16, 384, 5120, 2), (17, 300, 4096, 1), (32, 1000, 8192, 0), (33, 256, 1152, 3),
    (48, 520, 2048, 2), (64, 136, 11008, 1), (32, 2048, 3584, 3), (16, 40960, 256, 0), (24, 40960, 256, 2),
    (17, 1152, 1152, 0)])
def test_linear_int4_tensor_core(fp, m, n, k, epi):
    """int4 weights at 9-64 tokens, each weight expanded to bf16((q - z) s),
    the prefill expansion, and accumulated in fp32: the tcgen05 decode path
    from 17 tokens on, the CUDA-core GEMV below.  Cases: ragged row tiles,
    tokens padded to 32 / 64, K / 128 = 8, 40, 32, 64, 9, 16, 86, 28, 2
    groups (scale loads of 8 / 4 / 2 / 1 groups), row tiles shared by
    several CTAs and CTAs covering whole tiles."""
    w = synth.weight_bf16(50 + m, 0, 1, (n, k))
    x = synth.uniform_bf16(51, m, (m, k), -2.0, 2.0)
    r = synth.uniform_bf16(52, m, (m, n), -1.0, 1.0)
    codes, scales, zeros = _quantized_on_device(fp, 2, w)
    _, wd = quant.quantize_weight(w, 2)
    # (q - z) s is exact in fp32 (at most 13 significant bits); one rounding to bf16
    wb = quant.bf16_to_f32(synth.f32_to_bf16_bits(wd.astype(np.float32))).astype(np.float64)
    xf = quant.bf16_to_f32(x).astype(np.float64)
    nout = n // 2 if epi == 2 else n
    out = empty(m * nout * (4 if epi == 3 else 2))
    ws_b = fp.fp_op_linear_workspace_bytes(2, m, n, k)
    ws = empty(max(ws_b, 16))
    fp.fp_op_linear(2, epi, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), ptr(dev(r)), ptr(out),
                    ptr(ws), ws_b)
    if epi == 3:
        got = host(out, np.float32).reshape(m, n).astype(np.float64)
    else:
        got = quant.bf16_to_f32(host(out, np.uint16)).reshape(m, nout).astype(np.float64)
    # the tensor-core path multiplies the bf16 expansion; the CUDA-core GEMV
    # removes the zero point in fp32 and so matches the exact dequantisation
    tight = wb if m >= 17 else wd
    for wm, tol in ((wd, TAU[2] / 4), (tight, 1e-4 if epi == 3 else 6e-3)):
        y = xf @ wm.T
        if epi == 1:
            y = quant.bf16_to_f32(r).astype(np.float64) + y
        elif epi == 2:
            y = M.silu(y[:, :nout]) * y[:, nout:]
        assert rel_err(got, y) <= tol, (m, n, k, epi, tol, rel_err(got, y))


@pytest.mark.parametrize("m,n,k,epi", [
    (17, 300, 4096, 1), (32, 1000, 8192, 0), (33, 256, 1152, 3), (48, 520, 2048, 2), (64, 136, 11008, 1),
    (32, 2048, 3584, 3), (17, 1152, 1152, 0), (64, 2000, 128, 2), (40, 16384, 256, 0), (20, 384, 1088, 0),
    (24, 256, 16384, 1), (32, 512, 16384, 2), (17, 300, 20480, 3)])
def test_linear_int8_tensor_core(fp, m, n, k, epi):
    """int8 per-channel weights at 17-64 tokens: beyond 32 tokens, or with K
    of 16384 or more, the codes widened exactly to bf16 in TMEM, products
    accumulated in fp32 on tcgen05, the row scale applied to the sums; else
    the mma.sync GEMV.  Cases: ragged row tiles, tokens padded to 32 / 64,
    SwiGLU items of 64 k (K 128: two per row), row tiles shared by several
    CTAs and CTAs covering whole tiles; K = 1088 (not a multiple of 128)
    always takes the mma.sync GEMV."""
    w = synth.weight_bf16(60 + m, 0, 1, (n, k))
    x = synth.uniform_bf16(61, m, (m, k), -2.0, 2.0)
    r = synth.uniform_bf16(62, m, (m, n), -1.0, 1.0)
    codes, scales, zeros = _quantized_on_device(fp, 1, w)
    _, wd = quant.quantize_weight(w, 1)
    xf = quant.bf16_to_f32(x).astype(np.float64)
    nout = n // 2 if epi == 2 else n
    out = empty(m * nout * (4 if epi == 3 else 2))
    ws_b = fp.fp_op_linear_workspace_bytes(1, m, n, k)
    ws = empty(max(ws_b, 16))
    fp.fp_op_linear(1, epi, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), ptr(dev(r)), ptr(out),
                    ptr(ws), ws_b)
    if epi == 3:
        got = host(out, np.float32).reshape(m, n).astype(np.float64)
    else:
        got = quant.bf16_to_f32(host(out, np.uint16)).reshape(m, nout).astype(np.float64)
    y = xf @ wd.T
    if epi == 1:
        y = quant.bf16_to_f32(r).astype(np.float64) + y
    elif epi == 2:
        y = M.silu(y[:, :nout]) * y[:, nout:]
    # the tensor-core path sees x and the codes exactly (the mma.sync GEMV
    # stages x in fp16): fp32 sums against the exact product
    tight = k % 128 == 0 and (m > 32 or k >= 16384)
    tol = (1e-4 if epi == 3 else 6e-3) if tight else TAU[1] / 4
    assert rel_err(got, y) <= tol, (m, n, k, epi, tol, rel_err(got, y))


def test_linear_residual_in_place(fp):
    m, n, k = 5, 64, 256
    w = synth.weight_bf16(3, 0, 1, (n, k))
    x = synth.uniform_bf16(4, 1, (m, k), -1, 1)
    r = synth.uniform_bf16(4, 2, (m, n), -1, 1)
    codes, scales, zeros = _quantized_on_device(fp, 1, w)
    buf = dev(r)
    wsb = fp.fp_op_linear_workspace_bytes(1, m, n, k)
    ws = empty(max(wsb, 16))
    fp.fp_op_linear(1, 1, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), ptr(buf), ptr(buf), ptr(ws), wsb)
    _, wd = quant.quantize_weight(w, 1)
    ref = quant.bf16_to_f32(r) + quant.bf16_to_f32(x).astype(np.float64) @ wd.T
    assert rel_err(quant.bf16_to_f32(host(buf, np.uint16)).reshape(m, n), ref) < 5e-3


# ---------------------------------------------------------------- rows
# rows from a ragged single warp's worth (d 40) to 40960 elements
@pytest.mark.parametrize("m,d,stride,offset", [(1, 512, 1, 0), (7, 4096, 1, 0), (3, 1024, 5, 4), (32, 8192, 1, 0),
                                              (2, 8200, 1, 0), (2, 24576, 2, 1), (3, 40, 1, 0), (1, 40960, 1, 0)])
def test_rmsnorm(fp, m, d, stride, offset):
    rows = m * stride
    x = synth.uniform_bf16(21, d, (rows, d), -3, 3)
    g = synth.uniform_bf16(22, d, (d,), 0.5, 1.5)
    y = empty(m * d, np.uint16)
    fp.fp_op_rmsnorm(ptr(dev(x)), m, d, stride, offset, ptr(dev(g)), 1e-5, ptr(y))
    xs = quant.bf16_to_f32(x).astype(np.float64)[offset::stride][:m]
    ref = M.rmsnorm(xs, quant.bf16_to_f32(g).astype(np.float64), 1e-5)
    assert rel_err(quant.bf16_to_f32(host(y, np.uint16)).reshape(m, d), ref) < 1e-2


def test_embed_and_bad_id(fp):
    V, d = 100, 64
    E = synth.weight_bf16(1, -1, 0, (V, d))
    tok = np.array([5, 0, 99, 100, -1, 7], np.int32)
    h = empty(len(tok) * d, np.uint16)
    err = empty(1, np.int32)
    fp.fp_op_embed(ptr(dev(tok)), len(tok), ptr(dev(E)), V, d, ptr(h), ptr(err))
    out = host(h, np.uint16).reshape(len(tok), d)
    for i, t in enumerate(tok):
        assert np.array_equal(out[i], E[t] if 0 <= t < V else np.zeros(d, np.uint16))
    assert host(err, np.int32)[0] == 1


@pytest.mark.parametrize("V", [32000, 17, 1000])
def test_argmax_ties_lowest(fp, V):
    rng = np.random.default_rng(V)
    x = rng.normal(size=(4, V)).astype(np.float32)
    x[1, :] = 1.0
    x[2, [V // 3, V // 2, V - 1]] = 50.0
    x[3, V - 1] = 60.0
    out = empty(4, np.int32)
    fp.fp_op_argmax(ptr(dev(x)), 4, V, ptr(out))
    assert host(out, np.int32).tolist() == M.argmax(x.astype(np.float64)).tolist()


# ---------------------------------------------------------------- KV cache
class Cache:
    """A paged cache built on the host (values chosen by the test), uploaded."""

    def __init__(self, fp, kvq, B, T, Hkv, hd, seed, shuffle=True, vs_range=(0.001, 0.03)):
        self.P, self.pps = 16, (T + 15) // 16
        self.n_pages = B * self.pps
        rng = np.random.default_rng(seed)
        perm = rng.permutation(self.n_pages) if shuffle else np.arange(self.n_pages)
        self.table = perm.reshape(B, self.pps).astype(np.int32)
        shape = (self.n_pages, Hkv, self.P, hd)
        self.kvq, self.B, self.Hkv, self.hd = kvq, B, Hkv, hd
        if kvq == 0:
            self.k = synth.uniform_bf16(seed, 1, shape, -2, 2)
            self.v = synth.uniform_bf16(seed, 2, shape, -2, 2)
            self.kd, self.vd = dev(self.k), dev(self.v)
            self.ks = self.vs = None
        else:
            self.k = rng.integers(-127, 128, size=shape, dtype=np.int8)
            self.v = rng.integers(-127, 128, size=shape, dtype=np.int8)
            self.ksc = synth.uniform_f32(seed, 3, shape[:3], 0.001, 0.03)
            self.vsc = synth.uniform_f32(seed, 4, shape[:3], *vs_range)
            self.kd, self.vd = dev(self.k), dev(self.v)
            self.ks, self.vs = dev(self.ksc), dev(self.vsc)
        self.td = dev(self.table)
        self.view = fp.fp_kv_view(kvq, Hkv, hd, self.P, self.pps, self.n_pages, ptr(self.kd), ptr(self.vd),
                                  ptr(self.ks), ptr(self.vs), ptr(self.td))

    def seq(self, which, b, T):
        """Dequantised K or V of sequence b, positions 0..T-1: [T, Hkv, hd] fp64."""
        pages = self.table[b, np.arange(T) // 16]
        slot = np.arange(T) % 16
        if self.kvq == 0:
            src = self.k if which == "k" else self.v
            return quant.bf16_to_f32(src[pages, :, slot]).astype(np.float64)
        codes = (self.k if which == "k" else self.v)[pages, :, slot].astype(np.float64)
        sc = (self.ksc if which == "k" else self.vsc)[pages, :, slot].astype(np.float64)
        return codes * sc[..., None]


@pytest.mark.parametrize("kvq", [0, 1])
@pytest.mark.parametrize("hd,H,Hkv", [(64, 8, 8), (128, 8, 1), (128, 64, 8), (128, 4, 2), (128, 16, 4)])
@pytest.mark.parametrize("lens", [[1], [17, 300, 16], [1037, 5], [4000, 63, 2500]])
def test_attention_decode(fp, kvq, hd, H, Hkv, lens):
    B, T = len(lens), max(lens) + 3
    c = Cache(fp, kvq, B, T, Hkv, hd, seed=hd + H + kvq)
    q = synth.uniform_bf16(31, B, (B, H * hd), -2, 2)
    out = empty(B * H * hd, np.uint16)
    wsb = fp.fp_op_attention_decode_workspace_bytes(B, H, hd, T)
    ws = empty(wsb)
    err = empty(1, np.int32)
    fp.fp_op_attention_decode(ptr(dev(q)), H * hd, B, H, c.view, ptr(dev(np.array(lens, np.int32))), T, ptr(out),
                              ptr(ws), wsb, ptr(err))
    got = quant.bf16_to_f32(host(out, np.uint16)).reshape(B, H, hd)
    qf = quant.bf16_to_f32(q).astype(np.float64).reshape(B, H, hd)
    for b, L in enumerate(lens):
        ref = M.attention(qf[b][None], np.array([L - 1]), c.seq("k", b, L), c.seq("v", b, L))[0]
        assert rel_err(got[b], ref) <= TAU[0] / 2, (b, rel_err(got[b], ref))
    assert host(err, np.int32)[0] == 0


@pytest.mark.parametrize("kvq", [0, 1])
@pytest.mark.parametrize("hd,H,Hkv", [(64, 4, 4), (128, 8, 2)])
@pytest.mark.parametrize("S", [1, 17, 64, 130, 513])
def test_attention_prefill(fp, kvq, hd, H, Hkv, S):
    B = 2
    c = Cache(fp, kvq, B, S + 5, Hkv, hd, seed=S + hd + kvq)
    q = synth.uniform_bf16(41, S, (B * S, H * hd), -2, 2)
    out = empty(B * S * H * hd, np.uint16)
    fp.fp_op_attention_prefill(ptr(dev(q)), H * hd, B, S, H, c.view, ptr(out))
    got = quant.bf16_to_f32(host(out, np.uint16)).reshape(B, S, H, hd)
    qf = quant.bf16_to_f32(q).astype(np.float64).reshape(B, S, H, hd)
    for b in range(B):
        ref = M.attention(qf[b], np.arange(S), c.seq("k", b, S), c.seq("v", b, S))
        assert rel_err(got[b], ref) <= TAU[0] / 2, (b, rel_err(got[b], ref))


@pytest.mark.parametrize("vs_range", [(1e-7, 3e-7), (1e-3, 3e-2), (50.0, 400.0)])
def test_attention_prefill_int8_value_scales(fp, vs_range):
    """int8 cache, tcgen05 kernel (head_dim 128): P runs as fp16 carrying
    each key's V scale times a per-CTA power of two; values far below and far
    above the usual range of V must come out as accurately."""
    B, S, H, Hkv, hd = 2, 300, 8, 2, 128
    c = Cache(fp, 1, B, S + 5, Hkv, hd, seed=91, vs_range=vs_range)
    q = synth.uniform_bf16(42, S, (B * S, H * hd), -2, 2)
    out = empty(B * S * H * hd, np.uint16)
    err = empty(1, np.int32)
    fp.fp_op_attention_prefill(ptr(dev(q)), H * hd, B, S, H, c.view, ptr(out), ptr(err))
    got = quant.bf16_to_f32(host(out, np.uint16)).reshape(B, S, H, hd)
    qf = quant.bf16_to_f32(q).astype(np.float64).reshape(B, S, H, hd)
    for b in range(B):
        ref = M.attention(qf[b], np.arange(S), c.seq("k", b, S), c.seq("v", b, S))
        assert rel_err(got[b], ref) <= TAU[0] / 2, (b, rel_err(got[b], ref))
    assert host(err, np.int32)[0] == 0


def test_attention_prefill_int8_q_beyond_fp16_is_reported(fp):
    """The int8-cache tcgen05 kernel multiplies Q in fp16: a query element
    beyond 65504 sets the error word to 3 (the runtime reports it)."""
    B, S, H, Hkv, hd = 1, 64, 4, 2, 128
    c = Cache(fp, 1, B, S, Hkv, hd, seed=92)
    q = synth.uniform_bf16(43, S, (B * S, H * hd), -2, 2)
    q[3, 17] = synth.f32_to_bf16_bits(np.array([1.0e5], np.float32))[0]
    out = empty(B * S * H * hd, np.uint16)
    err = empty(1, np.int32)
    fp.fp_op_attention_prefill(ptr(dev(q)), H * hd, B, S, H, c.view, ptr(out), ptr(err))
    assert host(err, np.int32)[0] == 3


@pytest.mark.parametrize("kvq", [0, 1])
@pytest.mark.parametrize("hd,H,Hkv", [(64, 4, 4), (128, 8, 2)])
def test_attention_bad_page_reads_zeros(fp, kvq, hd, H, Hkv):
    """A page id outside [0, n_pages) reads as zero keys and values (zero
    codes and scales for int8) and sets the error word to 1, in prefill and
    in decode; the other pages are unaffected."""
    B, S = 2, 200
    c = Cache(fp, kvq, B, S + 5, Hkv, hd, seed=77 + hd + kvq)
    bad = {(0, 5): c.n_pages, (1, 9): -3}  # positions 80-95 of sequence 0, 144-159 of sequence 1
    table = c.table.copy()
    for (b, pg), v in bad.items():
        table[b, pg] = v
    td = dev(table)
    view = fp.fp_kv_view(kvq, Hkv, hd, c.P, c.pps, c.n_pages, ptr(c.kd), ptr(c.vd), ptr(c.ks), ptr(c.vs), ptr(td))

    def seq(which, b, T):
        x = c.seq(which, b, T)
        for (bb, pg) in bad:
            if bb == b:
                x[pg * 16:(pg + 1) * 16] = 0.0
        return x

    q = synth.uniform_bf16(43, hd, (B * S, H * hd), -2, 2)
    qf = quant.bf16_to_f32(q).astype(np.float64).reshape(B, S, H, hd)
    out = empty(B * S * H * hd, np.uint16)
    err = empty(1, np.int32)
    fp.fp_op_attention_prefill(ptr(dev(q)), H * hd, B, S, H, view, ptr(out), ptr(err))
    got = quant.bf16_to_f32(host(out, np.uint16)).reshape(B, S, H, hd)
    for b in range(B):
        ref = M.attention(qf[b], np.arange(S), seq("k", b, S), seq("v", b, S))
        assert rel_err(got[b], ref) <= TAU[0] / 2, ("prefill", b, rel_err(got[b], ref))
    assert host(err, np.int32)[0] == 1

    lens = [S, 150]
    qd = synth.uniform_bf16(44, hd, (B, H * hd), -2, 2)
    wsb = fp.fp_op_attention_decode_workspace_bytes(B, H, hd, S + 5)
    ws = empty(wsb)
    out = empty(B * H * hd, np.uint16)
    err = empty(1, np.int32)
    fp.fp_op_attention_decode(ptr(dev(qd)), H * hd, B, H, view, ptr(dev(np.array(lens, np.int32))), S + 5, ptr(out),
                              ptr(ws), wsb, ptr(err))
    got = quant.bf16_to_f32(host(out, np.uint16)).reshape(B, H, hd)
    qf = quant.bf16_to_f32(qd).astype(np.float64).reshape(B, H, hd)
    for b, L in enumerate(lens):
        ref = M.attention(qf[b][None], np.array([L - 1]), seq("k", b, L), seq("v", b, L))[0]
        assert rel_err(got[b], ref) <= TAU[0] / 2, ("decode", b, rel_err(got[b], ref))
    assert host(err, np.int32)[0] == 1


@pytest.mark.parametrize("kvq", [0, 1])
@pytest.mark.parametrize("hd", [64, 128])
def test_rope_kv_write(fp, kvq, hd):
    B, S, H, Hkv, T = 3, 5, 4, 2, 48
    c = Cache(fp, kvq, B, T, Hkv, hd, seed=7)
    base = 10000.0
    cs = empty(T * hd, np.float32)
    fp.fp_op_rope_table(T, hd, base, ptr(cs))
    row = (H + 2 * Hkv) * hd
    qkv = synth.uniform_bf16(51, hd, (B * S, row), -3, 3)
    pos = np.array([0, 9, 30], np.int32)
    qd = dev(qkv)
    err = empty(1, np.int32)
    fp.fp_op_rope_kv(ptr(qd), B, S, row, H, c.view, ptr(dev(pos)), ptr(cs), ptr(err))
    q_out = quant.bf16_to_f32(host(qd, np.uint16)).reshape(B, S, -1)
    x = quant.bf16_to_f32(qkv).astype(np.float64).reshape(B, S, H + 2 * Hkv, hd)
    kd = host(c.kd, np.int8 if kvq else np.uint16)
    vd = host(c.vd, np.int8 if kvq else np.uint16)
    for b in range(B):
        p = pos[b] + np.arange(S)
        qref = M.rope(x[b, :, :H][None], p, base)[0]
        assert rel_err(q_out[b, :, : H * hd].reshape(S, H, hd), qref) < 1e-2
        kref = M.rope(x[b, :, H:H + Hkv][None], p, base)[0]
        vref = x[b, :, H + Hkv:]
        pages, slot = c.table[b, p // 16], p % 16
        if kvq == 0:
            kg = quant.bf16_to_f32(kd.reshape(c.n_pages, Hkv, 16, hd)[pages, :, slot]).astype(np.float64)
            vg = quant.bf16_to_f32(vd.reshape(c.n_pages, Hkv, 16, hd)[pages, :, slot]).astype(np.float64)
            assert rel_err(kg, kref) < 1e-2 and np.array_equal(vg, vref)
        else:
            ks = host(c.ks, np.float32).reshape(c.n_pages, Hkv, 16)[pages, :, slot]
            vs = host(c.vs, np.float32).reshape(c.n_pages, Hkv, 16)[pages, :, slot]
            kg = kd.reshape(c.n_pages, Hkv, 16, hd)[pages, :, slot]
            vg = vd.reshape(c.n_pages, Hkv, 16, hd)[pages, :, slot]
            # values: bit-exact codes (V has no rotation; K at position 0 is unrotated)
            vq, vsr = quant.quantize_kv_int8(qkv.reshape(B, S, H + 2 * Hkv, hd)[b, :, H + Hkv:])
            assert np.array_equal(vg, vq) and np.array_equal(vs, vsr)
            if pos[b] == 0:
                kq, ksr = quant.quantize_kv_int8(qkv.reshape(B, S, H + 2 * Hkv, hd)[b, 0:1, H:H + Hkv])
                assert np.array_equal(kg[0:1], kq) and np.array_equal(ks[0:1], ksr)
            assert rel_err(kg * ks[..., None].astype(np.float64), kref) < 1.5e-2
    assert host(err, np.int32)[0] == 0


def test_linear_workspace_shared_by_different_shapes(fp):
    """One workspace serves consecutive launches of different shapes: the
    split-K tickets left by one launch must not disturb the next."""
    shapes = [(1, 8, 256, 4096), (1, 8, 12800, 512), (0, 1, 32000, 512), (2, 16, 2048, 1024)]
    need = max(fp.fp_op_linear_workspace_bytes(wq, m, n, k) for wq, m, n, k in shapes)
    ws = empty(need)
    for rep in range(2):
        for i, (wq, m, n, k) in enumerate(shapes):
            w = synth.weight_bf16(40 + i, 0, 1, (n, k))
            x = synth.uniform_bf16(41 + i, m, (m, k), -2, 2)
            codes, scales, zeros = _quantized_on_device(fp, wq, w)
            out = empty(m * n * 4)
            fp.fp_op_linear(wq, 3, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), None, ptr(out),
                            ptr(ws), need)
            _, wd = quant.quantize_weight(w, wq)
            ref = quant.bf16_to_f32(x).astype(np.float64) @ wd.T
            assert rel_err(host(out, np.float32).reshape(m, n), ref) <= TAU[wq] / 4, (rep, i)


@pytest.mark.parametrize("wq,scratch", [(0, True), (1, True), (2, True), (1, False), (2, False)])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
@pytest.mark.parametrize("m,n,k", [(65, 520, 1408), (300, 1024, 4096), (1000, 2304, 1024), (257, 392, 1040)])
def test_prefill_gemm_matches_oracle(fp, wq, scratch, epi, m, n, k):
    """Rows > 64 run on the tcgen05 GEMMs: ragged M and N tiles, K tails
    (K 1040: a partial last 64-k stage for bf16 and int8; int4 needs whole
    128-groups).  int8 / int4 weights are expanded to bf16 in the workspace
    when it has room (scratch), else dequantised inside the GEMM (no
    workspace at all)."""
    if wq == 2 and k % 128:
        pytest.skip("int4 group-128 weights need K % 128 == 0")
    w = synth.weight_bf16(60 + wq, 0, 1, (n, k))
    x = synth.uniform_bf16(61, m, (m, k), -2.0, 2.0)
    r = synth.uniform_bf16(62, m, (m, n), -1.0, 1.0)
    codes, scales, zeros = _quantized_on_device(fp, wq, w)
    _, wd = quant.quantize_weight(w, wq)
    yref = quant.bf16_to_f32(x).astype(np.float64) @ wd.T
    nout = n // 2 if epi == 2 else n
    out = empty(m * nout * (4 if epi == 3 else 2))
    rd = dev(r[:, :nout].copy())
    wsb = fp.fp_op_linear_workspace_bytes(wq, m, n, k) if scratch else 0
    ws = empty(max(wsb, 16))
    fp.fp_op_linear(wq, epi, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), ptr(rd), ptr(out),
                    ptr(ws) if scratch else None, wsb)
    if epi == 3:
        got = host(out, np.float32).reshape(m, n)
        ref = yref
    else:
        got = quant.bf16_to_f32(host(out, np.uint16)).reshape(m, nout)
        if epi == 0:
            ref = yref
        elif epi == 1:
            ref = quant.bf16_to_f32(r[:, :nout]).astype(np.float64) + yref
        else:
            ref = M.silu(yref[:, :nout]) * yref[:, nout:]
    assert rel_err(got, ref) <= TAU[wq] / 4, (wq, epi, m, n, k, rel_err(got, ref))


@pytest.mark.parametrize("scratch", [True, False])
@pytest.mark.parametrize("wq,m,n,k,epi", [(1, 200, 2 * 9000, 8192, 2), (2, 136, 20000, 4096, 1), (1, 130, 17000, 4096, 3)])
def test_prefill_linear_in_bands_of_columns(fp, scratch, wq, m, n, k, epi):
    """Quantised prefill weights are expanded to bf16 band by band of output
    columns (the scratch holds at most 128 MB): matrices larger than that run
    as several expansions and GEMM launches into slices of the output.  Cases:
    int8 SwiGLU (up rows' scales taken at an offset, 3 bands of 4096 + 808
    columns), int4 with residual (2 bands), int8 fp32 out (2 bands).  Without
    a workspace the same matrices run on the GEMM that dequantises inside the
    kernel, in one launch."""
    w = synth.weight_bf16(70 + wq, 0, 1, (n, k))
    x = synth.uniform_bf16(71, m, (m, k), -2.0, 2.0)
    nout = n // 2 if epi == 2 else n
    r = synth.uniform_bf16(72, m, (m, nout), -1.0, 1.0)
    codes, scales, zeros = _quantized_on_device(fp, wq, w)
    _, wd = quant.quantize_weight(w, wq)
    assert fp.fp_op_linear_workspace_bytes(wq, m, n, k) <= (128 << 20) + (1 << 20)
    out = empty(m * nout * (4 if epi == 3 else 2))
    ws_b = fp.fp_op_linear_workspace_bytes(wq, m, n, k) if scratch else 0
    ws = empty(max(ws_b, 16))
    fp.fp_op_linear(wq, epi, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros), ptr(dev(r)), ptr(out),
                    ptr(ws) if scratch else None, ws_b)
    got = host(out, np.float32) if epi == 3 else quant.bf16_to_f32(host(out, np.uint16))
    got = got.reshape(m, nout).astype(np.float64)
    y = quant.bf16_to_f32(x).astype(np.float64) @ wd.T
    if epi == 1:
        y = quant.bf16_to_f32(r).astype(np.float64) + y
    elif epi == 2:
        y = M.silu(y[:, :nout]) * y[:, nout:]
    assert rel_err(got, y) <= TAU[wq] / 4, rel_err(got, y)


@pytest.mark.parametrize("m", [17, 32, 33, 64])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
def test_linear_bf16_tensor_core(fp, m, epi):
    """bf16 weights at 17-64 tokens with enough work per SM run on the
    TMA-fed tcgen05 GEMV (the LM head's kernel): ragged last row tile (N not a
    multiple of 128) and a K tail (half of the last 128-k item past K); output
    columns checked on a sample, the first and the last included."""
    n, k = (2 * 16424, 4160) if epi == 2 else (16424, 8256)
    w = synth.weight_bf16(51, 0, 1, (n, k))
    x = synth.uniform_bf16(52, m, (m, k), -2.0, 2.0)
    nout = n // 2 if epi == 2 else n
    r = synth.uniform_bf16(53, m, (m, nout), -1.0, 1.0)
    out = empty(m * nout * (4 if epi == 3 else 2))
    ws_b = fp.fp_op_linear_workspace_bytes(0, m, n, k)
    ws = empty(max(ws_b, 16))
    fp.fp_op_linear(0, epi, ptr(dev(x)), m, n, k, ptr(dev(w)), None, None, ptr(dev(r)), ptr(out), ptr(ws), ws_b)
    got = host(out, np.float32) if epi == 3 else quant.bf16_to_f32(host(out, np.uint16))
    got = got.reshape(m, nout).astype(np.float64)
    cols = np.unique(np.concatenate([[0, nout - 1], np.random.default_rng(m + epi).integers(0, nout, 96)]))
    xf = quant.bf16_to_f32(x).astype(np.float64)
    wf = lambda rows: quant.bf16_to_f32(w[rows]).astype(np.float64)
    if epi == 2:
        ref = M.silu(xf @ wf(cols).T) * (xf @ wf(cols + nout).T)
    else:
        ref = xf @ wf(cols).T
        if epi == 1:
            ref = ref + quant.bf16_to_f32(r).astype(np.float64)[:, cols]
    assert rel_err(got[:, cols], ref) <= TAU[0] / 4, (m, epi, rel_err(got[:, cols], ref))
