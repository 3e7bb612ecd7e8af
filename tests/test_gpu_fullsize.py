"""Parity at the full sizes of the workloads, in the launch configuration the
bench times.

* Llama-2-7B- and 13B-shaped fingerprints end to end: the handle is created
  exactly as ``bench.py`` creates it (device-side seeded weights, seed 0, unit
  norm gains, the full batch, prompt and context), prefills the full batch and
  decodes a few steps.  The oracle runs a batch-1 slice per checked sequence
  (sequences are independent) from its own seeded weights and tokens; every
  hidden row of that sequence after each block, its logits and its greedy
  ids are compared (tolerance and near-tie rule as in test_gpu_model).  The
  decode steps feed the oracle's token to the checked sequences and the
  device's own token to the others.
* Llama-2-70B-shaped: the kernels at the workload's full shapes, through the
  op entry points (same kernels and plans as the runtime): the four int4
  decode linears and the LM head at M = 32 on sampled output rows, the GQA
  int8-KV decode attention at B 32 and context 2148 on sampled (sequence,
  head) pairs, and the prefill gate+up GEMM at M = 65536 on sampled entries.
"""
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import quant
from tests.gpu_helpers import TAU, arch_dict, dev, empty, host, ptr, rel_err, torch_mod, weight_getter

pytestmark = pytest.mark.gpu

FULL = {
    # name: (arch, wquant, kvquant, batch, prompt, decode steps of the bench, checked sequences)
    "l7b": (M.Arch(2, 4096, 32, 32, 128, 11008, 32000), 1, 0, 8, 512, 100, [0, 7]),
    "l13b": (M.Arch(2, 5120, 40, 40, 128, 13824, 32000), 2, 0, 16, 1024, 100, [5]),
}
N_CHECKED_DECODE = 3


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


def _near_tie_ok(got, ref_logits, tau):
    ref = int(M.argmax(ref_logits[None])[0])
    if got == ref:
        return True
    top = np.sort(ref_logits)[-2:]
    return top[1] - top[0] < 2 * tau * np.max(np.abs(ref_logits))


@pytest.mark.parametrize("name", list(FULL))
def test_full_size_sequences_match_oracle(fp, name):
    arch, wq, kvq, B, S, N, seqs = FULL[name]
    tau = TAU[wq]
    T = S + N + 1  # the bench's context
    get = weight_getter(0, gains="ones")  # the bench's device-side init: seed 0, unit gains
    with ThreadPoolExecutor(max_workers=8) as pool:
        w, payload = M.build_weights(arch, wq, get, map_fn=pool.map)
    h = fp.fp_create(arch_dict(arch), wq, kvq, B, T, seed=0, flags=fp.FP_FLAG_KEEP_HIDDEN)
    try:
        # device-side seeded weights and quantisation equal the oracle's, bit for bit
        for l in range(arch.n_layers):
            for m, mname in enumerate(("wqkv", "wo", "wgu", "wdown")):
                p = payload[(l, mname)]
                cdt = np.int8 if wq == 1 else np.uint8
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_CODES, l, m, cdt), p["codes"].reshape(-1))
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_SCALES, l, m, np.uint16),
                                      p["scales"].reshape(-1))
                if wq == 2:
                    assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_ZEROS, l, m, np.uint16),
                                          p["zeros"].reshape(-1))
        toks = synth.tokens(0, B * S, arch.vocab).reshape(B, S)
        nxt = fp.fp_prefill(h, toks)
        hid = [quant.bf16_to_f32(fp.fp_get_tensor(h, fp.FP_G_HIDDEN, l, 0, np.uint16)).reshape(B, S, arch.hidden)
               for l in range(arch.n_layers)]
        lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(B, arch.vocab)
        refs = {b: M.Fingerprint(arch, w, kvq, 1, T) for b in seqs}
        cur = nxt.copy()
        for b in seqs:
            out = refs[b].prefill(toks[b:b + 1])
            for l in range(arch.n_layers):
                e = rel_err(hid[l][b], out["hidden"][l][0])
                assert e <= tau, (name, "prefill hidden", b, l, e)
            e = rel_err(lg[b], out["logits"][0])
            assert e <= tau, (name, "prefill logits", b, e)
            assert _near_tie_ok(int(nxt[b]), out["logits"][0], tau), (name, "prefill token", b)
            cur[b] = out["tokens"][0]
        for step in range(N_CHECKED_DECODE):
            got = fp.fp_decode_step(h, cur)
            hid = [quant.bf16_to_f32(fp.fp_get_tensor(h, fp.FP_G_HIDDEN, l, 0, np.uint16)).reshape(B, arch.hidden)
                   for l in range(arch.n_layers)]
            lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(B, arch.vocab)
            nxt_cur = got.copy()
            for b in seqs:
                out = refs[b].decode([cur[b]])
                for l in range(arch.n_layers):
                    e = rel_err(hid[l][b], out["hidden"][l][0])
                    assert e <= tau, (name, "decode hidden", step, b, l, e)
                e = rel_err(lg[b], out["logits"][0])
                assert e <= tau, (name, "decode logits", step, b, e)
                assert _near_tie_ok(int(got[b]), out["logits"][0], tau), (name, "decode token", step, b)
                nxt_cur[b] = out["tokens"][0]
            cur = nxt_cur
    finally:
        fp.fp_destroy(h)


# ---------------------------------------------------------------- 70B shapes, op level
A70 = M.Arch(2, 8192, 64, 8, 128, 28672, 32000)
SAMPLE_ROWS = 48


def _device_weights(fp, wq, stream, n, k):
    """Seeded bf16 [n, k] generated and quantised on the device (the runtime's path)."""
    torch = torch_mod()
    w = torch.empty(n * k, dtype=torch.int16, device="cuda")
    fp.fp_op_init_weights(w.data_ptr(), n * k, 0, stream, 0)
    codes = empty(n * k * 2 if wq == 0 else (n * k if wq == 1 else n * k // 2))
    scales = empty(n if wq != 2 else n * (k // 128), np.uint16)
    zeros = empty(max(1, n * (k // 128)), np.uint16)
    if wq == 0:
        codes = w
    else:
        fp.fp_op_quantize(wq, w.data_ptr(), n, k, ptr(codes), ptr(scales), ptr(zeros))
        del w
    return codes, scales, zeros


def _oracle_rows(wq, stream, rows, k):
    """Dequantised rows of the same seeded matrix, generated and quantised on the host."""
    bits = np.stack([synth.normal_bf16(0, stream, int(r) * k, k) for r in rows])
    return quant.quantize_weight(bits, wq)[1]


@pytest.mark.parametrize("mat", ["qkv", "o", "gu", "down", "lm_head"])
def test_full_size_70b_decode_linears(fp, mat):
    d, f = A70.hidden, A70.ffn
    nqkv = A70.q_dim + 2 * A70.kv_dim
    wq, epi, n, k = {"qkv": (2, 0, nqkv, d), "o": (2, 1, d, A70.q_dim), "gu": (2, 2, 2 * f, d),
                     "down": (2, 1, d, f), "lm_head": (0, 3, A70.vocab, d)}[mat]
    m = 32
    stream = 7000 + ["qkv", "o", "gu", "down", "lm_head"].index(mat)
    codes, scales, zeros = _device_weights(fp, wq, stream, n, k)
    x = synth.uniform_bf16(41, stream, (m, k), -2.0, 2.0)
    r = synth.uniform_bf16(42, stream, (m, d), -1.0, 1.0) if epi == 1 else None
    nout = n // 2 if epi == 2 else n
    out = empty(m * nout * (4 if epi == 3 else 2))
    wsb = fp.fp_op_linear_workspace_bytes(wq, m, n, k)
    ws = empty(max(wsb, 16))
    fp.fp_op_linear(wq, epi, ptr(dev(x)), m, n, k, ptr(codes), ptr(scales), ptr(zeros),
                    ptr(dev(r)) if r is not None else None, ptr(out), ptr(ws), wsb)
    got = host(out, np.float32 if epi == 3 else np.uint16)
    got = (got if epi == 3 else quant.bf16_to_f32(got)).reshape(m, nout).astype(np.float64)
    rows = np.unique(np.concatenate([[0, nout - 1], np.random.default_rng(stream).integers(0, nout, SAMPLE_ROWS)]))
    xf = quant.bf16_to_f32(x).astype(np.float64)
    if epi == 2:
        yg = xf @ _oracle_rows(wq, stream, rows, k).T
        yu = xf @ _oracle_rows(wq, stream, rows + nout, k).T
        ref = M.silu(yg) * yu
    else:
        ref = xf @ _oracle_rows(wq, stream, rows, k).T
        if epi == 1:
            ref = ref + quant.bf16_to_f32(r).astype(np.float64)[:, rows]
    assert rel_err(got[:, rows], ref) <= TAU[wq] / 4, (mat, rel_err(got[:, rows], ref))


def test_full_size_70b_decode_attention(fp):
    from tests.test_gpu_ops import Cache

    B, H, Hkv, hd, T = 32, A70.n_heads, A70.n_kv_heads, A70.head_dim, 2148
    lens = [T - (b % 3) for b in range(B)]  # ragged tails of the last page
    c = Cache(fp, 1, B, T, Hkv, hd, seed=70)
    q = synth.uniform_bf16(43, 1, (B, H * hd), -2, 2)
    out = empty(B * H * hd, np.uint16)
    wsb = fp.fp_op_attention_decode_workspace_bytes(B, H, hd, T)
    ws = empty(wsb)
    err = empty(1, np.int32)
    fp.fp_op_attention_decode(ptr(dev(q)), H * hd, B, H, c.view, ptr(dev(np.array(lens, np.int32))), T, ptr(out),
                              ptr(ws), wsb, ptr(err))
    got = quant.bf16_to_f32(host(out, np.uint16)).reshape(B, H, hd)
    qf = quant.bf16_to_f32(q).astype(np.float64).reshape(B, H, hd)
    for b in (0, 13, B - 1):
        ref = M.attention(qf[b][None], np.array([lens[b] - 1]), c.seq("k", b, lens[b]), c.seq("v", b, lens[b]))[0]
        assert rel_err(got[b], ref) <= TAU[0] / 2, (b, rel_err(got[b], ref))
    assert host(err, np.int32)[0] == 0


def test_full_size_70b_prefill_gate_up(fp):
    """The tcgen05 GEMM at the 70B-shaped prefill: M = 32 x 2048 rows, SwiGLU epilogue, int4 weights."""
    torch = torch_mod()
    m, n, k, wq = 32 * 2048, 2 * A70.ffn, A70.hidden, 2
    stream = 7100
    codes, scales, zeros = _device_weights(fp, wq, stream, n, k)
    x = torch.empty(m * k, dtype=torch.int16, device="cuda")
    fp.fp_op_init_weights(x.data_ptr(), m * k, 1, stream, 0)  # seeded bf16 activations of N(0, 0.02) shape
    nout = n // 2
    out = empty(m * nout * 2)
    wsb = fp.fp_op_linear_workspace_bytes(wq, m, n, k)
    ws = empty(max(wsb, 16))
    fp.fp_op_linear(wq, 2, x.data_ptr(), m, n, k, ptr(codes), ptr(scales), ptr(zeros), None, ptr(out), ptr(ws), wsb)
    torch.cuda.synchronize()
    rng = np.random.default_rng(stream)
    mrows = np.unique(np.concatenate([[0, m - 1], rng.integers(0, m, 16)]))
    ncols = np.unique(np.concatenate([[0, nout - 1], rng.integers(0, nout, 32)]))
    y = out.view(torch.int16).view(m, nout)
    got = quant.bf16_to_f32(y[torch.as_tensor(mrows, device="cuda")].cpu().numpy().view(np.uint16))[:, ncols]
    xf = quant.bf16_to_f32(np.stack([synth.normal_bf16(1, stream, int(r) * k, k) for r in mrows])).astype(np.float64)
    yg = xf @ _oracle_rows(wq, stream, ncols, k).T
    yu = xf @ _oracle_rows(wq, stream, ncols + nout, k).T
    ref = M.silu(yg) * yu
    assert rel_err(got, ref) <= TAU[wq] / 4, rel_err(got, ref)
