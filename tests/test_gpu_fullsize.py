"""Parity at the full sizes of the workloads, in the launch configuration the
bench times.

* Llama-2-7B-, 13B- and 70B-shaped fingerprints end to end (the 70B shape:
  int4 g128 weights, int8 KV cache, GQA 64/8, batch 32, 2048-token prompts,
  the bench's default workload; and the same with GPTQ4 weights): the handle is created
  exactly as ``bench.py`` creates it (device-side seeded weights, seed 0, unit
  norm gains, the full batch, prompt and context), prefills the full batch and
  decodes a few steps.  The oracle runs a batch-1 slice per checked sequence
  (sequences are independent) from its own seeded weights and tokens; every
  hidden row of that sequence after each block, its logits and its greedy
  ids are compared (tolerance and near-tie rule as in test_gpu_model).  The
  decode steps feed the oracle's token to the checked sequences and the
  device's own token to the others.
* Llama-2-70B-shaped, op level as well: the kernels at the workload's full shapes, through the
  op entry points (same kernels and plans as the runtime): the four int4
  decode linears and the LM head at M = 32 on sampled output rows, the GQA
  int8-KV decode attention at B 32 and context 2148 on sampled (sequence,
  head) pairs, and the prefill gate+up GEMM at M = 65536 on sampled entries
  (both prefill paths: bf16 expansion and in-kernel dequantisation).
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
    # the first and the last sequence: rows at both ends of M = 65536 in prefill
    "l70b": (M.Arch(2, 8192, 64, 8, 128, 28672, 32000), 2, 1, 32, 2048, 100, [0, 31]),
    # the same with GPTQ4 weights (act orders drawn from the seed by fp_create)
    "l70b_gptq4": (M.Arch(2, 8192, 64, 8, 128, 28672, 32000), 3, 1, 32, 2048, 100, [0, 31]),
}
N_CHECKED_DECODE = 3


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


# int8 KV cache, end to end: the device and the oracle each quantise K and V
# per (token, head) from bf16 values that differ by one rounding, which flips
# codes by one step (about one in six); the 70B-shaped synthetic attention is
# sharp (scores with a standard deviation of about 3), and two blocks amplify
# the flips and the bf16 storage of activations to about 5 % of the logits'
# range (measured: 4.7 % and 5.1 % on the first and last sequence, while each
# block alone with the oracle's codes stays at about 1 %:
# test_full_size_70b_blocks_with_the_oracles_kv_codes).  End-to-end
# comparisons with an int8 cache are held to 1e-1; the kernels' own error is
# held to 2e-2 by that test.
TAU_E2E_KV8 = 1e-1


def _near_tie_ok(got, ref_logits, dev_logits):
    """A greedy id may differ from the oracle's only where the measured logit
    error could reorder the oracle's top two (their gap below twice the
    largest |device - oracle| logit difference of that row)."""
    ref = int(M.argmax(ref_logits[None])[0])
    if got == ref:
        return True
    top = np.sort(ref_logits)[-2:]
    return top[1] - top[0] < 2 * np.max(np.abs(np.asarray(dev_logits, np.float64) - ref_logits))


@pytest.mark.parametrize("name", list(FULL))
def test_full_size_sequences_match_oracle(fp, name):
    arch, wq, kvq, B, S, N, seqs = FULL[name]
    tau = TAU_E2E_KV8 if kvq == 1 else TAU[wq]
    T = S + N + 1  # the bench's context
    get = weight_getter(0, gains="ones")  # the bench's device-side init: seed 0, unit gains
    with ThreadPoolExecutor(max_workers=8) as pool:
        w, payload = M.build_weights(arch, wq, get, map_fn=pool.map,
                                     act_order=lambda l, m, k: synth.act_order(0, l, m, k))
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
                if wq in (2, 3):
                    assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_ZEROS, l, m, np.uint16),
                                          p["zeros"].reshape(-1))
                if wq == 3:
                    assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_PERM, l, m, np.int32), p["perm"])
        toks = synth.tokens(0, B * S, arch.vocab).reshape(B, S)
        nxt = fp.fp_prefill(h, toks)
        d = arch.hidden

        def seq_hidden(l, b, rows):
            """Block l's output rows of sequence b (rows per sequence), read alone."""
            bits = fp.fp_get_tensor(h, fp.FP_G_HIDDEN, l, 0, np.uint16, count=rows * d, offset=b * rows * d)
            return quant.bf16_to_f32(bits).reshape(rows, d)

        lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(B, arch.vocab)
        refs = {b: M.Fingerprint(arch, w, kvq, 1, T) for b in seqs}
        cur = nxt.copy()
        for b in seqs:
            out = refs[b].prefill(toks[b:b + 1])
            for l in range(arch.n_layers):
                e = rel_err(seq_hidden(l, b, S), out["hidden"][l][0])
                assert e <= tau, (name, "prefill hidden", b, l, e)
            e = rel_err(lg[b], out["logits"][0])
            assert e <= tau, (name, "prefill logits", b, e)
            assert _near_tie_ok(int(nxt[b]), out["logits"][0], lg[b]), (name, "prefill token", b)
            cur[b] = out["tokens"][0]
        for step in range(N_CHECKED_DECODE):
            got = fp.fp_decode_step(h, cur)
            lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(B, arch.vocab)
            nxt_cur = got.copy()
            for b in seqs:
                out = refs[b].decode([cur[b]])
                for l in range(arch.n_layers):
                    e = rel_err(seq_hidden(l, b, 1)[0], out["hidden"][l][0])
                    assert e <= tau, (name, "decode hidden", step, b, l, e)
                e = rel_err(lg[b], out["logits"][0])
                assert e <= tau, (name, "decode logits", step, b, e)
                assert _near_tie_ok(int(got[b]), out["logits"][0], lg[b]), (name, "decode token", step, b)
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


@pytest.mark.parametrize("scratch", [True, False])
def test_full_size_70b_prefill_gate_up(fp, scratch):
    """The tcgen05 GEMM at the 70B-shaped prefill: M = 32 x 2048 rows, SwiGLU
    epilogue, int4 weights -- expanded to bf16 in the workspace, or, with no
    workspace, dequantised inside the GEMM."""
    torch = torch_mod()
    m, n, k, wq = 32 * 2048, 2 * A70.ffn, A70.hidden, 2
    stream = 7100
    codes, scales, zeros = _device_weights(fp, wq, stream, n, k)
    x = torch.empty(m * k, dtype=torch.int16, device="cuda")
    fp.fp_op_init_weights(x.data_ptr(), m * k, 1, stream, 0)  # seeded bf16 activations of N(0, 0.02) shape
    nout = n // 2
    out = empty(m * nout * 2)
    wsb = fp.fp_op_linear_workspace_bytes(wq, m, n, k) if scratch else 0
    ws = empty(max(wsb, 16))
    fp.fp_op_linear(wq, 2, x.data_ptr(), m, n, k, ptr(codes), ptr(scales), ptr(zeros), None, ptr(out),
                    ptr(ws) if scratch else None, wsb)
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


def test_full_size_70b_blocks_with_the_oracles_kv_codes(fp):
    """The kernels of the 70B-shaped workload, block by block, with the int8
    KV reading taken out: one 2048-token sequence through the op entry points
    (RMSNorm, the int4 prefill GEMMs, RoPE + int8 KV append, tcgen05 prefill
    attention over the int8 cache, SwiGLU, residual adds, final norm, LM head)
    where each block starts from the oracle's own input to that block and its
    cache holds the oracle's K/V codes and scales, written over the ones the
    device quantised.  Two independent int8 quantisations of K and V from bf16
    values that differ by one rounding flip codes by one step, and sharp
    attention amplifies that through the blocks (the end-to-end comparison
    above); with the codes shared, what remains is the kernels' own error
    (bf16 storage of activations, fp32 accumulation), held to 2e-2."""
    torch = torch_mod()
    a = A70
    S, d, f, H, Hkv, hd = 2048, a.hidden, a.ffn, a.n_heads, a.n_kv_heads, a.head_dim
    nqkv = a.q_dim + 2 * a.kv_dim
    get = weight_getter(0, gains="ones")
    with ThreadPoolExecutor(max_workers=8) as pool:
        w, payload = M.build_weights(a, 2, get, map_fn=pool.map)
    toks = synth.tokens(0, S, a.vocab).reshape(1, S)
    # device weights: the oracle's codes, scales and zeros of every block matrix
    mats = {}
    for l in range(a.n_layers):
        for name in ("wqkv", "wo", "wgu", "wdown"):
            p = payload[(l, name)]
            mats[(l, name)] = (dev(p["codes"]), dev(p["scales"]), dev(p["zeros"]))
    ones = dev(synth.f32_to_bf16_bits(np.ones(d, np.float32)))
    head = dev(get(-1, 2, (a.vocab, d)))
    # a batch-1 paged int8 cache with the identity page table
    pps = S // 16
    kpool, vpool = empty(pps * Hkv * 16 * hd), empty(pps * Hkv * 16 * hd)
    ksc, vsc = empty(pps * Hkv * 16, np.float32), empty(pps * Hkv * 16, np.float32)
    table = dev(np.arange(pps, dtype=np.int32).reshape(1, pps))
    kv = fp.fp_kv_view(1, Hkv, hd, 16, pps, pps, ptr(kpool), ptr(vpool), ptr(ksc), ptr(vsc), ptr(table))
    cs = empty(pps * 16 * hd // 2 * 2, np.float32)
    fp.fp_op_rope_table(pps * 16, hd, a.rope_base, ptr(cs))
    pos = dev(np.zeros(1, np.int32))
    err = empty(1, np.int32)
    y, qkv = empty(S * d * 2), empty(S * nqkv * 2)
    att, act = empty(S * a.q_dim * 2), empty(S * f * 2)
    wsb = max(fp.fp_op_linear_workspace_bytes(2, S, n, k) for n, k in ((nqkv, d), (d, a.q_dim), (2 * f, d), (d, f)))
    ws = empty(wsb)

    def lin(epi, x, name, l, n, k, out, resid=None):
        c, sc, z = mats[(l, name)]
        fp.fp_op_linear(2, epi, ptr(x), S, n, k, ptr(c), ptr(sc), ptr(z), ptr(resid), ptr(out), ptr(ws), wsb)

    h_in = w["embed"][toks]  # [1, S, d], exact bf16 values
    for l in range(a.n_layers):
        # the oracle's block l from h_in, recording the K and V it stores
        seen = []
        orig = M.store_kv
        M.store_kv = lambda x, kvq: (seen.append(x), orig(x, kvq))[1]
        try:
            ref_out = M.Fingerprint(a, w, 1, 1, S)._block(l, h_in, 0)[0]
        finally:
            M.store_kv = orig
        kc, ks = quant.quantize_kv_int8(quant.f32_to_bf16_rne(seen[0][0].astype(np.float32)))  # [S, Hkv, hd]
        vc, vs = quant.quantize_kv_int8(quant.f32_to_bf16_rne(seen[1][0].astype(np.float32)))
        # the device's block l from the same input
        h = dev(synth.f32_to_bf16_bits(h_in[0].astype(np.float32)))
        fp.fp_op_rmsnorm(ptr(h), S, d, 1, 0, ptr(ones), a.rms_eps, ptr(y))
        lin(0, y, "wqkv", l, nqkv, d, qkv)
        fp.fp_op_rope_kv(ptr(qkv), 1, S, nqkv, H, kv, ptr(pos), ptr(cs), ptr(err))
        torch.cuda.synchronize()
        page = lambda x: np.ascontiguousarray(x.reshape(pps, 16, Hkv, *x.shape[2:]).swapaxes(1, 2))
        kpool.copy_(torch.from_numpy(page(kc).reshape(-1).view(np.uint8)))
        vpool.copy_(torch.from_numpy(page(vc).reshape(-1).view(np.uint8)))
        ksc.copy_(torch.from_numpy(page(ks).reshape(-1)))
        vsc.copy_(torch.from_numpy(page(vs).reshape(-1)))
        fp.fp_op_attention_prefill(ptr(qkv), nqkv, 1, S, H, kv, ptr(att), ptr(err))
        lin(1, att, "wo", l, d, a.q_dim, h, resid=h)
        fp.fp_op_rmsnorm(ptr(h), S, d, 1, 0, ptr(ones), a.rms_eps, ptr(y))
        lin(2, y, "wgu", l, 2 * f, d, act)
        lin(1, act, "wdown", l, d, f, h, resid=h)
        got = quant.bf16_to_f32(host(h, np.uint16)).reshape(S, d)
        e = rel_err(got, ref_out)
        assert e <= 2e-2, ("block", l, e)
        h_in = quant.bf16_to_f32(synth.f32_to_bf16_bits(ref_out.astype(np.float32))).astype(np.float64)[None]
    # final norm and LM head on the oracle's last hidden row
    last = dev(synth.f32_to_bf16_bits(h_in[0, -1:].astype(np.float32)))
    yl = empty(d * 2)
    fp.fp_op_rmsnorm(ptr(last), 1, d, 1, 0, ptr(ones), a.rms_eps, ptr(yl))
    lg = empty(a.vocab * 4)
    lws = fp.fp_op_linear_workspace_bytes(0, 1, a.vocab, d)
    lw = empty(max(lws, 16))
    fp.fp_op_linear(0, 3, ptr(yl), 1, a.vocab, d, ptr(head), None, None, None, ptr(lg), ptr(lw), lws)
    ref_lg = M.rmsnorm(h_in[0, -1], w["final_norm"], a.rms_eps) @ w["lm_head"].T
    assert rel_err(host(lg, np.float32), ref_lg) <= 2e-2
    assert host(err, np.int32)[0] == 0
