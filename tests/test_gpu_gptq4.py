"""GPTQ4 (int4 over act-order groups; GPTQ4 in the table "Models and
configurations", Sec. 3.2) through the C ABI against the oracle: the
quantiser bit for bit, the linear on its decode path (x gathered into the act
order, then the int4 decode linear) and its prefill path (weights expanded
back into channel order, then the tcgen05 GEMM), and a whole fingerprint
whose act orders the runtime draws from the seed."""
import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import quant
from tests.gpu_helpers import TAU, arch_dict, dev, empty, host, ptr, rel_err, torch_mod, upload_weights, weight_getter

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


def _on_device(fp, w, perm):
    n, k = w.shape
    codes = empty(n * k // 2)
    scales = empty(n * (k // 128), np.uint16)
    zeros = empty(n * (k // 128), np.uint16)
    fp.fp_op_quantize_gptq4(ptr(dev(w)), n, k, ptr(dev(perm)), ptr(codes), ptr(scales), ptr(zeros))
    return codes, scales, zeros


@pytest.mark.parametrize("n,k", [(37, 1408), (130, 4096)])
def test_quantize_bit_exact(fp, n, k):
    w = synth.weight_bf16(21, 1, 1, (n, k))
    w[0] = 0
    w[1, 7] = synth.f32_to_bf16_bits(np.array([0.75], np.float32))[0]
    perm = synth.act_order(4, 0, 2, k)
    codes, scales, zeros = _on_device(fp, w, perm)
    p, s, z = quant.quantize_gptq4(w, perm)
    assert np.array_equal(host(codes, np.uint8).reshape(n, k // 2), p)
    assert np.array_equal(host(scales, np.uint16).reshape(n, -1), s)
    assert np.array_equal(host(zeros, np.uint16).reshape(n, -1), z)


@pytest.mark.parametrize("m", [1, 8, 16, 17, 32, 64, 65, 300])
@pytest.mark.parametrize("epi", [0, 1, 2, 3])
@pytest.mark.parametrize("n,k", [(200, 512), (136, 4096)])
def test_linear_matches_oracle(fp, m, epi, n, k):
    """Decode sizes (gather + int4 GEMV on mma.sync or, at 17-64 rows,
    tcgen05) and prefill sizes (channel-order expansion + tcgen05 GEMM)."""
    w = synth.weight_bf16(23, 0, 1, (n, k))
    perm = synth.act_order(6, 1, 0, k)
    x = synth.uniform_bf16(24, m, (m, k), -2.0, 2.0)
    r = synth.uniform_bf16(25, m, (m, n), -1.0, 1.0)
    codes, scales, zeros = _on_device(fp, w, perm)
    _, wd = quant.quantize_weight(w, 3, perm)
    yref = quant.bf16_to_f32(x).astype(np.float64) @ wd.T
    nout = n // 2 if epi == 2 else n
    out = empty(m * nout * (4 if epi == 3 else 2))
    rd = dev(r[:, :nout].copy())
    wsb = fp.fp_op_linear_gptq4_workspace_bytes(m, n, k)
    ws = empty(wsb)
    err = empty(1, np.int32)
    fp.fp_op_linear_gptq4(epi, ptr(dev(x)), m, n, k, ptr(dev(perm)), ptr(codes), ptr(scales), ptr(zeros), ptr(rd),
                          ptr(out), ptr(ws), wsb, ptr(err))
    if epi == 3:
        got, ref = host(out, np.float32).reshape(m, n), yref
    else:
        got = quant.bf16_to_f32(host(out, np.uint16)).reshape(m, nout)
        if epi == 0:
            ref = yref
        elif epi == 1:
            ref = quant.bf16_to_f32(r[:, :nout]).astype(np.float64) + yref
        else:
            ref = M.silu(yref[:, :nout]) * yref[:, nout:]
    assert rel_err(got, ref) <= TAU[3] / 4, (m, epi, rel_err(got, ref))
    assert host(err, np.int32)[0] == 0


def test_act_order_entry_out_of_range_reads_zero(fp):
    """An act order with an entry outside [0, K) is read as a zero channel
    and reported in the error word; nothing is read outside x."""
    m, n, k = 4, 128, 256
    w = synth.weight_bf16(26, 0, 1, (n, k))
    perm = synth.act_order(7, 0, 0, k)
    codes, scales, zeros = _on_device(fp, w, perm)
    bad = perm.copy()
    bad[5] = k + 1000
    x = synth.uniform_bf16(27, m, (m, k), -2.0, 2.0)
    wsb = fp.fp_op_linear_gptq4_workspace_bytes(m, n, k)
    ws = empty(wsb)
    out = empty(m * n * 4)
    err = empty(1, np.int32)
    fp.fp_op_linear_gptq4(3, ptr(dev(x)), m, n, k, ptr(dev(bad)), ptr(codes), ptr(scales), ptr(zeros), None,
                          ptr(out), ptr(ws), wsb, ptr(err))
    assert host(err, np.int32)[0] == 1
    # the product is the stored matrix times x with act-order column 5 zeroed
    xa = quant.bf16_to_f32(x).astype(np.float64)[:, perm]
    xa[:, 5] = 0
    ref = xa @ quant.dequant_int4(*quant.quantize_gptq4(w, perm)).T
    assert rel_err(host(out, np.float32).reshape(m, n), ref) <= TAU[3] / 4


@pytest.mark.parametrize("B,S,N", [(2, 70, 4)])
def test_end_to_end(fp, B, S, N):
    """A 2-block GPTQ4 fingerprint with the int8 KV cache: the act orders the
    runtime draws equal the input generators', the codes equal the oracle's,
    and every block output and the logits match over prefill and decode."""
    arch = M.Arch(2, 1024, 16, 2, 128, 3584, 32000)
    seed = 4321
    get = weight_getter(seed)
    w, payload = M.build_weights(arch, 3, get, act_order=lambda l, m, k: synth.act_order(seed, l, m, k))
    T = S + N + 1
    h = fp.fp_create(arch_dict(arch), 3, 1, B, T, seed=seed, flags=fp.FP_FLAG_KEEP_HIDDEN | fp.FP_FLAG_NO_INIT)
    tau = TAU[3]
    try:
        upload_weights(fp, h, arch, get)
        for l in range(arch.n_layers):
            for mi, name in enumerate(("wqkv", "wo", "wgu", "wdown")):
                p = payload[(l, name)]
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_PERM, l, mi, np.int32), p["perm"]), (l, name)
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_CODES, l, mi, np.uint8), p["codes"].reshape(-1))
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_SCALES, l, mi, np.uint16), p["scales"].reshape(-1))
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_ZEROS, l, mi, np.uint16), p["zeros"].reshape(-1))
        toks = synth.tokens(seed, B * S, arch.vocab).reshape(B, S)
        ref = M.Fingerprint(arch, w, 1, B, T)

        def compare(out, rows, what):
            for l in range(arch.n_layers):
                g = quant.bf16_to_f32(fp.fp_get_tensor(h, fp.FP_G_HIDDEN, l, 0, np.uint16)).reshape(rows, -1)
                assert rel_err(g, out["hidden"][l].reshape(rows, -1)) <= tau, (what, l)
            lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(out["logits"].shape)
            assert rel_err(lg, out["logits"]) <= tau, (what, "logits", rel_err(lg, out["logits"]))

        def check_tokens(got, logits):
            want = M.argmax(logits)
            for b in range(B):
                if got[b] != want[b]:
                    top = np.sort(logits[b])[-2:]
                    assert top[1] - top[0] < 2 * tau * np.max(np.abs(logits[b])), b

        out = ref.prefill(toks)
        nxt = fp.fp_prefill(h, toks)
        compare(out, B * S, "prefill")
        check_tokens(nxt, out["logits"])
        tok = out["tokens"]
        for step in range(N):
            out = ref.decode(tok)
            got = fp.fp_decode_step(h, tok)
            compare(out, B, f"decode {step}")
            check_tokens(got, out["logits"])
            tok = out["tokens"]
    finally:
        fp.fp_destroy(h)


def test_seeded_handle_draws_the_generators_act_orders(fp):
    """fp_create without FP_FLAG_NO_INIT: act orders from the seed, and codes
    that are the oracle's GPTQ4 of the seeded weights."""
    arch = M.Arch(1, 512, 4, 4, 128, 1024, 32000)
    seed = 99
    h = fp.fp_create(arch_dict(arch), 3, 0, 1, 32, seed=seed)
    try:
        for mi in range(4):
            assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_PERM, 0, mi, np.int32),
                                  synth.act_order(seed, 0, mi, [512, 512, 512, 1024][mi]))
        wo = synth.weight_bf16(seed, 0, 4, (512, 512))
        p, s, z = quant.quantize_gptq4(wo, synth.act_order(seed, 0, 1, 512))
        assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_CODES, 0, 1, np.uint8), p.reshape(-1))
        assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_SCALES, 0, 1, np.uint16), s.reshape(-1))
    finally:
        fp.fp_destroy(h)
