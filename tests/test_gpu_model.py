"""End-to-end parity of the fingerprint forward pass through the C ABI (fp.h)
against the oracle: quantised codes bit for bit, each block's output and the
logits within max|d| <= tau * max|ref|, greedy ids equal except on oracle
near-ties (top-2 gap < 2 tau max|logit|), after which both sides follow the
oracle's token (teacher forcing).  Plus the status codes of fp.h."""
import numpy as np
import pytest

import synth
from oracle import memory
from oracle import model as M
from oracle import quant
from tests.gpu_helpers import TAU, arch_dict, rel_err, torch_mod, upload_weights, weight_getter

pytestmark = pytest.mark.gpu

TINY = M.Arch(1, 512, 8, 8, 64, 1376, 32000)
CASES = {
    # name: (arch, wquant, kvquant, batch, prompt, decode steps, weight scale)
    "tiny_bf16": (TINY, 0, 0, 1, 32, 16, 1.0),
    "tiny_bf16_sharp": (TINY, 0, 0, 2, 45, 6, 4.0),
    "l7b_shape_int8": (M.Arch(2, 1024, 8, 8, 128, 2752, 32000), 1, 0, 3, 40, 5, 1.0),
    "l13b_shape_int4": (M.Arch(2, 1280, 10, 10, 128, 3456, 32000), 2, 0, 2, 70, 4, 1.0),
    "l70b_shape_int4_kv8": (M.Arch(2, 1024, 16, 2, 128, 3584, 32000), 2, 1, 4, 33, 4, 1.0),
    "int8_kv8_mha": (M.Arch(1, 512, 4, 4, 128, 1024, 32000), 1, 1, 2, 64, 3, 1.0),
    # Stress case: weights 3x sharper than the workload's.  Both sides quantise
    # K/V independently (bf16 inputs differ by rounding), so about one code in
    # six differs by one step; sharp attention amplifies that to ~2.2 % of
    # max|h| -- the oracle re-run with the device's rounding points gives the
    # same 2.2 %.  Checked against the int4-path bound.
    "int8_kv8_mha_sharp": (M.Arch(1, 512, 4, 4, 128, 1024, 32000), 1, 1, 2, 64, 3, 3.0),
}
TAU_CASE = {"int8_kv8_mha_sharp": 5e-2}


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


def _check_tokens(gpu_tok, ref_logits, tau):
    ref_tok = M.argmax(ref_logits)
    for b in range(len(gpu_tok)):
        if gpu_tok[b] != ref_tok[b]:
            top = np.sort(ref_logits[b])[-2:]
            assert top[1] - top[0] < 2 * tau * np.max(np.abs(ref_logits[b])), (b, gpu_tok[b], ref_tok[b])


def _compare_step(fp, h, arch, ref_out, rows, tau, what):
    for l in range(arch.n_layers):
        g = quant.bf16_to_f32(fp.fp_get_tensor(h, fp.FP_G_HIDDEN, l, 0, np.uint16)).reshape(rows, arch.hidden)
        r = ref_out["hidden"][l].reshape(rows, arch.hidden)
        assert rel_err(g, r) <= tau, (what, "hidden", l, rel_err(g, r))
    lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(ref_out["logits"].shape)
    assert rel_err(lg, ref_out["logits"]) <= tau, (what, "logits", rel_err(lg, ref_out["logits"]))
    return lg


def _payload_matches(fp, h, arch, wq, payload):
    for l in range(arch.n_layers):
        for m, name in enumerate(("wqkv", "wo", "wgu", "wdown")):
            p = payload[(l, name)]
            if wq == 0:
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_CODES, l, m, np.uint16), p["w"].reshape(-1))
                continue
            cdt = np.int8 if wq == 1 else np.uint8
            assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_CODES, l, m, cdt), p["codes"].reshape(-1)), (l, name)
            assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_SCALES, l, m, np.uint16), p["scales"].reshape(-1))
            if wq == 2:
                assert np.array_equal(fp.fp_get_tensor(h, fp.FP_G_W_ZEROS, l, m, np.uint16), p["zeros"].reshape(-1))


@pytest.mark.parametrize("name", list(CASES))
def test_end_to_end(fp, name):
    arch, wq, kvq, B, S, N, scale = CASES[name]
    tau = TAU_CASE.get(name, TAU[wq])
    seed = 1234 + len(name)
    get = weight_getter(seed, scale=scale)
    w, payload = M.build_weights(arch, wq, get)
    T = S + N + 1
    h = fp.fp_create(arch_dict(arch), wq, kvq, B, T, flags=fp.FP_FLAG_KEEP_HIDDEN | fp.FP_FLAG_NO_INIT)
    try:
        upload_weights(fp, h, arch, get)
        _payload_matches(fp, h, arch, wq, payload)
        pps = (T + 15) // 16
        table = np.random.default_rng(seed).permutation(B * pps).reshape(B, pps).astype(np.int32)
        fp.fp_set_page_table(h, table)
        toks = synth.tokens(seed, B * S, arch.vocab).reshape(B, S)
        ref = M.Fingerprint(arch, w, kvq, B, T)
        out = ref.prefill(toks)
        nxt = fp.fp_prefill(h, toks)
        _compare_step(fp, h, arch, out, B * S, tau, "prefill")
        _check_tokens(nxt, out["logits"], tau)
        tok = out["tokens"]
        for step in range(N):
            out = ref.decode(tok)
            got = fp.fp_decode_step(h, tok)
            _compare_step(fp, h, arch, out, B, tau, f"decode {step}")
            _check_tokens(got, out["logits"], tau)
            tok = out["tokens"]
        assert fp.fp_get_tensor(h, fp.FP_G_LENGTH, 0, 0, np.int32).tolist() == [S + N] * B
    finally:
        fp.fp_destroy(h)


def test_device_tokens_follow_argmax(fp):
    """Without host tokens the decode graph feeds its own argmax back."""
    arch = TINY
    h = fp.fp_create(arch_dict(arch), 0, 0, 2, 40, seed=3)
    try:
        toks = synth.tokens(3, 2 * 8, arch.vocab).reshape(2, 8)
        first = fp.fp_prefill(h, toks)
        a = fp.fp_decode_step(h, None, batch=2)
        h2 = fp.fp_create(arch_dict(arch), 0, 0, 2, 40, seed=3)
        try:
            assert np.array_equal(fp.fp_prefill(h2, toks), first)
            b = fp.fp_decode_step(h2, first)
            assert np.array_equal(a, b)
            lg = fp.fp_get_tensor(h2, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(2, -1)
            assert np.array_equal(b, M.argmax(lg.astype(np.float64)))
        finally:
            fp.fp_destroy(h2)
    finally:
        fp.fp_destroy(h)


@pytest.mark.parametrize("wq", [0, 1, 2])
def test_seeded_init_matches_generator(fp, wq):
    arch = M.Arch(1, 512, 4, 2, 128, 1024, 1000)
    h = fp.fp_create(arch_dict(arch), wq, 0, 1, 32, seed=77)
    try:
        get = lambda l, t, shape: (synth.f32_to_bf16_bits(np.ones(shape, np.float32)) if len(shape) == 1
                                   else synth.weight_bf16(77, l, t, shape))
        _, payload = M.build_weights(arch, wq, get)
        _payload_matches(fp, h, arch, wq, payload)
        plan = fp.fp_get_plan(h)
        assert plan.weight_bytes == memory.weight_bytes(arch, wq)
        assert plan.total_bytes >= plan.weight_bytes + plan.kv_bytes + plan.act_bytes
    finally:
        fp.fp_destroy(h)


def test_status_codes(fp):
    arch = TINY
    h = fp.fp_create(arch_dict(arch), 0, 0, 2, 10, seed=1)
    try:
        with pytest.raises(fp.FPError) as e:
            fp.fp_decode_step(h, np.array([1, 2], np.int32))
        assert e.value.code == fp.FP_ERR_STATE
        with pytest.raises(fp.FPError) as e:
            fp.fp_prefill(h, np.array([[1, 2, 32000], [0, 0, 0]], np.int32))
        assert e.value.code == fp.FP_ERR_INVALID_ARG
        with pytest.raises(fp.FPError) as e:
            fp.fp_prefill(h, np.zeros((2, 11), np.int32))
        assert e.value.code == fp.FP_ERR_CAPACITY
        fp.fp_prefill(h, np.zeros((2, 9), np.int32))
        fp.fp_decode_step(h, None, batch=2)
        with pytest.raises(fp.FPError) as e:
            fp.fp_decode_step(h, None, batch=2)
        assert e.value.code == fp.FP_ERR_CAPACITY
        with pytest.raises(fp.FPError) as e:
            fp.fp_set_page_table(h, np.zeros((2, 1), np.int32))
        assert e.value.code == fp.FP_ERR_INVALID_ARG
        with pytest.raises(fp.FPError) as e:
            fp.fp_set_weight(h, 0, fp.FP_T_WQ, np.zeros(10, np.uint16))
        assert e.value.code == fp.FP_ERR_INVALID_ARG
        with pytest.raises(fp.FPError) as e:
            fp.fp_profile(h, 8, 5)
        assert e.value.code == fp.FP_ERR_CAPACITY
    finally:
        fp.fp_destroy(h)


def test_allocator_failure_is_clean(fp):
    arch = TINY
    for fail_after in (0, 1):
        alloc = fp.TorchAllocator(fail_after=fail_after)
        with pytest.raises(fp.FPError) as e:
            fp.fp_create(arch_dict(arch), 0, 0, 1, 64, allocator=alloc.struct)
        assert e.value.code == fp.FP_ERR_OOM
        assert not alloc.live
    alloc = fp.TorchAllocator()
    h = fp.fp_create(arch_dict(arch), 1, 1, 2, 64, allocator=alloc.struct)
    assert len(alloc.live) == 1
    fp.fp_prefill(h, np.ones((2, 5), np.int32))
    fp.fp_destroy(h)
    assert not alloc.live


def test_profile_reports(fp):
    arch = M.Arch(2, 1024, 8, 8, 128, 2752, 32000)
    h = fp.fp_create(arch_dict(arch), 1, 0, 4, 128, seed=5)
    try:
        r = fp.fp_profile(h, 64, 16, warmup=1, iters=2)
        assert r.ttft_ms > 0 and r.tpot_ms > 0 and r.decode_tokens_per_s > 0
        assert r.weight_bytes == memory.weight_bytes(arch, 1)
        assert r.decode_bytes_per_step == int(memory.decode_step_bytes(arch, 1, 0, 4, 64 + 8.5))
        assert r.prefill_flops == memory.prefill_flops(arch, 4, 64)
        assert all(x > 0 for x in list(r.block_ms)[:2])
        # embed + first norm; per block 7 launches (6 in the first) + decode attention (1, or 2 with a
        # combine pass); final norm, head, argmax (which also advances the positions)
        assert r.decode_launches in (1 + (7 + 1) * 2 - 1 + 3, 1 + (7 + 2) * 2 - 1 + 3)
        assert r.peak_hbm_bytes >= r.weight_bytes + r.kv_bytes
    finally:
        fp.fp_destroy(h)


def test_fp16_overflow_in_decode_linear_is_reported(fp):
    """The decode GEMV stages x as fp16 for int8 / int4 weights.  An
    activation beyond the fp16 range (here a pre-attention norm gain of
    about 1e5 makes |y| > 65504) must not pass silently: the step returns
    FP_ERR_DEVICE_ASSERT and says why; a later step with sane gains is clean."""
    arch = M.Arch(1, 512, 8, 8, 64, 1376, 32000)
    h = fp.fp_create(arch_dict(arch), 1, 0, 2, 64, seed=9)
    try:
        toks = synth.tokens(9, 2 * 40, arch.vocab).reshape(2, 40)
        fp.fp_prefill(h, toks)
        big = synth.f32_to_bf16_bits(np.full(arch.hidden, 1e5, np.float32))
        fp.fp_set_weight(h, 0, fp.FP_T_ATTN_NORM, big)
        with pytest.raises(fp.FPError) as e:
            fp.fp_decode_step(h, np.array([1, 2], np.int32))
        assert e.value.code == fp.FP_ERR_DEVICE_ASSERT
        assert "fp16" in str(e.value)
        fp.fp_set_weight(h, 0, fp.FP_T_ATTN_NORM, synth.f32_to_bf16_bits(np.ones(arch.hidden, np.float32)))
        fp.fp_prefill(h, toks)
        fp.fp_decode_step(h, np.array([1, 2], np.int32))  # clean again: the error word was cleared
    finally:
        fp.fp_destroy(h)


def test_expired_wait_in_the_tcgen05_gemm_is_reported(fp):
    """The failure path of the pipelined tensor-core kernels, without a fault:
    the test lowers the prefill GEMM's stage wait to zero rounds, so its MMA
    thread gives up at the first stage; the CTA drains what it issued, frees
    its tensor memory and records status 2.  The prefill then returns
    FP_ERR_DEVICE_ASSERT, and with the default restored the same handle runs
    clean and matches the oracle."""
    arch = M.Arch(1, 512, 8, 8, 64, 1376, 32000)
    B, S = 2, 40  # 80 prompt rows: the prefill linears run on the tcgen05 GEMM
    get = weight_getter(13)
    w, _ = M.build_weights(arch, 0, get)
    h = fp.fp_create(arch_dict(arch), 0, 0, B, 64, flags=fp.FP_FLAG_NO_INIT)
    try:
        upload_weights(fp, h, arch, get)
        toks = synth.tokens(13, B * S, arch.vocab).reshape(B, S)
        fp.fp_debug_set_wait_limit(0)
        try:
            with pytest.raises(fp.FPError) as e:
                fp.fp_prefill(h, toks)
        finally:
            fp.fp_debug_set_wait_limit(-1)
        assert e.value.code == fp.FP_ERR_DEVICE_ASSERT
        assert "bounded wait" in str(e.value)
        nxt = fp.fp_prefill(h, toks)
        out = M.Fingerprint(arch, w, 0, B, 64).prefill(toks)
        lg = fp.fp_get_tensor(h, fp.FP_G_LOGITS, 0, 0, np.float32).reshape(B, -1)
        assert rel_err(lg, out["logits"]) <= TAU[0]
        assert nxt.shape == (B,)
    finally:
        fp.fp_destroy(h)
