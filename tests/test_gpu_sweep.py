"""The configuration sweep on the Llama-2-70B-shaped block (one decoder block
with the embedding and LM head): weights {bf16, int8 per channel, int4 g128}
x KV cache {bf16, int8} x batch {1, 8, 32, 64} x context {128, 512, 2048,
4096}.

Every point runs the way the sweep measures it: fp_create with device-side
seeded weights, a prefill of the full batch at the full context, then
fp_profile with decode steps.  Each point is checked against the oracle on a
batch-1 slice: every sequence's prompt opens with the same 64 tokens, and the
first 64 positions after the block of the first AND the last sequence are
compared -- the last sequence's rows sit at the end of the prefill's
M = batch x context rows (the last tiles of the GEMMs' persistent schedule,
the last (sequence, head) pairs of the attention).  Attention is causal, so
those rows do not depend on the rest of the prompt; their reference is
computed once per (weights, KV) pair, from the oracle's own seeded weights
and tokens.  Decode steps at these shapes are checked by
test_gpu_fullsize and test_gpu_model.
"""
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import quant
from tests.gpu_helpers import TAU, arch_dict, rel_err, torch_mod, weight_getter

pytestmark = pytest.mark.gpu

A70_BLOCK = M.Arch(1, 8192, 64, 8, 128, 28672, 32000)
BATCH = (1, 8, 32, 64)
CONTEXT = (128, 512, 2048, 4096)
PREFIX = 64
SEED = 3
PROFILE_DECODE = 4
TAU_KV8 = 5e-2


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


@pytest.fixture(scope="module")
def raw_weights():
    """bf16 tensors of the sweep (seed 3, unit gains), drawn once for all formats."""
    get = weight_getter(SEED, gains="ones")
    cache = {}

    def cached(layer, t, shape):
        if (layer, t) not in cache:
            cache[(layer, t)] = get(layer, t, shape)
        return cache[(layer, t)]

    return cached


@pytest.mark.parametrize("kvq", [0, 1])
@pytest.mark.parametrize("wq", [0, 1, 2])
def test_sweep_points_match_oracle(fp, raw_weights, wq, kvq):
    a = A70_BLOCK
    with ThreadPoolExecutor(max_workers=8) as pool:
        w, _ = M.build_weights(a, wq, raw_weights, map_fn=pool.map)
    stream = synth.tokens(SEED, max(BATCH) * max(CONTEXT), a.vocab)  # sequence 0's prompt opens the stream
    ref = M.Fingerprint(a, w, kvq, 1, PREFIX).prefill(stream[None, :PREFIX])["hidden"][0][0]
    del w
    # int8 KV: both sides quantise K and V independently from bf16 values that
    # may differ by one rounding, so codes flip by one step (s = amax / 127,
    # twice bf16's relative step) -- held to the quantised-path bound
    tau = max(TAU[wq], TAU_KV8) if kvq == 1 else TAU[wq]
    for B in BATCH:
        for ctx in CONTEXT:
            toks = stream[: B * ctx].reshape(B, ctx).copy()
            toks[:, :PREFIX] = stream[:PREFIX]  # the shared prefix the reference covers
            h = fp.fp_create(arch_dict(a), wq, kvq, B, ctx + 100 + 1, seed=SEED, flags=fp.FP_FLAG_KEEP_HIDDEN)
            try:
                fp.fp_prefill(h, toks, want_next=False)
                for b in sorted({0, B - 1}):
                    got = fp.fp_get_tensor(h, fp.FP_G_HIDDEN, 0, 0, np.uint16, count=PREFIX * a.hidden,
                                           offset=b * ctx * a.hidden)
                    got = quant.bf16_to_f32(got).reshape(PREFIX, a.hidden)
                    e = rel_err(got, ref)
                    assert e <= tau, (wq, kvq, B, ctx, b, e)
                r = fp.fp_profile(h, ctx, PROFILE_DECODE, warmup=0, iters=1, prompt=toks)
                assert r.ttft_ms > 0 and r.tpot_ms > 0, (wq, kvq, B, ctx)
                assert r.peak_hbm_bytes >= r.weight_bytes + r.kv_bytes, (wq, kvq, B, ctx)
            finally:
                fp.fp_destroy(h)
