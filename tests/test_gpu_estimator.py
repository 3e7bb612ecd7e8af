"""The paper's latency estimator (L2: Eqs. 1-3, Sec. 5.3) and memory
estimator (M2, TP = PP = 1, Sec. 5.2) on GB300 measurements.

Fingerprints of the Llama-2-7B-shaped workload (int8 weights, bf16 KV,
batch 8, prompt 512) with 1 and 2 hidden layers are profiled at two output
lengths; each gives TTFT and TPOT by Eq. 1, and the pair gives the per-layer
and "other" terms of Eqs. 2-3.  The prediction is then checked against
measured deeper models: 4 layers and the full 32-layer depth of Llama-2-7B.
The footprint (the handle's arena) extrapolates linearly from 1 and 2
layers and must equal the deeper handles' own byte plans exactly; the device
memory observed at the end of each profile (cudaMemGetInfo, what a monitor
of the GPU sees: arena, decode graph, driver rounding) must be predicted by
the same extrapolation within 2 %."""
import pytest

from tests.gpu_helpers import torch_mod

pytestmark = pytest.mark.gpu

ARCH = dict(hidden=4096, n_heads=32, n_kv_heads=32, head_dim=128, ffn=11008, vocab=32000, rms_eps=1e-5,
            rope_base=1e4)
WQ, KVQ, B, S = 1, 0, 8, 512
LENS = (16, 64)
N_CHECK = 100
REL_TOL = 0.05


@pytest.fixture(scope="module")
def fp():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    return fp


def _handle(fp, layers, n):
    return fp.fp_create(dict(ARCH, n_layers=layers), WQ, KVQ, B, S + n + 1, seed=0)


def _request_ms(fp, layers, n, iters=3):
    h = _handle(fp, layers, n)
    try:
        r = fp.fp_profile(h, S, n, warmup=1, iters=iters)
        return r.request_ms, r.peak_hbm_bytes, r.observed_hbm_bytes
    finally:
        fp.fp_destroy(h)


def test_l2_latency_and_m2_memory_predict_deeper_models(fp):
    _request_ms(fp, 1, LENS[0], iters=1)  # every kernel loaded once before any reading
    fits, mem, obs = {}, {}, {}
    for L in (1, 2):
        lat = [_request_ms(fp, L, n)[0] for n in LENS]
        obs[L] = _request_ms(fp, L, N_CHECK, iters=1)[2]  # the deeper handles' context capacity
        fits[L] = fp.fp_solve_eq1(LENS[0], lat[0], LENS[1], lat[1])
        assert fits[L].ttft > 0 and fits[L].tpot > 0
        h = _handle(fp, L, N_CHECK)
        try:
            mem[L] = fp.fp_get_plan(h).total_bytes
        finally:
            fp.fp_destroy(h)
    terms = fp.fp_solve_eq23(1, fits[1], 2, fits[2])
    assert terms.ttft_layer > 0 and terms.tpot_layer > 0
    for L in (4, 32):
        measured, peak, seen = _request_ms(fp, L, N_CHECK, iters=2)
        predicted = fp.fp_predict_latency(terms, L, N_CHECK)
        assert abs(predicted - measured) <= REL_TOL * measured, (L, predicted, measured)
        assert fp.fp_extrapolate_memory(1, mem[1], 2, mem[2], L) == peak, L
        assert seen >= peak, (L, seen, peak)  # the observed reading holds the arena and more
        pobs = fp.fp_extrapolate_memory(1, obs[1], 2, obs[2], L)
        assert abs(pobs - seen) <= 0.02 * seen, (L, pobs, seen)
