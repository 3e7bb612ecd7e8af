"""Pins of the oracle's byte counts and estimators (CPU only).

Byte counts: the closed forms of oracle/memory.py against the arrays the
quantisers produce, and the paper's statement that INT8 and INT4 cut weight
memory by about 50 % and 75 % (Sec. 3.2).  Estimators: Eq. 1-3 (Sec. 5.3) and
the linear layer-count extrapolation (Sec. 5.2, M2) recover known values from
exactly linear observations.
"""
import numpy as np
import pytest

import synth
from oracle import estimator, memory, quant
from oracle.model import Arch

L7 = Arch(2, 4096, 32, 32, 128, 11008, 32000)
L70 = Arch(2, 8192, 64, 8, 128, 28672, 32000)


@pytest.mark.parametrize("wq", [0, 1, 2])
def test_matrix_bytes_match_quantiser_output(wq):
    w = synth.weight_bf16(0, 0, 1, (6, 384))
    payload, _ = quant.quantize_weight(w, wq)
    assert sum(a.nbytes for a in payload.values()) == memory.matrix_bytes(6, 384, wq)


def test_quantisation_memory_ratios_match_paper():
    bf16 = memory.block_weight_bytes(L70, 0)
    assert abs(memory.block_weight_bytes(L70, 1) / bf16 - 0.50) < 0.01
    assert abs(memory.block_weight_bytes(L70, 2) / bf16 - 0.25) < 0.02


def test_decode_bytes_known_config():
    # 7B-shaped block: Wqkv 12288 x 4096 int8 = 50,331,648 + 24,576 bytes
    assert memory.matrix_bytes(12288, 4096, 1) == 50_356_224
    kv = memory.kv_bytes_per_token_block(L7, 0)
    assert kv == 2 * 32 * 128 * 2
    total = memory.decode_step_bytes(L7, 1, 0, 8, 600)
    assert total == 2 * (memory.block_weight_bytes(L7, 1) + 8 * 600 * kv) + 2 * 32000 * 4096


def test_eq1_recovers_ttft_tpot():
    ttft, tpot = 0.137, 0.0123
    lat = lambda n: ttft + n * tpot
    a, b = estimator.solve_eq1(25, lat(25), 100, lat(100))
    assert abs(a - ttft) < 1e-14 and abs(b - tpot) < 1e-15


def test_eq23_recovers_layer_terms():
    tl, to, pl, po = 0.011, 0.030, 0.0009, 0.0021
    f = lambda n: (n * tl + to, n * pl + po)
    r = estimator.solve_eq23(1, *f(1), 2, *f(2))
    assert np.allclose(r, (tl, to, pl, po), rtol=1e-12)
    assert abs(estimator.predict_latency(80, 100, *r) - (80 * tl + to + 100 * (80 * pl + po))) < 1e-12


def test_memory_extrapolation_linear():
    per, base = 1.25e9, 3.0e9
    m = estimator.extrapolate_memory(1, base + per, 2, base + 2 * per, 80)
    assert m == base + 80 * per
