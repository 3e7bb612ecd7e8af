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


@pytest.mark.parametrize("wq", [0, 1, 2, 3])
def test_matrix_bytes_match_quantiser_output(wq):
    w = synth.weight_bf16(0, 0, 1, (6, 384))
    payload, _ = quant.quantize_weight(w, wq, synth.act_order(0, 0, 0, 384) if wq == 3 else None)
    assert sum(a.nbytes for a in payload.values()) == memory.matrix_bytes(6, 384, wq)


def test_quantisation_memory_ratios_match_paper():
    """INT8 halves and INT4 quarters the weight memory; GPTQ4 cuts it by about
    75 % too (Sec. 3.2 "Effect of Quantization")."""
    bf16 = memory.block_weight_bytes(L70, 0)
    assert abs(memory.block_weight_bytes(L70, 1) / bf16 - 0.50) < 0.01
    assert abs(memory.block_weight_bytes(L70, 2) / bf16 - 0.25) < 0.02
    assert abs(memory.block_weight_bytes(L70, 3) / bf16 - 0.25) < 0.02


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


# ---------------------------------------------------------------- prefill FLOPs
def _golden(name):
    import json
    import os

    return json.load(open(os.path.join(os.path.dirname(__file__), "golden", name)))


def test_prefill_flops_hand_counted_example():
    g = _golden("prefill_flops_example.json")
    a = Arch(**g["arch"])
    assert memory.prefill_flops(a, g["batch"], g["prompt"]) == g["total"]


def _loop_count_macs(arch, B, S):
    """Multiply-adds of a prefill, counted by walking the forward pass with
    explicit loops: each output element of a linear costs K multiply-adds,
    each causal (query, key) pair hd for the score and hd for the value
    product, the LM head one row of the last position per sequence."""
    lin = att_pairs = head = 0
    d, f, hd = arch.hidden, arch.ffn, arch.head_dim
    for _ in range(arch.n_layers):
        for _b in range(B):
            for _s in range(S):
                for n_out, k in ((arch.q_dim + 2 * arch.kv_dim, d), (d, arch.q_dim), (2 * f, d), (d, f)):
                    lin += n_out * k
            for _h in range(arch.n_heads):
                for i in range(S):
                    for _j in range(i + 1):
                        att_pairs += 1
    for _b in range(B):
        head += arch.vocab * d
    return lin, att_pairs * 2 * hd, head


@pytest.mark.parametrize("shape", [(1, 4, 2, 1, 2, 3, 5, 2, 3), (2, 64, 4, 2, 16, 96, 50, 3, 7),
                                   (1, 32, 8, 8, 4, 40, 11, 1, 1)])
def test_prefill_flops_against_loop_count(shape):
    *arch_t, B, S = shape
    a = Arch(*arch_t)
    lin, att, head = _loop_count_macs(a, B, S)
    # the closed form counts S^2/2 (query, key) pairs per head where the loops
    # count S(S+1)/2: S/2 pairs fewer, 2 hd multiply-adds each, per head,
    # sequence and layer
    fewer = a.n_layers * B * a.n_heads * S * a.head_dim
    assert memory.prefill_flops(a, B, S) == 2 * (lin + att - fewer + head)
