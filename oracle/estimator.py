"""Latency and memory estimators of the paper, written out plainly (test infrastructure only).

Eq. 1 (Sec. 5.3):   latency = TTFT + output_length * TPOT
Eq. 2:              TTFT = num_layers * TTFT_layer + TTFT_other
Eq. 3:              TPOT = num_layers * TPOT_layer + TPOT_other

L2 (Sec. 5.3): profile the one- and two-layer fingerprints, each at two
output lengths; each fingerprint's 2x2 system (Eq. 1) gives its TTFT and
TPOT, and Eqs. 2-3 then give the per-layer and "other" terms.  The 4x4
system decouples into one 2x2 system for TTFT and one for TPOT.

M2 (Sec. 5.2), TP = PP = 1 column only: memory is linear in the number of
hidden layers (Sec. 5, Fig. "fingerprint scaling"), so two fingerprint
footprints give a per-layer slope and an intercept that extrapolate to the
full depth.
"""
from __future__ import annotations

import numpy as np


def solve_eq1(len_a, lat_a, len_b, lat_b):
    """Two (output_length, latency) observations -> (TTFT, TPOT)."""
    A = np.array([[1.0, len_a], [1.0, len_b]])
    ttft, tpot = np.linalg.solve(A, np.array([lat_a, lat_b], dtype=np.float64))
    return float(ttft), float(tpot)


def solve_eq23(layers_a, ttft_a, tpot_a, layers_b, ttft_b, tpot_b):
    """Two fingerprints -> (TTFT_layer, TTFT_other, TPOT_layer, TPOT_other)."""
    A = np.array([[layers_a, 1.0], [layers_b, 1.0]], dtype=np.float64)
    t_layer, t_other = np.linalg.solve(A, np.array([ttft_a, ttft_b], dtype=np.float64))
    p_layer, p_other = np.linalg.solve(A, np.array([tpot_a, tpot_b], dtype=np.float64))
    return float(t_layer), float(t_other), float(p_layer), float(p_other)


def predict_latency(num_layers, output_length, ttft_layer, ttft_other, tpot_layer, tpot_other):
    """Eq. 1 with Eqs. 2-3 substituted."""
    ttft = num_layers * ttft_layer + ttft_other
    tpot = num_layers * tpot_layer + tpot_other
    return ttft + output_length * tpot


def extrapolate_memory(layers_a, mem_a, layers_b, mem_b, num_layers):
    """Linear extrapolation of the footprint to ``num_layers`` hidden layers."""
    slope = (mem_b - mem_a) / (layers_b - layers_a)
    return mem_a + slope * (num_layers - layers_a)
