"""Closed-form byte counts of a fingerprint (test infrastructure only).

The paper splits a deployment's footprint into weights W, activations A and
pipeline activations A_p (Sec. 5.2, "Breaking down an LLM's memory
footprint"), with mem_base = W + A for TP = PP = 1, and notes that INT8 and
INT4 cut weight memory by about 50 % and 75 % (Sec. 3.2).  These are the
exact byte counts of the storage formats read in ``quant.py``:

    bf16 matrix [N, K]:  2 N K
    int8 matrix:         N K + 2 N              (codes + bf16 scale per row)
    int4 matrix:         N K / 2 + 4 N K / 128  (packed codes + bf16 scale and zero per group)
    GPTQ4 matrix:        the int4 bytes + 4 K   (+ the int32 act order of the K input channels)
    KV per token per block: bf16 2 * Hkv * hd * 2;  int8 2 * Hkv * hd + 2 * Hkv * 4 (fp32 scales)

Decode reads every block matrix, the K/V of every cached token and the LM
head once per step; that sum is the algorithmic byte count of a step.
"""
from __future__ import annotations


def matrix_bytes(n: int, k: int, wquant: int) -> int:
    if wquant == 0:
        return 2 * n * k
    if wquant == 1:
        return n * k + 2 * n
    if wquant == 2:
        return n * k // 2 + 4 * n * (k // 128)
    if wquant == 3:
        return n * k // 2 + 4 * n * (k // 128) + 4 * k
    raise ValueError(wquant)


def block_matrices(arch):
    """(N, K) of the fused matrices of one block: Wqkv, Wo, Wgu, Wdown."""
    d, f = arch.hidden, arch.ffn
    return [(arch.q_dim + 2 * arch.kv_dim, d), (d, arch.q_dim), (2 * f, d), (d, f)]


def block_weight_bytes(arch, wquant: int) -> int:
    """Linear-layer bytes of one block (codes + scales/zeros), norms excluded."""
    return sum(matrix_bytes(n, k, wquant) for n, k in block_matrices(arch))


def block_norm_bytes(arch) -> int:
    return 2 * 2 * arch.hidden


def global_weight_bytes(arch) -> int:
    """Embedding, final norm gain and LM head, all bf16."""
    return 2 * arch.vocab * arch.hidden * 2 + 2 * arch.hidden


def weight_bytes(arch, wquant: int) -> int:
    return arch.n_layers * (block_weight_bytes(arch, wquant) + block_norm_bytes(arch)) + global_weight_bytes(arch)


def kv_bytes_per_token_block(arch, kvquant: int) -> int:
    if kvquant == 0:
        return 2 * arch.n_kv_heads * arch.head_dim * 2
    return 2 * arch.n_kv_heads * arch.head_dim + 2 * arch.n_kv_heads * 4


def decode_step_bytes(arch, wquant: int, kvquant: int, batch: int, cached: int) -> int:
    """Algorithmic HBM bytes of one decode step with ``cached`` tokens per sequence
    (including the new one): block matrices + K/V reads + LM head."""
    per_block = block_weight_bytes(arch, wquant) + batch * cached * kv_bytes_per_token_block(arch, kvquant)
    return arch.n_layers * per_block + 2 * arch.vocab * arch.hidden


def prefill_flops(arch, batch: int, prompt: int) -> int:
    """2 * tokens * block linear params * layers + causal attention (both matmuls)
    + the LM head on the last position of each sequence."""
    params = sum(n * k for n, k in block_matrices(arch))
    lin = 2 * batch * prompt * params * arch.n_layers
    att = 2 * batch * arch.n_heads * prompt * prompt * arch.head_dim * arch.n_layers
    head = 2 * batch * arch.vocab * arch.hidden
    return lin + att + head
