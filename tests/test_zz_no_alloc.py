"""fp_op_attention_decode_noalloc: decode attention for callers that cannot
allocate device memory.  Its results must equal those of the allocating
entry point (fp_op_attention_decode) on the same inputs, call after call,
with the scratch the library holds instead of a caller workspace.  This file
sorts last so that a run stopping at the first failure has run every other
test before it."""
import ctypes

import numpy as np
import pytest

import synth
from oracle import quant
from tests.gpu_helpers import TAU, dev, empty, host, ptr, rel_err, torch_mod


def _paged_cache(fp, B, T, Hkv, hd, seed):
    pps = (T + 15) // 16
    n_pages = B * pps
    table = np.random.default_rng(seed).permutation(n_pages).reshape(B, pps).astype(np.int32)
    shape = (n_pages, Hkv, 16, hd)
    k = dev(synth.uniform_bf16(seed, 1, shape, -2, 2))
    v = dev(synth.uniform_bf16(seed, 2, shape, -2, 2))
    td = dev(table)
    return fp.fp_kv_view(0, Hkv, hd, 16, pps, n_pages, ptr(k), ptr(v), None, None, ptr(td))


@pytest.mark.gpu
def test_noalloc_matches_allocating_entry_point_twice_in_a_row():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    cases = [  # (lens, H, Hkv, hd, seed): a GQA call, then an MHA call with other sizes
        ([17, 300, 5], 16, 2, 128, 1),
        ([1, 129, 64, 1000], 8, 8, 64, 2),
    ]
    for lens, H, Hkv, hd, seed in cases:
        B, T = len(lens), max(lens) + 7
        kv = _paged_cache(fp, B, T, Hkv, hd, seed)
        q = dev(synth.uniform_bf16(seed, 3, (B, H * hd), -2, 2))
        ln = dev(np.array(lens, np.int32))
        wsb = fp.fp_op_attention_decode_workspace_bytes(B, H, hd, T)
        ws = empty(wsb)
        ref = empty(B * H * hd, np.uint16)
        got = empty(B * H * hd, np.uint16)
        err = empty(1, np.int32)
        fp.fp_op_attention_decode(ptr(q), H * hd, B, H, kv, ptr(ln), T, ptr(ref), ptr(ws), wsb, ptr(err))
        fp.fp_op_attention_decode_noalloc(ptr(q), H * hd, B, H, kv, ptr(ln), T, ptr(got), ptr(err))
        r = quant.bf16_to_f32(host(ref, np.uint16))
        g = quant.bf16_to_f32(host(got, np.uint16))
        assert rel_err(g, r) <= TAU[0]
        assert host(err, np.int32)[0] == 0


def test_noalloc_rejects_requests_beyond_its_scratch():
    """Checked on the host before any CUDA call: runs without a GPU."""
    import paper_2501_13111_gb300 as fp

    B, H, hd, max_len = 1, 128, 128, 40000
    assert fp.fp_op_attention_decode_workspace_bytes(B, H, hd, max_len) > fp.FP_NOALLOC_SCRATCH_BYTES
    kv = fp.fp_kv_view(0, 16, hd, 16, (max_len + 15) // 16, B * ((max_len + 15) // 16), 1, 1, None, None, 1)
    code = fp._lib.fp_op_attention_decode_noalloc(1, H * hd, B, H, ctypes.byref(kv), 1, max_len, 1, None, None)
    assert code == fp.FP_ERR_UNSUPPORTED
