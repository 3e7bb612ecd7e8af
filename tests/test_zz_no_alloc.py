"""fp_op_attention_decode_noalloc: decode attention for callers that cannot
allocate device memory (a host whose device memory is all reserved by another
framework's pool, a plugin that must not call the allocator, a loop that
cannot afford the synchronisation of cudaMalloc).  It runs the same kernels as
the allocating entry point (fp_op_attention_decode), with the split partials
in a scratch array the library holds instead of a caller workspace, so its
results must equal that entry point's bit for bit, call after call.  Every
case is one the split geometry cuts into several context splits, so the
scratch really carries partials and the combine kernel reads them back.
This file sorts last so that a run stopping at the first failure has run
every other test before it."""
import ctypes

import numpy as np
import pytest

import synth
from tests.gpu_helpers import dev, empty, host, ptr, torch_mod


def _paged_cache(fp, kvq, B, T, Hkv, hd, seed):
    pps = (T + 15) // 16
    n_pages = B * pps
    table = np.random.default_rng(seed).permutation(n_pages).reshape(B, pps).astype(np.int32)
    shape = (n_pages, Hkv, 16, hd)
    if kvq == 0:
        k = dev(synth.uniform_bf16(seed, 1, shape, -2, 2))
        v = dev(synth.uniform_bf16(seed, 2, shape, -2, 2))
        ks = vs = None
    else:
        rng = np.random.default_rng(seed + 100)
        k = dev(rng.integers(-127, 128, shape, dtype=np.int8))
        v = dev(rng.integers(-127, 128, shape, dtype=np.int8))
        ks = dev(synth.uniform_f32(seed, 4, (n_pages, Hkv, 16), 0.001, 0.02))
        vs = dev(synth.uniform_f32(seed, 5, (n_pages, Hkv, 16), 0.001, 0.02))
    td = dev(table)
    return fp.fp_kv_view(kvq, Hkv, hd, 16, pps, n_pages, ptr(k), ptr(v), ptr(ks), ptr(vs), ptr(td))


def _both(fp, kvq, lens, H, Hkv, hd, seed):
    """(allocating result, no-allocation result, error words) for one shape."""
    B, T = len(lens), max(lens) + 7
    assert fp.fp_op_attention_decode_splits(B, Hkv, hd, kvq, T) > 1, "the case must use the split partials"
    kv = _paged_cache(fp, kvq, B, T, Hkv, hd, seed)
    q = dev(synth.uniform_bf16(seed, 3, (B, H * hd), -2, 2))
    ln = dev(np.array(lens, np.int32))
    wsb = fp.fp_op_attention_decode_workspace_bytes(B, H, hd, T)
    assert wsb <= fp.FP_NOALLOC_SCRATCH_BYTES
    ws = empty(wsb)
    ref = empty(B * H * hd, np.uint16)
    got = empty(B * H * hd, np.uint16)
    err = empty(2, np.int32)
    fp.fp_op_attention_decode(ptr(q), H * hd, B, H, kv, ptr(ln), T, ptr(ref), ptr(ws), wsb, ptr(err))
    fp.fp_op_attention_decode_noalloc(ptr(q), H * hd, B, H, kv, ptr(ln), T, ptr(got), ptr(err) + 4)
    return host(ref, np.uint16), host(got, np.uint16), host(err, np.int32)


@pytest.mark.gpu
def test_noalloc_equals_allocating_entry_point_bit_for_bit():
    torch_mod()
    import paper_2501_13111_gb300 as fp

    cases = [  # (kvq, lens, H, Hkv, hd, seed)
        (0, [17, 300, 5], 16, 2, 128, 1),        # GQA, bf16 cache
        (1, [700, 129, 64, 1000], 8, 8, 64, 2),  # MHA, int8 cache, other sizes
        (1, [2148, 2000], 64, 8, 128, 3),        # the 70B-shaped GQA int8 layout
        (1, [2148, 2000], 64, 8, 128, 3),        # the same shape twice in a row
    ]
    for kvq, lens, H, Hkv, hd, seed in cases:
        ref, got, err = _both(fp, kvq, lens, H, Hkv, hd, seed)
        assert np.array_equal(ref, got), (kvq, lens, H, Hkv, hd)
        assert err.tolist() == [0, 0]


def test_noalloc_rejects_requests_beyond_its_scratch():
    """Checked on the host before any CUDA call: runs without a GPU."""
    import paper_2501_13111_gb300 as fp

    B, H, hd, max_len = 1, 128, 128, 40000
    assert fp.fp_op_attention_decode_workspace_bytes(B, H, hd, max_len) > fp.FP_NOALLOC_SCRATCH_BYTES
    kv = fp.fp_kv_view(0, 16, hd, 16, (max_len + 15) // 16, B * ((max_len + 15) // 16), 1, 1, None, None, 1)
    code = fp._lib.fp_op_attention_decode_noalloc(1, H * hd, B, H, ctypes.byref(kv), 1, max_len, 1, None, None)
    assert code == fp.FP_ERR_UNSUPPORTED
