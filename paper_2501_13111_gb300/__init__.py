"""Python binding of libfp.so: the C ABI of include/fp.h and include/fp_ops.h.

Argument marshalling only: every step of the fingerprint forward pass runs in
the library's CUDA kernels.  Functions keep the C names.  Device buffers are
passed as integers (``tensor.data_ptr()``), streams as ``cudaStream_t``
integers (``torch.cuda.current_stream().cuda_stream``).  A call that returns
a negative status raises ``FPError`` with the library's message.

The library must have been built (``python paper_2501_13111_gb300/build.py``
or ``__graft_entry__.build()``); importing this module without it raises
ImportError -- there is no fallback implementation.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfp.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                      "(or python paper_2501_13111_gb300/build.py)")
_lib = C.CDLL(LIB_PATH)

# ------------------------------------------------------------------ constants
FP_OK, FP_ERR_INVALID_ARG, FP_ERR_UNSUPPORTED, FP_ERR_OOM = 0, -1, -2, -3
FP_ERR_CUDA, FP_ERR_CAPACITY, FP_ERR_DEVICE_ASSERT, FP_ERR_STATE = -4, -5, -6, -7
FP_W_BF16, FP_W_INT8, FP_W_INT4_G128, FP_W_GPTQ4 = 0, 1, 2, 3
FP_KV_BF16, FP_KV_INT8 = 0, 1
FP_FLAG_KEEP_HIDDEN, FP_FLAG_NO_INIT = 1, 2
FP_MAX_LAYERS = 80
(FP_T_ATTN_NORM, FP_T_WQ, FP_T_WK, FP_T_WV, FP_T_WO, FP_T_FFN_NORM, FP_T_WGATE, FP_T_WUP,
 FP_T_WDOWN) = range(9)
FP_T_EMBED, FP_T_FINAL_NORM, FP_T_LM_HEAD = 0, 1, 2
FP_M_QKV, FP_M_O, FP_M_GU, FP_M_DOWN = 0, 1, 2, 3
(FP_G_W_CODES, FP_G_W_SCALES, FP_G_W_ZEROS, FP_G_K_POOL, FP_G_V_POOL, FP_G_K_SCALES, FP_G_V_SCALES,
 FP_G_HIDDEN, FP_G_LOGITS, FP_G_TOKENS, FP_G_PAGE_TABLE, FP_G_LENGTH, FP_G_W_PERM) = range(13)
KERNEL_CLASSES = ("embed", "rmsnorm", "lin_qkv", "rope_kv", "attn", "attn_combine", "lin_o", "lin_gu",
                  "lin_down", "lm_head", "argmax")
FP_K_COUNT = len(KERNEL_CLASSES)
FP_EPI_STORE, FP_EPI_RESID, FP_EPI_SWIGLU, FP_EPI_F32 = 0, 1, 2, 3


class FPError(RuntimeError):
    def __init__(self, code, message):
        super().__init__(f"{_lib.fp_strerror(code).decode()} ({code}): {message}")
        self.code = code


# ------------------------------------------------------------------ structs
class fp_arch(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("hidden", C.c_int), ("n_heads", C.c_int), ("n_kv_heads", C.c_int),
                ("head_dim", C.c_int), ("ffn", C.c_int), ("vocab", C.c_int), ("rms_eps", C.c_float),
                ("rope_base", C.c_float)]


ALLOC_FN = C.CFUNCTYPE(C.c_void_p, C.c_size_t, C.c_void_p)
FREE_FN = C.CFUNCTYPE(None, C.c_void_p, C.c_void_p)


class fp_allocator(C.Structure):
    _fields_ = [("alloc", ALLOC_FN), ("free", FREE_FN), ("ctx", C.c_void_p)]


class fp_profile_result(C.Structure):
    _fields_ = [("ttft_ms", C.c_double), ("tpot_ms", C.c_double), ("tpot_ms_p50", C.c_double),
                ("decode_tokens_per_s", C.c_double), ("prefill_tflops", C.c_double),
                ("prefill_flops", C.c_double), ("block_ms", C.c_double * FP_MAX_LAYERS),
                ("other_ms", C.c_double), ("kernel_ms", C.c_double * FP_K_COUNT),
                ("kernel_launches", C.c_int * FP_K_COUNT), ("decode_launches", C.c_int),
                ("prefill_launches", C.c_int),
                ("block_bytes", C.c_ulonglong * FP_MAX_LAYERS), ("peak_hbm_bytes", C.c_ulonglong),
                ("weight_bytes", C.c_ulonglong), ("kv_bytes", C.c_ulonglong), ("act_bytes", C.c_ulonglong),
                ("workspace_bytes", C.c_ulonglong), ("memgetinfo_bytes", C.c_ulonglong),
                ("decode_bytes_per_step", C.c_ulonglong), ("n_layers", C.c_int), ("prompt_len", C.c_int),
                ("n_decode", C.c_int), ("iters", C.c_int), ("request_ms", C.c_double),
                ("observed_hbm_bytes", C.c_ulonglong)]

    def as_dict(self):
        d = {}
        for name, _ in self._fields_:
            v = getattr(self, name)
            d[name] = list(v) if hasattr(v, "__len__") else v
        d["block_ms"] = d["block_ms"][: self.n_layers]
        d["block_bytes"] = d["block_bytes"][: self.n_layers]
        d["kernel_ms"] = dict(zip(KERNEL_CLASSES, d["kernel_ms"]))
        d["kernel_launches"] = dict(zip(KERNEL_CLASSES, d["kernel_launches"]))
        return d


class fp_plan(C.Structure):
    _fields_ = [("weight_bytes", C.c_ulonglong), ("kv_bytes", C.c_ulonglong), ("act_bytes", C.c_ulonglong),
                ("workspace_bytes", C.c_ulonglong), ("total_bytes", C.c_ulonglong),
                ("pages_per_seq", C.c_int), ("max_rows", C.c_int)]


class fp_kv_view(C.Structure):
    _fields_ = [("kvquant", C.c_int), ("n_kv_heads", C.c_int), ("head_dim", C.c_int), ("page_size", C.c_int),
                ("pages_per_seq", C.c_int), ("n_pages", C.c_int), ("k_pool", C.c_void_p),
                ("v_pool", C.c_void_p), ("k_scale", C.c_void_p), ("v_scale", C.c_void_p),
                ("page_table", C.c_void_p)]


class fp_eq1_fit(C.Structure):
    _fields_ = [("ttft", C.c_double), ("tpot", C.c_double)]


class fp_l2_terms(C.Structure):
    _fields_ = [("ttft_layer", C.c_double), ("ttft_other", C.c_double), ("tpot_layer", C.c_double),
                ("tpot_other", C.c_double)]


# ------------------------------------------------------------------ prototypes
_P = C.c_void_p
_I, _U, _F, _SZ, _LL, _ULL = C.c_int, C.c_uint, C.c_float, C.c_size_t, C.c_longlong, C.c_ulonglong
_PROTOS = {
    "fp_create": (_I, [C.POINTER(fp_arch), _I, _I, _I, _I, _I, _ULL, _U, C.POINTER(fp_allocator), _P,
                       C.POINTER(_P)]),
    "fp_set_weight": (_I, [_P, _I, _I, _P, _SZ]),
    "fp_set_page_table": (_I, [_P, _P]),
    "fp_load_prompt": (_I, [_P, _P, _I]),
    "fp_prefill": (_I, [_P, _P, _I, _P]),
    "fp_decode_steps": (_I, [_P, _I]),
    "fp_decode_step": (_I, [_P, _P, _P]),
    "fp_profile": (_I, [_P, _I, _I, _I, _I, _P, C.POINTER(fp_profile_result)]),
    "fp_get_tensor": (_LL, [_P, _I, _I, _I, _P, _SZ]),
    "fp_get_tensor_at": (_LL, [_P, _I, _I, _I, _SZ, _P, _SZ]),
    "fp_get_plan": (_I, [_P, C.POINTER(fp_plan)]),
    "fp_last_error": (C.c_char_p, [_P]),
    "fp_strerror": (C.c_char_p, [_I]),
    "fp_destroy": (None, [_P]),
    "fp_op_quantize": (_I, [_I, _P, _I, _I, _P, _P, _P, _P]),
    "fp_op_init_weights": (_I, [_P, _LL, _ULL, _LL, _LL, _P]),
    "fp_op_linear": (_I, [_I, _I, _P, _I, _I, _I, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "fp_op_linear_workspace_bytes": (_SZ, [_I, _I, _I, _I]),
    "fp_op_quantize_gptq4": (_I, [_P, _I, _I, _P, _P, _P, _P, _P]),
    "fp_op_linear_gptq4": (_I, [_I, _P, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _SZ, _P, _P]),
    "fp_op_linear_gptq4_workspace_bytes": (_SZ, [_I, _I, _I]),
    "fp_op_rmsnorm": (_I, [_P, _I, _I, _I, _I, _P, _F, _P, _P]),
    "fp_op_embed": (_I, [_P, _I, _P, _I, _I, _P, _P, _P]),
    "fp_op_rope_table": (_I, [_I, _I, _F, _P, _P]),
    "fp_op_rope_kv": (_I, [_P, _I, _I, _I, _I, C.POINTER(fp_kv_view), _P, _P, _P, _P]),
    "fp_op_attention_decode": (_I, [_P, _I, _I, _I, C.POINTER(fp_kv_view), _P, _I, _P, _P, _SZ, _P, _P]),
    "fp_op_attention_decode_workspace_bytes": (_SZ, [_I, _I, _I, _I]),
    "fp_op_attention_decode_splits": (_I, [_I, _I, _I, _I, _I]),
    "fp_op_attention_decode_noalloc": (_I, [_P, _I, _I, _I, C.POINTER(fp_kv_view), _P, _I, _P, _P, _P]),
    "fp_op_attention_prefill": (_I, [_P, _I, _I, _I, _I, C.POINTER(fp_kv_view), _P, _P, _P]),
    "fp_op_argmax": (_I, [_P, _I, _I, _P, _P]),
    "fp_debug_set_wait_limit": (_I, [_LL]),
    "fp_solve_eq1": (_I, [_I, C.c_double, _I, C.c_double, C.POINTER(fp_eq1_fit)]),
    "fp_solve_eq23": (_I, [_I, C.POINTER(fp_eq1_fit), _I, C.POINTER(fp_eq1_fit), C.POINTER(fp_l2_terms)]),
    "fp_predict_latency": (_I, [C.POINTER(fp_l2_terms), _I, _I, C.POINTER(C.c_double)]),
    "fp_extrapolate_memory": (_I, [_I, C.c_double, _I, C.c_double, _I, C.POINTER(C.c_double)]),
}
for _name, (_res, _args) in _PROTOS.items():
    _f = getattr(_lib, _name)
    _f.restype = _res
    _f.argtypes = _args

EXPORTED = tuple(_PROTOS)


def _check(code, handle=None):
    if code < 0:
        msg = _lib.fp_last_error(handle).decode() if handle is not None else _lib.fp_last_error(None).decode()
        raise FPError(int(code), msg)
    return code


def _ptr(a):
    """Host numpy array -> void*; device pointers (ints) pass through."""
    if a is None:
        return None
    if isinstance(a, int):
        return a
    return a.ctypes.data_as(C.c_void_p)


# ------------------------------------------------------------------ fp.h
def fp_create(arch, wquant, kvquant, batch, max_context, page_size=16, seed=0, flags=0, allocator=None,
              stream=None):
    """Returns the handle (opaque int).  ``arch``: fp_arch or a dict of its fields."""
    if isinstance(arch, dict):
        arch = fp_arch(**arch)
    out = C.c_void_p()
    code = _lib.fp_create(C.byref(arch), wquant, kvquant, batch, max_context, page_size, seed, flags,
                          C.byref(allocator) if allocator is not None else None, stream, C.byref(out))
    _check(code)
    return out.value


def fp_set_weight(h, layer, tensor, host_bf16: np.ndarray):
    a = np.ascontiguousarray(host_bf16, dtype=np.uint16)
    return _check(_lib.fp_set_weight(h, layer, tensor, _ptr(a), a.size), h)


def fp_set_page_table(h, table: np.ndarray):
    t = np.ascontiguousarray(table, dtype=np.int32)
    return _check(_lib.fp_set_page_table(h, _ptr(t)), h)


def fp_load_prompt(h, tokens, prompt_len=None):
    """tokens int32 [batch][prompt_len], or None for the seeded prompt of length prompt_len."""
    if tokens is None:
        return _check(_lib.fp_load_prompt(h, None, prompt_len), h)
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    return _check(_lib.fp_load_prompt(h, _ptr(t), t.shape[1]), h)


def fp_prefill(h, tokens, want_next=True, prompt_len=None, out=None):
    """tokens int32 [batch][prompt_len] (None: the resident prompt of length
    prompt_len); returns the next tokens [batch] (``out`` if given) or None."""
    if tokens is None:
        t, S = None, prompt_len
    else:
        t = tokens if (isinstance(tokens, np.ndarray) and tokens.dtype == np.int32 and tokens.flags.c_contiguous) \
            else np.ascontiguousarray(tokens, dtype=np.int32)
        S = t.shape[1]
    nxt = out
    if want_next and nxt is None:
        nxt = np.empty(fp_get_tensor(h, FP_G_TOKENS) // 4, np.int32)
    _check(_lib.fp_prefill(h, _ptr(t), S, _ptr(nxt) if want_next else None), h)
    return nxt if want_next else None


def fp_decode_steps(h, n):
    return _check(_lib.fp_decode_steps(h, n), h)


def fp_decode_step(h, tokens_in=None, want_out=True, batch=None, out=None):
    tin = None if tokens_in is None else np.ascontiguousarray(tokens_in, dtype=np.int32)
    if want_out and out is None:
        n = batch if batch is not None else (tin.shape[0] if tin is not None else
                                              fp_get_tensor(h, FP_G_TOKENS) // 4)
        out = np.empty(n, np.int32)
    _check(_lib.fp_decode_step(h, _ptr(tin), _ptr(out) if want_out else None), h)
    return out if want_out else None


def fp_profile(h, prompt_len, n_decode, warmup=1, iters=3, prompt=None):
    res = fp_profile_result()
    p = None if prompt is None else np.ascontiguousarray(prompt, dtype=np.int32)
    _check(_lib.fp_profile(h, prompt_len, n_decode, warmup, iters, _ptr(p), C.byref(res)), h)
    return res


def fp_get_tensor(h, what, layer=0, mat=0, dtype=None, count=None, offset=0):
    """With dtype None returns the byte size, else a host array of that dtype
    (its first ``count`` elements when given, from element ``offset`` on)."""
    if dtype is None:
        return _check(_lib.fp_get_tensor(h, what, layer, mat, None, 0), h)
    isz = np.dtype(dtype).itemsize
    n = _check(_lib.fp_get_tensor_at(h, what, layer, mat, offset * isz, None, 0), h)
    k = n // isz
    buf = np.empty(k if count is None else min(k, count), dtype=dtype)
    _check(_lib.fp_get_tensor_at(h, what, layer, mat, offset * isz, _ptr(buf), buf.nbytes), h)
    return buf


def fp_get_plan(h):
    p = fp_plan()
    _check(_lib.fp_get_plan(h, C.byref(p)), h)
    return p


def fp_last_error(h=None):
    return _lib.fp_last_error(h).decode()


def fp_strerror(code):
    return _lib.fp_strerror(code).decode()


def fp_destroy(h):
    _lib.fp_destroy(h)


# ------------------------------------------------------------------ fp_ops.h
def fp_op_quantize(wquant, w, N, K, codes, scales, zeros, stream=None):
    return _check(_lib.fp_op_quantize(wquant, w, N, K, codes, scales, zeros, stream))


def fp_op_init_weights(w, n, seed, stream_id, start=0, stream=None):
    return _check(_lib.fp_op_init_weights(w, n, seed, stream_id, start, stream))


def fp_op_linear_workspace_bytes(wquant, M, N, K):
    return _lib.fp_op_linear_workspace_bytes(wquant, M, N, K)


def fp_op_quantize_gptq4(w, N, K, perm, codes, scales, zeros, stream=None):
    return _check(_lib.fp_op_quantize_gptq4(w, N, K, perm, codes, scales, zeros, stream))


def fp_op_linear_gptq4_workspace_bytes(M, N, K):
    return _lib.fp_op_linear_gptq4_workspace_bytes(M, N, K)


def fp_op_linear_gptq4(epilogue, x, M, N, K, perm, codes, scales, zeros, residual, y, workspace, workspace_bytes,
                       err=None, stream=None):
    return _check(_lib.fp_op_linear_gptq4(epilogue, x, M, N, K, perm, codes, scales, zeros, residual, y, workspace,
                                          workspace_bytes, err, stream))


def fp_op_linear(wquant, epilogue, x, M, N, K, codes, scales, zeros, residual, y, workspace=None,
                 workspace_bytes=0, stream=None):
    return _check(_lib.fp_op_linear(wquant, epilogue, x, M, N, K, codes, scales, zeros, residual, y, workspace,
                                    workspace_bytes, stream))


def fp_op_rmsnorm(x, M, d, row_stride, row_offset, g, eps, y, stream=None):
    return _check(_lib.fp_op_rmsnorm(x, M, d, row_stride, row_offset, g, eps, y, stream))


def fp_op_embed(tok, M, E, V, d, h, err=None, stream=None):
    return _check(_lib.fp_op_embed(tok, M, E, V, d, h, err, stream))


def fp_op_rope_table(max_pos, head_dim, base, cs, stream=None):
    return _check(_lib.fp_op_rope_table(max_pos, head_dim, base, cs, stream))


def fp_op_rope_kv(qkv, B, S, row_stride, n_heads, kv: fp_kv_view, pos, rope_cs, err=None, stream=None):
    return _check(_lib.fp_op_rope_kv(qkv, B, S, row_stride, n_heads, C.byref(kv), pos, rope_cs, err, stream))


def fp_op_attention_decode_workspace_bytes(B, n_heads, head_dim, max_len):
    return _lib.fp_op_attention_decode_workspace_bytes(B, n_heads, head_dim, max_len)


def fp_op_attention_decode(q, q_stride, B, n_heads, kv: fp_kv_view, lens, max_len, out, workspace,
                           workspace_bytes, err=None, stream=None):
    return _check(_lib.fp_op_attention_decode(q, q_stride, B, n_heads, C.byref(kv), lens, max_len, out, workspace,
                                              workspace_bytes, err, stream))


def fp_op_attention_decode_splits(B, n_kv_heads, head_dim, kvquant, max_len):
    return _lib.fp_op_attention_decode_splits(B, n_kv_heads, head_dim, kvquant, max_len)


FP_NOALLOC_SCRATCH_BYTES = 32 << 20  # FP_NOALLOC_SCRATCH_BYTES of fp_ops.h (a CPU test keeps the two equal)


def fp_op_attention_decode_noalloc(q, q_stride, B, n_heads, kv: fp_kv_view, lens, max_len, out, err=None,
                                   stream=None):
    """Decode attention with the library's own fixed scratch (no workspace argument)."""
    return _check(_lib.fp_op_attention_decode_noalloc(q, q_stride, B, n_heads, C.byref(kv), lens, max_len, out,
                                                      err, stream))


def fp_op_attention_prefill(q, q_stride, B, S, n_heads, kv: fp_kv_view, out, err=None, stream=None):
    return _check(_lib.fp_op_attention_prefill(q, q_stride, B, S, n_heads, C.byref(kv), out, err, stream))


def fp_op_argmax(logits, M, V, out, stream=None):
    return _check(_lib.fp_op_argmax(logits, M, V, out, stream))


def fp_debug_set_wait_limit(rounds):
    """Test hook: polling rounds of the prefill GEMM's stage wait (< 0: default)."""
    return _check(_lib.fp_debug_set_wait_limit(rounds))


# ------------------------------------------------------------------ torch plumbing
class TorchAllocator:
    """fp_allocator backed by torch's caching allocator (device memory plumbing only).

    Keeps each returned block alive in a dict until the library frees it.
    ``fail_after`` makes the n-th call return NULL (host-side fault injection).
    """

    def __init__(self, device=0, fail_after=None):
        import torch

        self._torch = torch
        self.device = device
        self.live = {}
        self.calls = 0
        self.fail_after = fail_after
        self._alloc = ALLOC_FN(self._do_alloc)
        self._free = FREE_FN(self._do_free)
        self.struct = fp_allocator(self._alloc, self._free, None)

    def _do_alloc(self, nbytes, ctx):
        self.calls += 1
        if self.fail_after is not None and self.calls > self.fail_after:
            return None
        try:
            t = self._torch.empty(int(nbytes) + 256, dtype=self._torch.uint8, device=f"cuda:{self.device}")
        except RuntimeError:
            return None
        p = (t.data_ptr() + 255) // 256 * 256
        self.live[p] = t
        return p

    def _do_free(self, ptr, ctx):
        self.live.pop(ptr, None)


# ------------------------------------------------------------------ fp_estimate.h
def _check_est(code):
    if code < 0:
        raise FPError(int(code), "estimator: singular system (equal output lengths or layer counts) or NULL")
    return code


def fp_solve_eq1(len_a, lat_a, len_b, lat_b):
    """Eq. 1 fitted to two requests of one fingerprint -> fp_eq1_fit (ttft, tpot)."""
    out = fp_eq1_fit()
    _check_est(_lib.fp_solve_eq1(len_a, lat_a, len_b, lat_b, C.byref(out)))
    return out


def fp_solve_eq23(layers_a, fit_a, layers_b, fit_b):
    """Eqs. 2-3 from two fingerprint depths -> fp_l2_terms."""
    out = fp_l2_terms()
    _check_est(_lib.fp_solve_eq23(layers_a, C.byref(fit_a), layers_b, C.byref(fit_b), C.byref(out)))
    return out


def fp_predict_latency(terms, num_layers, output_length):
    v = C.c_double()
    _check_est(_lib.fp_predict_latency(C.byref(terms), num_layers, output_length, C.byref(v)))
    return v.value


def fp_extrapolate_memory(layers_a, mem_a, layers_b, mem_b, num_layers):
    v = C.c_double()
    _check_est(_lib.fp_extrapolate_memory(layers_a, mem_a, layers_b, mem_b, num_layers, C.byref(v)))
    return v.value
