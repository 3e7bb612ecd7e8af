"""The C ABI library loads and exports every function include/*.h declares;
host-side argument checks answer without a GPU (no compute call is made)."""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for hdr in sorted(f for f in os.listdir(os.path.join(ROOT, "include")) if f.endswith(".h")):
        src = open(os.path.join(ROOT, "include", hdr)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w\s\*]*?\b(fp_\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return names


@pytest.fixture(scope="module")
def fp():
    import __graft_entry__

    __graft_entry__.build()
    import paper_2501_13111_gb300 as fp

    return fp


def test_every_declared_symbol_is_exported(fp):
    import ctypes

    names = _declared()
    assert len(names) >= 20
    lib = ctypes.CDLL(fp.LIB_PATH)
    for n in sorted(names):
        assert hasattr(lib, n), n
    # the binding covers the same names
    assert set(fp.EXPORTED) == names


def _arch(**kw):
    a = dict(n_layers=1, hidden=512, n_heads=8, n_kv_heads=8, head_dim=64, ffn=1376, vocab=32000, rms_eps=1e-5,
             rope_base=1e4)
    a.update(kw)
    return a


@pytest.mark.parametrize("kw,wq,code", [
    (dict(head_dim=96), 0, -2),
    (dict(n_heads=8, n_kv_heads=3), 0, -1),
    (dict(n_layers=81), 0, -2),
    (dict(hidden=520), 0, -2),
    (dict(ffn=1376), 2, -2),   # int4 needs ffn % 128
    (dict(ffn=1376), 3, -2),   # so does GPTQ4
    (dict(n_heads=32, n_kv_heads=2), 0, -2),  # group of 16 is not built
    (dict(vocab=0), 0, -1),
])
def test_create_rejects_bad_shapes_on_host(fp, kw, wq, code):
    with pytest.raises(fp.FPError) as e:
        fp.fp_create(_arch(**kw), wq, 0, 1, 64)
    assert e.value.code == code


def test_create_rejects_bad_modes_on_host(fp):
    for args in [(_arch(), 4, 0, 1, 64), (_arch(), 0, 2, 1, 64), (_arch(), 0, 0, 0, 64), (_arch(), 0, 0, 1, 0)]:
        with pytest.raises(fp.FPError) as e:
            fp.fp_create(*args)
        assert e.value.code == fp.FP_ERR_INVALID_ARG
    with pytest.raises(fp.FPError) as e:
        fp.fp_create(_arch(), 0, 0, 1, 64, page_size=32)
    assert e.value.code == fp.FP_ERR_UNSUPPORTED


def test_op_argument_checks_on_host(fp):
    assert fp._lib.fp_op_linear(0, 0, None, 1, 8, 8, None, None, None, None, None, None, 0, None) == -1
    assert fp._lib.fp_op_linear(5, 0, 1, 1, 8, 8, 1, 1, 1, None, 1, None, 0, None) == -1
    # int4 needs K % 128
    assert fp._lib.fp_op_linear(2, 0, 1, 1, 8, 64, 1, 1, 1, None, 1, None, 0, None) == -2
    # GPTQ4: the act order is required, K % 128, a workspace
    assert fp._lib.fp_op_linear_gptq4(0, 1, 1, 8, 128, None, 1, 1, 1, None, 1, 1, 1 << 20, None, None) == -1
    assert fp._lib.fp_op_linear_gptq4(0, 1, 1, 8, 64, 1, 1, 1, 1, None, 1, 1, 1 << 20, None, None) == -2
    assert fp._lib.fp_op_linear_gptq4(0, 1, 1, 8, 128, 1, 1, 1, 1, None, 1, None, 0, None, None) == -1
    assert fp._lib.fp_op_quantize_gptq4(1, 8, 128, None, 1, 1, 1, None) == -1
    assert fp._lib.fp_op_quantize_gptq4(1, 8, 64, 1, 1, 1, 1, None) == -2
    assert fp._lib.fp_op_quantize(2, 1, 4, 100, 1, 1, 1, None) == -2
    assert fp._lib.fp_op_rmsnorm(1, 1, 12, 1, 0, 1, 1e-5, 1, None) == -2
    kv = fp.fp_kv_view(0, 2, 96, 16, 4, 8, 1, 1, None, None, 1)
    assert fp.fp_op_attention_decode_workspace_bytes(2, 4, 128, 100) > 0
    import ctypes
    assert fp._lib.fp_op_attention_prefill(1, 1024, 1, 4, 4, ctypes.byref(kv), 1, None, None) == -2
    assert fp.fp_strerror(-5) == "KV cache capacity exceeded"


def test_empty_inputs_are_no_ops(fp):
    """Zero rows, sequences or tokens: every op returns success without
    launching anything (this runs with no GPU at all)."""
    import ctypes

    L = fp._lib
    kv = fp.fp_kv_view(0, 2, 128, 16, 4, 8, 1, 1, None, None, 1)
    assert L.fp_op_attention_prefill(1, 1024, 0, 4, 4, ctypes.byref(kv), 1, None, None) == 0  # B = 0
    assert L.fp_op_attention_prefill(1, 1024, 2, 0, 4, ctypes.byref(kv), 1, None, None) == 0  # S = 0
    assert L.fp_op_attention_decode(1, 1024, 0, 4, ctypes.byref(kv), 1, 64, 1, None, 0, None, None) == 0
    assert L.fp_op_rope_kv(1, 0, 4, 1536, 4, ctypes.byref(kv), 1, 1, None, None) == 0
    assert L.fp_op_linear(1, 0, 1, 0, 128, 128, 1, 1, None, None, 1, None, 0, None) == 0
    assert L.fp_op_rmsnorm(1, 0, 128, 128, 0, 1, ctypes.c_float(1e-5), 1, None) == 0
    assert L.fp_op_embed(1, 0, 1, 32000, 128, 1, None, None) == 0
    assert L.fp_op_argmax(1, 0, 32000, 1, None) == 0
    assert L.fp_op_quantize(1, 1, 0, 128, 1, 1, None, None) == 0


def test_kernels_have_no_unbounded_waits_or_traps():
    """Static check of the CUDA sources: no kernel can hang or trap the GPU
    by construction.  mbarrier polling lives only in the bounded helpers of
    tc.cuh (a fixed number of try_wait rounds, then the caller records an
    error and leaves); there are no open-ended loops, no __trap() and no
    device-side assert()."""
    csrc = os.path.join(ROOT, "paper_2501_13111_gb300", "csrc")
    bad = []
    for name in sorted(os.listdir(csrc)):
        if not name.endswith((".cu", ".cuh")):
            continue
        src = open(os.path.join(csrc, name)).read()
        for pat in (r"while\s*\(\s*(true|1)\s*\)", r"for\s*\(\s*;\s*;\s*\)", r"__trap\s*\(", r"(?<![\w_])assert\s*\("):
            for m in re.finditer(pat, src):
                bad.append((name, src[: m.start()].count("\n") + 1, m.group(0)))
        if name != "tc.cuh" and "try_wait" in src:
            bad.append((name, 0, "mbarrier try_wait outside the bounded helpers"))
    assert not bad, bad
    tc = open(os.path.join(csrc, "tc.cuh")).read()
    assert "kTcSpinLimit" in tc and tc.count("for (long long it = 0; it < kTcSpinLimit; ++it)") == tc.count("mbarrier.try_wait")


def test_binding_struct_layouts_match_the_headers(fp, tmp_path):
    """The ctypes mirrors of the ABI structs have the C compiler's sizes and
    field offsets (a C program built against include/*.h prints them)."""
    import ctypes
    import shutil
    import subprocess

    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    structs = [fp.fp_arch, fp.fp_allocator, fp.fp_profile_result, fp.fp_plan, fp.fp_kv_view, fp.fp_eq1_fit,
               fp.fp_l2_terms]
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "fp.h"', '#include "fp_ops.h"',
             '#include "fp_estimate.h"', "int main(void) {"]
    for st in structs:
        n = st.__name__
        lines.append(f'  printf("{n} sizeof %zu\\n", sizeof({n}));')
        for fname, _ in st._fields_:
            lines.append(f'  printf("{n} {fname} %zu\\n", offsetof({n}, {fname}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    subprocess.run([cc, "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    want = {}
    for line in out:
        if line.strip():
            name, field, val = line.split()
            want[(name, field)] = int(val)
    for st in structs:
        n = st.__name__
        assert want[(n, "sizeof")] == ctypes.sizeof(st), n
        for fname, _ in st._fields_:
            assert want[(n, fname)] == getattr(st, fname).offset, (n, fname)


def test_forward_kernels_wait_for_their_predecessor():
    """Kernels of the forward pass are launched with programmatic dependent
    launch, so each must execute pdl_wait() before it reads or writes
    activations; a missing wait is a race.  Static check of the sources: every
    __global__ kernel outside the weight set-up calls pdl_wait()."""
    csrc = os.path.join(ROOT, "paper_2501_13111_gb300", "csrc")
    setup_only = {"init_weights_kernel", "quantize_int8_kernel", "quantize_int4_kernel"}
    missing = []
    for name in os.listdir(csrc):
        if not name.endswith(".cu"):
            continue
        src = open(os.path.join(csrc, name)).read()
        for m in re.finditer(r"__global__\s+void\s+(?:__launch_bounds__\([^)]*\)\s+)?(\w+)\s*\(", src):
            kname = m.group(1)
            if kname in setup_only:
                continue
            body_start = src.index("{", m.end())
            depth, i = 0, body_start
            while True:
                depth += {"{": 1, "}": -1}.get(src[i], 0)
                if depth == 0:
                    break
                i += 1
            if "pdl_wait()" not in src[body_start:i]:
                missing.append(f"{name}:{kname}")
    assert not missing, missing


def test_binding_constants_match_the_headers(fp):
    """Constants the binding restates (the no-allocation scratch limit, the
    layer cap) equal the header macros they copy."""
    src = open(os.path.join(ROOT, "include", "fp_ops.h")).read() + open(os.path.join(ROOT, "include", "fp.h")).read()
    m = re.search(r"#define\s+FP_NOALLOC_SCRATCH_BYTES\s+\((\d+)u\s*<<\s*(\d+)\)", src)
    assert m, "FP_NOALLOC_SCRATCH_BYTES not found"
    assert fp.FP_NOALLOC_SCRATCH_BYTES == int(m.group(1)) << int(m.group(2))
    m = re.search(r"#define\s+FP_MAX_LAYERS\s+(\d+)", src)
    assert fp.FP_MAX_LAYERS == int(m.group(1))


def test_decode_splits_query_answers_on_host(fp):
    """The split count is host arithmetic (no GPU call): one split for a short
    context, several for the 70B-shaped decode attention."""
    assert fp.fp_op_attention_decode_splits(0, 8, 128, 1, 100) == 0
    assert fp.fp_op_attention_decode_splits(1, 1, 128, 0, 10) == 1
    assert fp.fp_op_attention_decode_splits(2, 8, 128, 1, 2155) > 1
    # the 70B-shaped decode: 256 (sequence, KV head) pairs fill the GPU, one split
    assert fp.fp_op_attention_decode_splits(32, 8, 128, 1, 2149) == 1
