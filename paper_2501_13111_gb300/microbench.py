"""Op-level microbenchmark of the fingerprint's kernels at the workload shapes.

Each case calls one C-ABI op entry point on device-resident inputs and times
it with CUDA events on the current stream.  Decode cases cycle over enough
copies of the weights (or KV pools) to exceed the 129 MB L2, so every launch
reads HBM; prefill GEMMs are compute-bound and run on one copy.

    python -m paper_2501_13111_gb300.microbench            # every case
    python -m paper_2501_13111_gb300.microbench --only 7b-lmhead --iters 1

With ``--only`` a case runs one copy and one timed iteration after two warm-up
calls, which is the shape a profiler capture wants (``-s 2 -c 1``).

Decode linears report GB/s of algorithmic bytes (codes + scales/zeros +
activations in and out); attention reports GB/s of cached K/V (+ int8 scales);
the prefill GEMM reports TFLOP/s of 2·M·N·K (``-inkernel`` cases: int8 / int4
weights dequantised inside the GEMM, no workspace) and prefill attention those of
both matmuls over the causal half, 2·B·H·S²·hd.  Weights and caches hold random
values: speed does not depend on them.
"""
import argparse
import json
import os

import numpy as np
import torch

import paper_2501_13111_gb300 as fp

L2_BYTES = 129 << 20


def weight_bytes(n, k, wq):
    """Codes plus scales/zeros of one [n, k] matrix (bf16, int8 per row, int4 g128)."""
    return {0: 2 * n * k, 1: n * k + 2 * n, 2: n * k // 2 + 4 * n * (k // 128)}[wq]


def timed(fn, iters, warmup=2):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ts = []
    for _ in range(iters):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        fn()
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b))
    return float(np.median(ts))


def quantized(wq, n, k):
    w = torch.randint(-3000, 3000, (n * k,), dtype=torch.int16, device="cuda")
    w = (w.to(torch.float32) * 1e-5).to(torch.bfloat16).view(torch.int16)
    codes = torch.empty(weight_bytes(n, k, 0), dtype=torch.uint8, device="cuda")
    g = max(1, k // 128)
    sc = torch.zeros(n * g, dtype=torch.int16, device="cuda")
    ze = torch.zeros(n * g, dtype=torch.int16, device="cuda")
    fp.fp_op_quantize(wq, w.data_ptr(), n, k, codes.data_ptr(), sc.data_ptr(), ze.data_ptr())
    return codes, sc, ze


def case_linear(wq, epi, M, N, K, scratch=True, *, single, iters):
    nbytes = weight_bytes(N, K, wq)
    copies = 1 if single else max(2, min(8, -(-3 * L2_BYTES // nbytes)))
    mats = [quantized(wq, N, K) for _ in range(copies)]
    x = torch.randn(M, K, device="cuda").to(torch.bfloat16)
    nout = N // 2 if epi == 2 else N
    y = torch.zeros(M * nout * 4, dtype=torch.uint8, device="cuda")
    r = torch.zeros(M * nout, dtype=torch.bfloat16, device="cuda")
    wsb = fp.fp_op_linear_workspace_bytes(wq, M, N, K) if scratch else 0
    ws = torch.zeros(max(wsb, 16), dtype=torch.uint8, device="cuda")
    wsp = ws.data_ptr() if scratch else None

    def f():
        for codes, sc, ze in mats:
            fp.fp_op_linear(wq, epi, x.data_ptr(), M, N, K, codes.data_ptr(), sc.data_ptr(), ze.data_ptr(),
                            r.data_ptr(), y.data_ptr(), wsp, wsb)

    ms = timed(f, iters) / copies
    out_elt = 4 if epi == 3 else 2
    moved = nbytes + 2 * M * K + out_elt * M * nout + (2 * M * nout if epi == 1 else 0)
    if M > 64:
        return ms, 2.0 * M * N * K / (ms * 1e-3) / 1e12, "TFLOP/s"
    return ms, moved / ms / 1e6, "GB/s"


def case_linear_gptq4(epi, M, N, K, *, single, iters):
    """GPTQ4 linear (fp_op_linear_gptq4): decode gathers x into the act order
    before the int4 linear; prefill expands the weights back into channel order."""
    nbytes = weight_bytes(N, K, 2) + 4 * K
    copies = 1 if single else max(2, min(8, -(-3 * L2_BYTES // nbytes)))
    perm = torch.randperm(K, device="cuda").to(torch.int32)
    mats = []
    for _ in range(copies):
        w = torch.randint(-3000, 3000, (N * K,), dtype=torch.int16, device="cuda")
        w = (w.to(torch.float32) * 1e-5).to(torch.bfloat16).view(torch.int16)
        codes = torch.empty(N * K // 2, dtype=torch.uint8, device="cuda")
        sc = torch.zeros(N * (K // 128), dtype=torch.int16, device="cuda")
        ze = torch.zeros(N * (K // 128), dtype=torch.int16, device="cuda")
        fp.fp_op_quantize_gptq4(w.data_ptr(), N, K, perm.data_ptr(), codes.data_ptr(), sc.data_ptr(), ze.data_ptr())
        mats.append((codes, sc, ze))
    x = torch.randn(M, K, device="cuda").to(torch.bfloat16)
    nout = N // 2 if epi == 2 else N
    y = torch.zeros(M * nout * 4, dtype=torch.uint8, device="cuda")
    r = torch.zeros(M * nout, dtype=torch.bfloat16, device="cuda")
    wsb = fp.fp_op_linear_gptq4_workspace_bytes(M, N, K)
    ws = torch.zeros(max(wsb, 256), dtype=torch.uint8, device="cuda")

    def f():
        for codes, sc, ze in mats:
            fp.fp_op_linear_gptq4(epi, x.data_ptr(), M, N, K, perm.data_ptr(), codes.data_ptr(), sc.data_ptr(),
                                  ze.data_ptr(), r.data_ptr(), y.data_ptr(), ws.data_ptr(), wsb)

    ms = timed(f, iters) / copies
    moved = nbytes + 2 * M * K + 2 * M * nout + (2 * M * nout if epi == 1 else 0)
    if M > 64:
        return ms, 2.0 * M * N * K / (ms * 1e-3) / 1e12, "TFLOP/s"
    return ms, moved / ms / 1e6, "GB/s"


def case_attention(B, H, Hkv, hd, ctx, kvq, single, iters):
    P = 16
    pps = -(-ctx // P)
    npg = B * pps
    elt = 2 if kvq == 0 else 1
    pool = npg * Hkv * P * hd * elt
    copies = 1 if single else max(2, min(8, -(-3 * L2_BYTES // (2 * pool))))
    sets = []
    for _ in range(copies):
        if kvq == 0:
            kp = (torch.randn(pool // 2, device="cuda") * 0.5).to(torch.bfloat16)
            vp = (torch.randn(pool // 2, device="cuda") * 0.5).to(torch.bfloat16)
        else:
            kp = torch.randint(-100, 100, (pool,), dtype=torch.int8, device="cuda")
            vp = torch.randint(-100, 100, (pool,), dtype=torch.int8, device="cuda")
        ks = torch.rand(npg * Hkv * P, device="cuda") * 0.01
        vs = torch.rand(npg * Hkv * P, device="cuda") * 0.01
        pt = torch.randperm(npg, device="cuda").to(torch.int32)
        kv = fp.fp_kv_view(kvq, Hkv, hd, P, pps, npg, kp.data_ptr(), vp.data_ptr(),
                           ks.data_ptr() if kvq else None, vs.data_ptr() if kvq else None, pt.data_ptr())
        sets.append((kp, vp, ks, vs, pt, kv))
    q = torch.randn(B, H * hd, device="cuda").to(torch.bfloat16)
    lens = torch.full((B,), ctx, dtype=torch.int32, device="cuda")
    out = torch.empty(B * H * hd, dtype=torch.bfloat16, device="cuda")
    wsb = fp.fp_op_attention_decode_workspace_bytes(B, H, hd, ctx)
    ws = torch.zeros(max(wsb, 16), dtype=torch.uint8, device="cuda")

    def f():
        for st in sets:
            fp.fp_op_attention_decode(q.data_ptr(), H * hd, B, H, st[5], lens.data_ptr(), ctx, out.data_ptr(),
                                      ws.data_ptr(), wsb)

    ms = timed(f, iters) / copies
    moved = B * ctx * Hkv * hd * elt * 2 + (B * ctx * Hkv * 8 if kvq else 0)
    return ms, moved / ms / 1e6, "GB/s"


def case_attention_prefill(B, H, Hkv, hd, S, kvq, single, iters):
    P = 16
    pps = -(-S // P)
    npg = B * pps
    elt = 2 if kvq == 0 else 1
    pool = npg * Hkv * P * hd * elt
    if kvq == 0:
        kp = (torch.randn(pool // 2, device="cuda") * 0.5).to(torch.bfloat16)
        vp = (torch.randn(pool // 2, device="cuda") * 0.5).to(torch.bfloat16)
    else:
        kp = torch.randint(-100, 100, (pool,), dtype=torch.int8, device="cuda")
        vp = torch.randint(-100, 100, (pool,), dtype=torch.int8, device="cuda")
    ks = torch.rand(npg * Hkv * P, device="cuda") * 0.01
    vs = torch.rand(npg * Hkv * P, device="cuda") * 0.01
    pt = torch.randperm(npg, device="cuda").to(torch.int32)
    kv = fp.fp_kv_view(kvq, Hkv, hd, P, pps, npg, kp.data_ptr(), vp.data_ptr(),
                       ks.data_ptr() if kvq else None, vs.data_ptr() if kvq else None, pt.data_ptr())
    q = torch.randn(B * S, H * hd, device="cuda").to(torch.bfloat16)
    out = torch.empty(B * S * H * hd, dtype=torch.bfloat16, device="cuda")

    def f():
        fp.fp_op_attention_prefill(q.data_ptr(), H * hd, B, S, H, kv, out.data_ptr())

    ms = timed(f, iters)
    flops = 2.0 * B * H * S * S * hd  # both matmuls over the causal half
    return ms, flops / (ms * 1e-3) / 1e12, "TFLOP/s"


def case_argmax(M, V, single, iters):
    copies = 1 if single else 8
    logits = [torch.randn(M, V, device="cuda") for _ in range(copies)]
    out = torch.empty(M, dtype=torch.int32, device="cuda")

    def f():
        for lg in logits:
            fp.fp_op_argmax(lg.data_ptr(), M, V, out.data_ptr())

    ms = timed(f, iters) / copies
    return ms, 4 * M * V / ms / 1e6, "GB/s"


# name -> (kind, args).  Shapes are the Llama-2 7B / 13B / 70B blocks of the
# three workloads at their decode batch (8 / 16 / 32) and prefill M = B·S.
CASES = {}
for tag, (wq, d, H, Hkv, f, Mdec) in {"7b": (1, 4096, 32, 32, 11008, 8), "13b": (2, 5120, 40, 40, 13824, 16),
                                       "70b": (2, 8192, 64, 8, 28672, 32)}.items():
    nqkv = (H + 2 * Hkv) * 128
    CASES[f"{tag}-qkv"] = ("linear", (wq, 0, Mdec, nqkv, d))
    CASES[f"{tag}-o"] = ("linear", (wq, 1, Mdec, d, H * 128))
    CASES[f"{tag}-gu"] = ("linear", (wq, 2, Mdec, 2 * f, d))
    CASES[f"{tag}-down"] = ("linear", (wq, 1, Mdec, d, f))
    CASES[f"{tag}-lmhead"] = ("linear", (0, 3, Mdec, 32000, d))
    CASES[f"{tag}-argmax"] = ("argmax", (Mdec, 32000))
# the 70B-shaped block's linears with int8 weights at the 70B decode batch
for _tag, (_epi, _n, _k) in {"qkv": (0, 10240, 8192), "o": (1, 8192, 8192), "gu": (2, 57344, 8192),
                             "down": (1, 8192, 28672)}.items():
    CASES[f"70b-i8-{_tag}"] = ("linear", (1, _epi, 32, _n, _k))
    CASES[f"70b-i8-{_tag}-b64"] = ("linear", (1, _epi, 64, _n, _k))
CASES["7b-attn"] = ("attention", (8, 32, 32, 128, 612, 0))
CASES["13b-attn"] = ("attention", (16, 40, 40, 128, 1124, 0))
CASES["70b-attn"] = ("attention", (32, 64, 8, 128, 2148, 1))
CASES["7b-attn-prefill"] = ("attention_prefill", (8, 32, 32, 128, 512, 0))
CASES["13b-attn-prefill"] = ("attention_prefill", (16, 40, 40, 128, 1024, 0))
CASES["70b-attn-prefill"] = ("attention_prefill", (32, 64, 8, 128, 2048, 1))
CASES["7b-qkv-prefill"] = ("linear", (1, 0, 4096, 12288, 4096))
CASES["7b-gu-prefill"] = ("linear", (1, 2, 4096, 22016, 4096))
CASES["7b-down-prefill"] = ("linear", (1, 1, 4096, 4096, 11008))
CASES["13b-gu-prefill"] = ("linear", (2, 2, 16384, 27648, 5120))
CASES["70b-qkv-prefill"] = ("linear", (2, 0, 65536, 10240, 8192))
CASES["70b-gu-prefill"] = ("linear", (2, 2, 65536, 57344, 8192))
CASES["70b-down-prefill"] = ("linear", (2, 1, 65536, 8192, 28672))
CASES["bf16-8k-prefill"] = ("linear", (0, 0, 8192, 8192, 8192))
# the 70B-shaped block's linears with GPTQ4 weights, decode (M 32) and prefill
for _tag, (_epi, _n, _k) in {"qkv": (0, 10240, 8192), "o": (1, 8192, 8192), "gu": (2, 57344, 8192),
                             "down": (1, 8192, 28672)}.items():
    CASES[f"70b-gptq4-{_tag}"] = ("linear_gptq4", (_epi, 32, _n, _k))
CASES["70b-gptq4-gu-prefill"] = ("linear_gptq4", (2, 65536, 57344, 8192))
# the same quantised prefill linears without a workspace: dequantised inside the GEMM
for _name in ["7b-qkv-prefill", "7b-gu-prefill", "7b-down-prefill", "13b-gu-prefill", "70b-qkv-prefill",
              "70b-gu-prefill", "70b-down-prefill"]:
    CASES[_name + "-inkernel"] = ("linear", CASES[_name][1] + (False,))

RUNNERS = {"linear": case_linear, "linear_gptq4": case_linear_gptq4, "attention": case_attention,
           "attention_prefill": case_attention_prefill, "argmax": case_argmax}


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--only", default=None, help="run one case (single copy, for a profiler capture)")
    ap.add_argument("--cases", default=None, help="comma-separated cases to run (L2-defeating copies)")
    ap.add_argument("--iters", type=int, default=10)
    ap.add_argument("--json", default=None, help="write the results here")
    ap.add_argument("--list", action="store_true")
    args = ap.parse_args(argv)
    if args.list:
        for k, (kind, a) in CASES.items():
            print(k, kind, a)
        return
    torch.cuda.set_device(0)
    names = [args.only] if args.only else (args.cases.split(",") if args.cases else list(CASES))
    res = {}
    for name in names:
        kind, a = CASES[name]
        ms, rate, unit = RUNNERS[kind](*a, single=args.only is not None, iters=args.iters)
        res[name] = {"us": ms * 1e3, "rate": rate, "unit": unit}
        print(f"{name:18s} {kind:9s} {str(a):38s} {ms * 1e3:9.1f} us {rate:9.1f} {unit}", flush=True)
        torch.cuda.empty_cache()
    if args.json:
        os.makedirs(os.path.dirname(os.path.abspath(args.json)), exist_ok=True)
        with open(args.json, "w") as fh:
            json.dump(res, fh, indent=1)


if __name__ == "__main__":
    main()
