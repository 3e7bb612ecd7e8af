"""Benchmark of the fingerprint forward pass on GB300 (one JSON line on rank 0).

A step is one request batch through the whole hot path: prefill of the
batch's prompts, then greedy decode steps (the decode step is a replayed CUDA
graph).  The default workload is the largest configuration, the
Llama-2-70B-shaped fingerprint: 2 decoder blocks (d 8192, 64 query / 8 KV
heads x 128, FFN 28672, vocab 32000), int4 group-128 weight-only
quantisation, int8 KV cache (per-token, per-head scales, 16-token pages),
batch 32, 2048-token prompts, 100 generated tokens.  Weights are synthetic
(SplitMix64 / Irwin-Hall N(0, 0.02), drawn on the device), prompts are
seeded uniform ids.  --config picks the tiny, 7B- or 13B-shaped workload.

value      decode tokens/s over all ranks = ranks * batch * decode steps / max-over-ranks
           device time of the decode phases (CUDA events on the library's stream)
e2e        decode tokens/s of whole requests through the C ABI with host buffers:
           each step uploads the prompt from pinned memory, prefills, reads the
           first token back, and runs the decode steps with every step's input
           tokens uploaded and its output tokens read back -- the prefill (TTFT)
           is inside the timed region, as in the request latency of Eq. 1
roofline   the dominant decode kernel: algorithmic bytes per launch / mean launch
           duration (CUDA events between kernels, instrumented decode steps)
cpu_baseline  the oracle (numpy, fp64) on the host cores, a bounded sample

--impl reference times the oracle alone as the reference arm.
Multi-GPU: one independent replica per rank (the path does not shard).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode tokens/s and achieved HBM GB/s per fingerprint block; prefill TFLOP/s"

# name: (n_layers, hidden, heads, kv heads, head_dim, ffn, vocab), wquant, kvquant, batch, prompt, decode
CONFIGS = {
    "tiny": ((1, 512, 8, 8, 64, 1376, 32000), 0, 0, 1, 32, 16),
    "l7b": ((2, 4096, 32, 32, 128, 11008, 32000), 1, 0, 8, 512, 100),
    "l13b": ((2, 5120, 40, 40, 128, 13824, 32000), 2, 0, 16, 1024, 100),
    "l70b": ((2, 8192, 64, 8, 128, 28672, 32000), 2, 1, 32, 2048, 100),
    # the 70B-shaped workload with GPTQ-format int4 weights (act-order groups)
    "l70b_gptq4": ((2, 8192, 64, 8, 128, 28672, 32000), 3, 1, 32, 2048, 100),
}
WQ_NAME = {0: "bf16", 1: "int8-per-channel", 2: "int4-g128", 3: "gptq4-g128-act-order"}
KV_NAME = {0: "bf16", 1: "int8-per-token-head"}


def arch_dict(t):
    keys = ("n_layers", "hidden", "n_heads", "n_kv_heads", "head_dim", "ffn", "vocab")
    d = dict(zip(keys, t))
    d.update(rms_eps=1e-5, rope_base=10000.0)
    return d


# ---------------------------------------------------------------- byte model
def mat_bytes(n, k, wq):
    """Stored bytes of one [n, k] matrix (GPTQ4: int4 plus the int32 act order)."""
    return {0: 2 * n * k, 1: n * k + 2 * n, 2: n * k // 2 + 4 * n * (k // 128),
            3: n * k // 2 + 4 * n * (k // 128) + 4 * k}[wq]


def kernel_bytes(a, wq, kvq, B, ctx):
    """Algorithmic HBM bytes of one launch of each decode kernel class:
    weight codes + scales/zeros + activations in and out (+ K/V rows read)."""
    d, f, V = a["hidden"], a["ffn"], a["vocab"]
    qd = a["n_heads"] * a["head_dim"]
    kvd = a["n_kv_heads"] * a["head_dim"]
    nqkv = qd + 2 * kvd
    kv_tok = 2 * kvd * 2 if kvq == 0 else 2 * kvd + 2 * a["n_kv_heads"] * 4
    return {
        "lin_qkv": mat_bytes(nqkv, d, wq) + 2 * B * (d + nqkv),
        "lin_o": mat_bytes(d, qd, wq) + 2 * B * (qd + 2 * d),
        "lin_gu": mat_bytes(2 * f, d, wq) + 2 * B * (d + f),
        "lin_down": mat_bytes(d, f, wq) + 2 * B * (f + 2 * d),
        "lm_head": 2 * V * d + 2 * B * d + 4 * B * V,
        "attn": B * ctx * kv_tok + 2 * B * 2 * qd,
    }


def class_roofline(cls, kb, cls_time, launches, peak):
    """GB/s and fraction of the HBM peak of one decode kernel class: its
    algorithmic bytes per launch over its mean instrumented launch time."""
    ms = cls_time[cls] / max(1, launches[cls])
    gbs = kb[cls] / (ms * 1e-3) / 1e9 if ms > 0 else 0.0
    return {"achieved": gbs, "frac": gbs / peak, "launch_ms": ms, "bytes_per_launch": kb[cls]}


# ---------------------------------------------------------------- ncu traffic
# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of the
# decode kernels from the ncu captures summarised in profiles/ (microbench
# cases of the workload's shapes), keyed by (workload, kernel class), with the
# sha256 prefix of the kernel's source code at capture time (comments and
# blank lines left out, see source_code_sha): changed code makes the figure
# stale and it is reported as null.  Attention traffic is per
# cached token row (units = B x context of the capture) and scales with the
# bench's B x context.
NCU_TRAFFIC = {
    # profiles/dram_traffic_l70b.md and dram_traffic_l7b.md: microbench cases, one launch each
    ("l70b", "lin_gu"): {"bytes": 273504512, "units": None, "src": "fp_gemv_tc.cu", "sha": "4ce5acf290c2928d"},
    ("l70b", "lin_down"): {"bytes": 130917632, "units": None, "src": "fp_gemv_tc.cu", "sha": "4ce5acf290c2928d"},
    ("l70b", "lin_qkv"): {"bytes": 45146880, "units": None, "src": "fp_gemv_tc.cu", "sha": "4ce5acf290c2928d"},
    ("l70b", "lin_o"): {"bytes": 36759552, "units": None, "src": "fp_gemv_tc.cu", "sha": "4ce5acf290c2928d"},
    ("l70b", "lm_head"): {"bytes": 533911808, "units": None, "src": "fp_gemv_btc.cu", "sha": "ac6ffae462038acd"},
    ("l70b", "attn"): {"bytes": 149513984, "units": 32 * 2148, "src": "fp_attention.cu", "sha": "011e2b422a5fa35c"},
    ("l7b", "attn"): {"bytes": 81405952, "units": 8 * 612, "src": "fp_attention.cu", "sha": "011e2b422a5fa35c"},
    ("l7b", "lm_head"): {"bytes": 270177792, "units": None, "src": "fp_linear.cu", "sha": "136661144db50e97"},
    ("l7b", "lin_gu"): {"bytes": 94035456, "units": None, "src": "fp_linear.cu", "sha": "136661144db50e97"},
    ("l7b", "lin_qkv"): {"bytes": 50459904, "units": None, "src": "fp_linear.cu", "sha": "136661144db50e97"},
    ("l7b", "lin_o"): {"bytes": 16946176, "units": None, "src": "fp_linear.cu", "sha": "136661144db50e97"},
    ("l7b", "lin_down"): {"bytes": 45368320, "units": None, "src": "fp_linear.cu", "sha": "136661144db50e97"},
}


def source_code_sha(path):
    """sha256 prefix of a C++/CUDA source with its comments, leading and
    trailing blanks and empty lines left out: an edit of the comments keeps
    it, any change of the code changes it."""
    import hashlib
    import re

    with open(path, encoding="utf-8") as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    lines = [line.strip() for line in text.splitlines()]
    return hashlib.sha256("\n".join(line for line in lines if line).encode()).hexdigest()[:16]


def ncu_traffic(cls, cfg_name, B, ctx):
    """Per-launch DRAM bytes of kernel class `cls` from the recorded capture, or None."""
    t = NCU_TRAFFIC.get((cfg_name, cls))
    if t is None:
        return None
    src = os.path.join(ROOT, "paper_2501_13111_gb300", "csrc", t["src"])
    try:
        sha = source_code_sha(src)
    except OSError:
        return None
    if sha != t["sha"]:
        return None
    return t["bytes"] if t["units"] is None else t["bytes"] * (B * ctx) / t["units"]


# ---------------------------------------------------------------- clocks
CLOCK_Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
           "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
           "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    """nvidia-smi sampling SM clocks and throttle reasons every 25 ms.  The
    timed region starts only once the first sample has arrived (so the
    samples that follow fall inside it); that first sample is kept apart and
    reported only when the region ended before the next one."""

    PERIOD_MS = 25

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.first = []
        self.lines = []

    def __enter__(self):
        for period in (self.PERIOD_MS, 200):  # 200 ms if this nvidia-smi refuses the shorter period
            if self._start(period) != "refused":
                break
        return self

    def _start(self, period):
        import select

        self.first = []
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={CLOCK_Q}", "--format=csv,noheader,nounits",
                 "-lms", str(period)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return "absent"
        # wait (at most 5 s) for the sampler's first line, reading the raw pipe
        # so that communicate() later sees every byte that follows
        fd, buf, eof = self.proc.stdout.fileno(), b"", False
        deadline = time.time() + 5.0
        while b"\n" not in buf:
            left = deadline - time.time()
            if left <= 0 or not select.select([fd], [], [], left)[0]:
                break
            chunk = os.read(fd, 4096)
            if not chunk:
                eof = True
                break
            buf += chunk
        self.first = [l for l in buf.decode(errors="replace").splitlines() if l.strip()]
        if not self.first and eof:  # it closed its output without a sample: it refused the arguments
            try:
                self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.proc.communicate()
            self.proc = None
            return "refused"
        return "ok"

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()] or self.first
        return False

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------- oracle timing
# The oracle's bounded sample of each workload: (batch, prompt) of the timed
# decode.  The full shapes and the full batch are kept; where the workload's
# prompt would make the untimed prefill set-up take minutes on the host
# (the 70B-shaped prompt is 229 TFLOP at batch 32), a short prompt stands in.
ORACLE_SAMPLE = {"tiny": (1, 32), "l7b": (8, 512), "l13b": (16, 64), "l70b": (32, 16), "l70b_gptq4": (32, 16)}


def oracle_sample(cfg, batch, prompt, steps, decode_tokens, warmup=0):
    """Time the oracle (numpy fp64, test infrastructure) on the workload's
    shapes: the full config at ``batch`` sequences with ``prompt``-token
    prompts; the prompt's prefill is set-up, each step is ``decode_tokens``
    greedy decode steps, the first ``warmup`` steps untimed.  Returns
    (tokens/s, seconds per timed step, description)."""
    from concurrent.futures import ThreadPoolExecutor

    import synth
    from oracle import model as M

    t, wq, kvq, B, S, N = cfg
    arch = M.Arch(*t)
    get = lambda l, k, shape: (synth.f32_to_bf16_bits(np.ones(shape, np.float32)) if len(shape) == 1
                               else synth.weight_bf16(0, l, k, shape))
    with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as pool:  # set-up: quantise in parallel
        w, _ = M.build_weights(arch, wq, get, map_fn=pool.map,
                               act_order=lambda l, m, k: synth.act_order(0, l, m, k))
    ref = M.Fingerprint(arch, w, kvq, batch, prompt + (warmup + steps) * decode_tokens + 1)
    toks = synth.tokens(0, batch * prompt, arch.vocab).reshape(batch, prompt)
    out = ref.prefill(toks)
    tok = out["tokens"]
    times = []
    for _ in range(warmup + steps):
        t0 = time.perf_counter()
        for _ in range(decode_tokens):
            tok = ref.decode(tok)["tokens"]
        times.append(time.perf_counter() - t0)
    times = times[warmup:]
    tps = batch * decode_tokens * steps / sum(times)
    desc = (f"oracle decode of the full {arch.n_layers}-block shape, batch {batch} of {B}, prompt {prompt} of {S} "
            f"(prefill untimed), {decode_tokens} tokens x {steps} timed steps"
            + (f" after {warmup} untimed" if warmup else "") + ", fp64 numpy")
    return tps, times, desc


def blas_threads():
    try:
        from threadpoolctl import threadpool_info

        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count()


def run_reference(args, cfg):
    """Reference arm: the oracle on the host cores (rank 0 only)."""
    if int(os.environ.get("RANK", "0")) != 0:
        return 0
    t, wq, kvq, B, S, N = cfg
    ob, op = ORACLE_SAMPLE[args.config]
    tps, times, desc = oracle_sample(cfg, ob, op, args.steps, 2, warmup=args.warmup)
    line = {
        "metric": METRIC, "value": tps, "unit": "tokens/s", "n_gpus": args.gpus, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * sum(times) / len(times), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": config_json(args, cfg),
        "cpu_baseline": {"value": tps, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle",
                         "sample": desc},
        "e2e": {"value": tps, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- replicas
# One independent fingerprint per rank (the path does not shard): the ranks
# exchange nothing but their timings.
def rank_max(x, world, device):
    """The largest of the ranks' values of x (the slowest rank's time)."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_tokens_per_s(world, batch, tokens_per_sequence, slowest_ms):
    """Whole-job decode throughput: every rank decodes batch x tokens_per_sequence
    tokens of its own replica, and the job takes as long as its slowest rank."""
    return world * batch * tokens_per_sequence / (slowest_ms * 1e-3)


def config_json(args, cfg):
    t, wq, kvq, B, S, N = cfg
    a = arch_dict(t)
    return {"workload": f"{args.config}-shaped fingerprint", "layers": a["n_layers"], "hidden": a["hidden"],
            "heads": a["n_heads"], "kv_heads": a["n_kv_heads"], "head_dim": a["head_dim"], "ffn": a["ffn"],
            "vocab": a["vocab"], "weights": WQ_NAME[wq], "kv_cache": KV_NAME[kvq], "batch": B, "prompt": S,
            "decode_tokens": N, "parallelism": f"replicas{args.gpus}",
            "l2": "inputs larger than L2 (every decode step streams all block weights and the LM head)"}


# ---------------------------------------------------------------- sweep
SWEEP_ARCH = (1, 8192, 64, 8, 128, 28672, 32000)  # the 70B-shaped block with embedding and LM head


def run_sweep(args):
    """The configuration sweep: weights x KV x batch x context on the 70B-shaped
    block, fp_profile (device events) per point; one JSON line per point."""
    import torch

    import paper_2501_13111_gb300 as fp

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    a = arch_dict(SWEEP_ARCH)
    N = 100
    for wq in (0, 1, 2):
        for kvq in (0, 1):
            for B in (1, 8, 32, 64):
                for ctx in (128, 512, 2048, 4096):
                    h = fp.fp_create(a, wq, kvq, B, ctx + N + 1, seed=0)
                    try:
                        r = fp.fp_profile(h, ctx, N, warmup=1, iters=1).as_dict()
                    finally:
                        fp.fp_destroy(h)
                    print(json.dumps({"weights": WQ_NAME[wq], "kv_cache": KV_NAME[kvq], "batch": B, "context": ctx,
                                      "decode_tokens": N, "ttft_ms": r["ttft_ms"], "tpot_ms": r["tpot_ms"],
                                      "decode_tokens_per_s": r["decode_tokens_per_s"],
                                      "peak_hbm_bytes": r["peak_hbm_bytes"],
                                      "decode_bytes_per_step": r["decode_bytes_per_step"]}), flush=True)
    return 0


# ---------------------------------------------------------------- estimator
def run_estimate(args, cfg):
    """L2 / M2 of the paper on this config: fingerprints with 1 and 2 hidden
    layers at two output lengths -> Eqs. 1-3 -> predicted request latency
    and footprint of deeper models, next to the measured ones (3, 4 and the
    full depth of the named model)."""
    import torch

    import paper_2501_13111_gb300 as fp

    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    arch, wq, kvq, B, S, N = cfg
    full = {"l7b": 32, "l13b": 40, "l70b": 80, "l70b_gptq4": 80, "tiny": 4}[args.config]
    lens = (16, 64)

    def measure(L, n, iters):
        h = fp.fp_create(arch_dict((L,) + tuple(arch[1:])), wq, kvq, B, S + N + 1, seed=0)
        try:
            r = fp.fp_profile(h, S, n, warmup=1, iters=iters)
            return r.request_ms, r.ttft_ms, r.tpot_ms, r.peak_hbm_bytes, r.observed_hbm_bytes
        finally:
            fp.fp_destroy(h)

    measure(1, lens[0], 1)  # loads every kernel once, so no reading below carries that one-time cost
    fits, mem, obs = {}, {}, {}
    for L in (1, 2):
        lat = [measure(L, n, 3) for n in lens]
        fits[L] = fp.fp_solve_eq1(lens[0], lat[0][0], lens[1], lat[1][0])
        mem[L] = lat[0][3]
        obs[L] = lat[1][4]
    t = fp.fp_solve_eq23(1, fits[1], 2, fits[2])
    rows = []
    for L in (3, 4, full):
        req, ttft, tpot, peak, seen = measure(L, N, 2)
        pred = fp.fp_predict_latency(t, L, N)
        pmem = fp.fp_extrapolate_memory(1, mem[1], 2, mem[2], L)
        pobs = fp.fp_extrapolate_memory(1, obs[1], 2, obs[2], L)
        rows.append({"layers": L, "output_length": N, "predicted_ms": pred, "measured_ms": req,
                     "rel_err": (pred - req) / req, "predicted_ttft_ms": L * t.ttft_layer + t.ttft_other,
                     "measured_ttft_ms": ttft, "predicted_tpot_ms": L * t.tpot_layer + t.tpot_other,
                     "measured_tpot_ms": tpot, "predicted_peak_hbm_bytes": pmem, "measured_peak_hbm_bytes": peak,
                     "predicted_observed_bytes": pobs, "observed_bytes": seen,
                     "observed_rel_err": (pobs - seen) / seen if seen else None})
    print(json.dumps({"config": config_json(args, cfg), "fits": {L: {"ttft_ms": f.ttft, "tpot_ms": f.tpot}
                                                                 for L, f in fits.items()},
                      "terms_ms": {"ttft_layer": t.ttft_layer, "ttft_other": t.ttft_other,
                                   "tpot_layer": t.tpot_layer, "tpot_other": t.tpot_other},
                      "checks": rows}), flush=True)
    return 0


# ---------------------------------------------------------------- our arm
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="l70b", choices=list(CONFIGS))
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle timing (profiling runs)")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end pass (profiling runs)")
    ap.add_argument("--sweep", action="store_true", help="profile the 96-point configuration sweep instead")
    ap.add_argument("--estimate", action="store_true", help="run the paper's L2/M2 estimators on --config instead")
    args = ap.parse_args()
    if args.sweep:
        return run_sweep(args)
    cfg = CONFIGS[args.config]
    if args.estimate:
        return run_estimate(args, cfg)
    if args.impl == "reference":
        return run_reference(args, cfg)

    import torch
    import torch.distributed as dist

    import paper_2501_13111_gb300 as fp

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if world > 1:
            dist.barrier()

    def max_over_ranks(x):
        return rank_max(x, world, "cuda")

    t, wq, kvq, B, S, N = cfg
    a = arch_dict(t)
    stream = torch.cuda.Stream()
    h = fp.fp_create(a, wq, kvq, B, S + N + 1, seed=0, stream=stream.cuda_stream)
    try:
        fp.fp_load_prompt(h, None, S)
        for _ in range(args.warmup):
            fp.fp_prefill(h, None, want_next=False, prompt_len=S)
            fp.fp_decode_steps(h, N)
        torch.cuda.synchronize()
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
        with ClockSampler(local) as clk:  # sampling before the barrier, so every rank's region starts together
            barrier()
            torch.cuda.synchronize()
            for k in range(args.steps):
                ev[k][0].record(stream)
                fp.fp_prefill(h, None, want_next=False, prompt_len=S)
                ev[k][1].record(stream)
                fp.fp_decode_steps(h, N)
                ev[k][2].record(stream)
            torch.cuda.synchronize()
        barrier()
        ttft = [ev[k][0].elapsed_time(ev[k][1]) for k in range(args.steps)]
        dec = [ev[k][1].elapsed_time(ev[k][2]) for k in range(args.steps)]
        total_ms = max_over_ranks(sum(ttft) + sum(dec))
        dec_ms = max_over_ranks(sum(dec))
        ttft_ms = max_over_ranks(sum(ttft) / args.steps)
        value = replica_tokens_per_s(world, B, N * args.steps, dec_ms)

        # instrumented decode steps: per-block and per-kernel device time
        prof = fp.fp_profile(h, S, N, warmup=0, iters=1).as_dict()
        mean_ctx = S + (min(N, 8) + 1) / 2.0
        kb = kernel_bytes(a, wq, kvq, B, mean_ctx)
        cls_time = {c: prof["kernel_ms"][c] for c in kb}
        dom = max(cls_time, key=cls_time.get)
        per_launch_ms = cls_time[dom] / max(1, prof["kernel_launches"][dom])
        achieved = kb[dom] / (per_launch_ms * 1e-3) / 1e9
        peaks = {}
        pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
        if os.path.exists(pk):
            peaks = json.load(open(pk))
        peak, peak_src = (peaks["hbm_gbs"], "measured") if "hbm_gbs" in peaks else (6800.0, "fallback")
        block_gbs = [bb / (bm * 1e-3) / 1e9 for bb, bm in zip(prof["block_bytes"], prof["block_ms"])]
        launches = args.steps * (prof["prefill_launches"] + N * prof["decode_launches"])

        # end to end through the C ABI with host buffers: whole requests, the
        # prompt uploaded from pinned host memory and prefilled, the first
        # token read back, then every decode step's input tokens uploaded and
        # its output tokens read back (Eq. 1's request latency, TTFT included)
        e2e = None
        if not args.no_e2e:
            pin_prompt = torch.empty((B, S), dtype=torch.int32, pin_memory=True)
            host_prompt = pin_prompt.numpy()
            import synth

            host_prompt[:] = synth.tokens(0, B * S, a["vocab"]).reshape(B, S)
            pin_in = torch.empty(B, dtype=torch.int32, pin_memory=True).numpy()
            pin_out = torch.empty(B, dtype=torch.int32, pin_memory=True).numpy()

            def host_request():
                t0 = time.perf_counter()
                fp.fp_prefill(h, host_prompt, out=pin_out)
                for _ in range(N):
                    pin_in[:] = pin_out
                    fp.fp_decode_step(h, pin_in, out=pin_out)
                return time.perf_counter() - t0

            host_request()
            barrier()
            t_req = sum(host_request() for _ in range(args.steps))
            barrier()
            t_req = max_over_ranks(t_req)
            e2e = {"value": replica_tokens_per_s(world, B, N * args.steps, 1e3 * t_req), "unit": "tokens/s",
                   "h2d_bytes_per_step": B * S * 4 + B * 4 * N, "d2h_bytes_per_step": B * 4 * (N + 1),
                   "request_ms": 1e3 * t_req / args.steps, "covers": "prompt upload + prefill + decode steps"}

        cpu = None
        if rank == 0 and world == 1 and not args.no_cpu_baseline:
            ob, op = ORACLE_SAMPLE[args.config]
            tps, times, desc = oracle_sample(cfg, ob, op, 3, 2)
            cpu = {"value": tps, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle", "sample": desc}

        if rank == 0:
            line = {
                "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
                "data": "synthetic (seeded weights and prompts)", "config": config_json(args, cfg),
                "ttft_ms": ttft_ms, "tpot_ms": dec_ms / (args.steps * N),
                "prefill_tflops": prof["prefill_flops"] / (ttft_ms * 1e-3) / 1e12,
                "block_hbm_gbs": block_gbs, "block_ms": prof["block_ms"],
                "peak_hbm_bytes": prof["peak_hbm_bytes"], "weight_bytes": prof["weight_bytes"],
                "kernel_ms_per_step": prof["kernel_ms"],
                "roofline": {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": peak,
                             "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                             "bytes_per_launch": kb[dom], "launch_ms": per_launch_ms,
                             "traffic": ncu_traffic(dom, args.config, B, mean_ctx)},
                # every decode kernel class the same way (instrumented launches, algorithmic bytes)
                "roofline_by_class": {c: class_roofline(c, kb, cls_time, prof["kernel_launches"], peak)
                                      for c in kb if prof["kernel_launches"].get(c)},
                "gpu_launches": launches,
                "clocks": clk.summary(),
                "e2e": e2e,
                "cpu_baseline": cpu,
            }
            print(json.dumps(line), flush=True)
    finally:
        fp.fp_destroy(h)
        if world > 1:
            dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
