"""Throughput of the joint next-k-token decode step on one GB300 (per rank).

A bench "step" is one full generation of the workload: every sequence of
the batch decodes gen_len tokens from its prefilled prompt (gen_len / k
calls of kf_decode_step, after kf_rewind restores the prefilled state).
``value`` = generated tokens / second over all ranks with inputs resident in
HBM; ``e2e`` = the same through the C ABI with host noise and host tokens,
host<->device copies inside the timed region.  The k = 1 AR teacher step
(kf_decode_step with k = 0) is measured the same way for the speedup.

Default workload: the LM1B-shaped model (12 L, d 768, 12 heads, MLP 3072,
V 30522, bf16), batch 64, prompt 32 -> 128, k = 4 vs the AR step.
``--impl reference`` times the CPU oracle on a bounded sample instead.
Launch with torchrun for N > 1: each rank runs an independent replica.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "generated tokens/s per GB300 at k=4 vs k=1, batch 1–512; % of roofline"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="kforcing", choices=["kforcing", "reference"])
    p.add_argument("--workload", default="lm1b")
    p.add_argument("--batch", type=int, default=0)
    p.add_argument("--k", type=int, default=4)
    p.add_argument("--gen", type=int, default=0, help="tokens per sequence (0: workload)")
    p.add_argument("--no-cpu", action="store_true", help="skip the cpu_baseline leg")
    p.add_argument("--no-ar", action="store_true", help="skip the k=1 AR leg")
    p.add_argument("--train-attention", action="store_true",
                   help="SingleForward / DoubleForward training attention (App. C.2)")
    p.add_argument("--serving", action="store_true",
                   help="the G* teacher call and continuous batching (LM1B, batch 64)")
    p.add_argument("--sweep-only", default="",
                   help="comma-separated workload names: run only these sweep configurations")
    p.add_argument("--sweep", action="store_true",
                   help="one line per configuration: OWT-shaped batch 1..256, OWT paged "
                        "batch 512, medium batch 256 (k vs the AR step)")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


def max_over_ranks(x: float, dist) -> float:
    """Largest value of x over all ranks (the slowest rank's time)."""
    if dist is None:
        return x
    import torch
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def dist_init(n):
    import torch
    if n <= 1 or "RANK" not in os.environ:
        return 0, 1, None
    import torch.distributed as dist
    rank = int(os.environ["RANK"])
    local = int(os.environ.get("LOCAL_RANK", rank))
    torch.cuda.set_device(local)
    dist.init_process_group("nccl")
    return rank, dist.get_world_size(), dist


# ------------------------------------------------------------------ roofline
def kind_costs(model, B, P, k, ctx_lens):
    """Algorithmic bytes and flops per launch of each kernel kind for one
    decode call of shape (B, P, k) whose sequences have ctx_lens cached."""
    d, F, V, H = model.d_model, model.d_ff, model.vocab, model.n_head
    hd = d // H
    e = 2 if model.dtype == "bf16" else 4
    kz = 1 if (getattr(model, "mtp_k", 0) and k) else k     # noise rows per sequence
    R = B * (P + kz)
    nh = B * max(k, 1)
    nchunk = -(-V // 32)

    def gemm(M, N, K, out_bytes):
        return {"bytes": N * K * e + M * K * e + out_bytes, "flops": 2.0 * M * N * K}
    keys = sum(int(c) + P + kz for c in ctx_lens)
    vis = sum(sum(int(c) + i + 1 for i in range(P + kz)) for c in ctx_lens)
    head = gemm(nh, V, d, nh * nchunk * 16)
    if kz != k:        # MTP: k heads over B rows
        head = {"bytes": k * V * d * e + B * d * e + nh * nchunk * 16, "flops": 2.0 * nh * V * d}
    return {
        "gemm_qkv": gemm(R, 3 * d, d, R * 3 * d * e),
        "gemm_o": gemm(R, d, d, 2 * R * d * 4),
        "gemm_up": gemm(R, F, d, R * F * e),
        "gemm_down": gemm(R, d, F, 2 * R * d * 4),
        "gemm_head": head,
        "attention": {"bytes": keys * H * hd * 2 * e + R * d * 4 + R * d * e,
                      "flops": 4.0 * vis * H * hd},
    }


def step_bytes_flops(model, B, P, k, ctx_lens):
    """Algorithmic bytes/flops of one decode call (weights once, KV once)."""
    d, F, V, L, H = model.d_model, model.d_ff, model.vocab, model.n_layer, model.n_head
    e = 2 if model.dtype == "bf16" else 4
    mtp = bool(getattr(model, "mtp_k", 0) and k)
    kz = 1 if mtp else k                           # noise rows per sequence
    ne_in = k * d if mtp else d                    # NoiseEnc input width
    heads = k if mtp else 1
    w = L * (4 * d * d + 2 * d * F) * e + heads * V * d * e + \
        ((model.ne_hidden * ne_in + model.ne_hidden * d) * e if k else 0)
    kv_tok = 2 * L * d * e
    byt = w + sum(int(c) for c in ctx_lens) * kv_tok + B * (P + kz) * kv_tok
    R = B * (P + kz)
    fl = 2.0 * R * L * (4 * d * d + 2 * d * F) + 2.0 * B * max(k, 1) * V * d + \
        (2.0 * B * kz * model.ne_hidden * (ne_in + d) if k else 0) + \
        4.0 * L * d * sum(sum(int(c) + i + 1 for i in range(P + kz)) for c in ctx_lens)
    return byt, fl


# ------------------------------------------------------------------ clocks
class Clocks:
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                p = [x.strip() for x in line.split(",")]
                if len(p) >= 8:
                    rows.append(p)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if "Active" in r[4 + i]
                          and "Not" not in r[4 + i]})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


# ------------------------------------------------------------------ CPU oracle
def cpu_oracle_rate(model, w, prompts, k, budget_s=12.0, max_calls=6):
    """Oracle tokens/s over a bounded sample: decode calls on the given
    prompts until the time budget is spent."""
    import oracle
    from synth import make_noise
    dec = oracle.OracleDecoder(oracle.OracleModel(model, w))
    dec.prefill(prompts)
    B = len(prompts)
    zs = make_noise(max_calls, B, k)
    toks, t0, calls = 0, time.perf_counter(), 0
    while calls < max_calls and time.perf_counter() - t0 < budget_s:
        dec.step(k, zs[calls])
        toks += B * max(k, 1)
        calls += 1
    el = time.perf_counter() - t0
    return toks / el, calls, el


def cpu_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads") for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count()


# ------------------------------------------------------------------ main
def bench_config(w, B, gen, k):
    """The `config` object of the bench line (both arms)."""
    model = w.model
    return {"workload": f"{w.name}: {model.n_layer}L d{model.d_model} H{model.n_head} "
                        f"F{model.d_ff} V{model.vocab}, batch {B}, prompt "
                        f"{w.prompt_len or 'ragged'} +{gen} tokens, k={k}",
            "batch": B, "k": k, "gen_tokens_per_seq": gen,
            "calls_per_step": -(-gen // max(k, 1)), "map": model.map,
            "l2": "working set larger than L2 (weights + KV), no flush"}


def workload_of(args):
    from synth import WORKLOADS
    w = WORKLOADS[args.workload]
    B = args.batch or w.batch
    gen = args.gen or w.gen_len
    return w, B, gen


def run_reference(args):
    """The reference arm: the CPU oracle, as it stands, on the same workload."""
    from synth import make_weights, workload_prompts
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w, B, gen = workload_of(args)
    model = w.model
    weights = make_weights(model)
    Bs = min(B, 16)
    prompts = workload_prompts(w, Bs)
    rates = []
    for _ in range(max(1, args.warmup and 1)):
        cpu_oracle_rate(model, weights, prompts, args.k, budget_s=5.0, max_calls=2)
    t_all = time.perf_counter()
    for _ in range(args.steps):
        r, calls, el = cpu_oracle_rate(model, weights, prompts, args.k, budget_s=10.0, max_calls=24)
        rates.append(r)
    el = time.perf_counter() - t_all
    v = statistics.median(rates)
    sample = f"{Bs} sequences x decode calls of k={args.k} for up to 10 s per step (prompt {w.prompt_len})"
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000 * el / max(1, args.steps), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": bench_config(w, B, gen, args.k),
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cpu_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def measured_traffic(kind, workload, B, k):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) of
    the dominant kernel from the committed ncu capture of the LM1B batch-64
    k=4 step, or None when the workload differs or the kernel's sources have
    changed since the capture (checked by SHA-256)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "ncu_dram_traffic_lm1b_b64_k4.json")
    if not (workload == "lm1b" and B == 64 and k == 4 and os.path.exists(path)):
        return None
    with open(path) as f:
        rec = json.load(f)
    if rec.get("kind") != kind:
        return None
    for src, digest in rec.get("sources_sha256", {}).items():
        fp = os.path.join(ROOT, src)
        if not os.path.exists(fp) or hashlib.sha256(open(fp, "rb").read()).hexdigest() != digest:
            return None
    return rec["dram_bytes_per_launch"]


SWEEP = [  # (workload, batch, ks) -- the non-headline configurations
    ("owt", 1, (4, 2, 1)), ("owt", 8, (4, 2, 1)), ("owt", 32, (4, 2, 1)),
    ("owt", 128, (4, 2, 1)), ("owt", 256, (4, 2, 1)),
    ("owt_paged", 512, (4, 1)),
    ("medium", 256, (8, 4, 1)),
    ("lm1b_mtp", 64, (4, 1)),
]


def run_sweep(args):
    """Tokens/s of full generations per configuration, k vs the AR step, with
    the step roofline fraction; one JSON line each (rank 0, N = 1)."""
    import torch
    from paper_2606_10820_gb300 import build as kbuild
    from paper_2606_10820_gb300 import kforcing as kf
    from synth import WORKLOADS, make_weights, workload_prompts
    kbuild.build()
    kf.load_library()
    pk, peak_src = peaks()
    by_wl = {}
    only = [x for x in args.sweep_only.split(",") if x]
    for name, B, ks in SWEEP:
        if not only or name in only:
            by_wl.setdefault(name, []).append((B, ks))
    for name, runs in by_wl.items():
        w = WORKLOADS[name]
        model = w.model
        weights = make_weights(model)
        maxB = max(B for B, _ in runs)
        maxk = max(max(ks) for _, ks in runs)
        stream = torch.cuda.Stream()
        dec = kf.Decoder(model, weights, max_batch=maxB, max_k=maxk, stream=stream.cuda_stream)
        del weights
        for B, ks in runs:
            prompts = workload_prompts(w, B)
            dec.prefill(prompts)
            gen = w.gen_len
            res = {}
            for k in ks:
                kk = 0 if k == 1 else k          # k=1 is the AR teacher step
                nout = max(kk, 1)
                calls = -(-gen // nout)
                z = torch.rand((calls, B, nout), device="cuda")
                o = torch.zeros((calls, B, nout), dtype=torch.int32, device="cuda")

                def one():
                    dec.rewind()
                    for i in range(calls):
                        kf.kf_decode_step(dec.ctx, B, kk, z[i], o[i])
                for _ in range(max(1, args.warmup)):
                    one()
                torch.cuda.synchronize()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for _ in range(args.steps):
                    one()
                e1.record(stream)
                torch.cuda.synchronize()
                ms = e0.elapsed_time(e1) / args.steps
                t_roof = 0.0
                for i in range(calls):
                    P = 1 if i == 0 else nout
                    lens = np.array([len(p) - 1 + (0 if i == 0 else 1 + (i - 1) * nout) for p in prompts])
                    byt, fl = step_bytes_flops(model, B, P, kk, lens)
                    t_roof += max(byt / (pk["hbm_gbs"] * 1e9), fl / (pk["bf16_tflops_sustained"] * 1e12))
                res[k] = {"value": B * calls * nout / (ms / 1e3), "ms_per_step": ms,
                          "step_roofline_frac": t_roof * 1e3 / ms}
            kmax = max(ks)
            line = {"metric": METRIC, "value": res[kmax]["value"], "unit": "tokens/s", "n_gpus": 1,
                    "steps": args.steps, "warmup": args.warmup,
                    "ms_per_step": res[kmax]["ms_per_step"], "higher_is_better": True,
                    "scaling": "weak", "vs_baseline": None, "dtype": model.dtype,
                    "data": "synthetic", "sweep": True,
                    "config": {"workload": f"{name}: {model.n_layer}L d{model.d_model} V{model.vocab}, "
                                           f"batch {B}, prompt {w.prompt_len or list(w.ragged)} +{gen}",
                               "batch": B, "k": kmax},
                    "per_k": {str(k): {kk_: round(v, 4) for kk_, v in r.items()} for k, r in res.items()},
                    "speedup_vs_k1": {str(k): res[k]["value"] / res[1]["value"] for k in ks if 1 in res},
                    "peak_source": peak_src}
            print(json.dumps(line), flush=True)
        dec.close()
        del dec
        torch.cuda.empty_cache()
    return 0


def run_serving(args):
    """The serving entry points on the LM1B-shaped model, batch 64 (rank 0, N = 1):
    the G* teacher call (k AR steps in one graph) against k separate AR calls,
    and continuous batching: every finished sequence is replaced by a new
    request at the step boundary (kf_admit), pages recycled; throughput
    counts the requests' generated tokens and includes the admissions."""
    import torch
    from paper_2606_10820_gb300 import build as kbuild
    from paper_2606_10820_gb300 import kforcing as kf
    from synth import WORKLOADS, make_requests, make_weights, workload_prompts
    kbuild.build()
    kf.load_library()
    w = WORKLOADS["lm1b"]
    model, B, k, gen = w.model, w.batch, 4, w.gen_len
    weights = make_weights(model)
    stream = torch.cuda.Stream()
    dec = kf.Decoder(model, weights, max_batch=B, max_k=k, stream=stream.cuda_stream)
    dec.prefill(workload_prompts(w, B))
    calls = gen // k
    z = torch.rand((calls, B, k), device="cuda")
    zc = z.permute(0, 2, 1).contiguous()            # [calls][k][B]: AR call j of block i
    o = torch.zeros((calls, B, k), dtype=torch.int32, device="cuda")
    o1 = torch.zeros((calls, k, B), dtype=torch.int32, device="cuda")

    def teacher():
        dec.rewind()
        for i in range(calls):
            kf.kf_teacher_step(dec.ctx, B, k, z[i], o[i])

    def ar_calls():
        dec.rewind()
        for i in range(calls):
            for j in range(k):
                kf.kf_decode_step(dec.ctx, B, 0, zc[i, j], o1[i, j])

    def timed(fn):
        for _ in range(max(3, args.warmup)):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / args.steps

    ms_t, ms_a = timed(teacher), timed(ar_calls)
    toks = B * calls * k
    print(json.dumps({"metric": "G* teacher tokens/s (k AR steps per call)", "unit": "tokens/s",
                      "value": toks / (ms_t / 1e3), "ar_calls_value": toks / (ms_a / 1e3),
                      "ms_per_generation": ms_t, "ar_calls_ms_per_generation": ms_a,
                      "config": {"workload": "lm1b", "batch": B, "k": k, "gen_tokens_per_seq": gen},
                      "data": "synthetic", "dtype": "bf16"}))

    # continuous batching: requests of prompt 32 and 32..96 generated tokens
    n_req = 4 * B
    reqs = make_requests(n_req, w.prompt_len, 32, gen, k, model.vocab)
    zr = torch.rand((64, B, k), device="cuda")
    orr = torch.zeros((B, k), dtype=torch.int32, device="cuda")
    for rep in range(2):                             # the second pass is timed
        dec.prefill([r[0] for r in reqs[:B]])
        left = [r[1] for r in reqs[:B]]
        nxt, done, produced, steps, adm_s, n_calls = B, 0, 0, 0, 0.0, 0
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        while done < n_req:
            kf.kf_decode_step(dec.ctx, B, k, zr[steps % 64], orr)
            steps += 1
            slots, prompts = [], []
            for b in range(B):
                if left[b] > 0:
                    produced += min(k, left[b])
                    left[b] -= k
                    if left[b] <= 0:
                        done += 1
                        slots.append(b)
                        if nxt < n_req:
                            prompts.append(reqs[nxt][0])
                            left[b] = reqs[nxt][1]
                            nxt += 1
                        else:
                            # no request left: an idle slot restarts a short prompt
                            # (not counted) so its length stays within max_len
                            prompts.append(reqs[0][0][:k])
            if slots:
                ta = time.perf_counter()
                dec.admit(slots, prompts)          # all of this step's finished slots at once
                adm_s += time.perf_counter() - ta
                n_calls += 1
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    print(json.dumps({"metric": "continuous batching: generated tokens/s with admissions",
                      "unit": "tokens/s", "value": produced / wall, "requests": n_req,
                      "decode_steps": steps, "admissions": n_req, "admit_calls": n_calls,
                      "admit_ms_per_call": 1e3 * adm_s / max(1, n_calls),
                      "config": {"workload": "lm1b", "slots": B, "k": k, "prompt_len": w.prompt_len,
                                 "gen_len": [32, gen]},
                      "data": "synthetic", "dtype": "bf16", "timing": "host wall clock (admissions synchronise)"}))
    dec.close()
    return 0


def run_train_attention(args):
    """SingleForward / DoubleForward attention (App. C.2), bf16, head_dim 64:
    the mask-aware kernel against the same kernel visiting every key tile
    (the dense-mask cost).  Reports TFLOP/s over the mask's pairs
    (4 * 64 flops per visible (query, key) pair)."""
    import ctypes
    import torch
    from paper_2606_10820_gb300 import build as kbuild
    from paper_2606_10820_gb300 import kforcing as kf
    kbuild.build()
    lib = kf.load_library()
    lib.kf_op_train_attention.argtypes = [ctypes.c_int32] * 7 + [ctypes.c_void_p] * 4 + \
        [ctypes.c_int32, ctypes.c_void_p]
    pk, peak_src = peaks()
    for blocks, B, H, N, k in [(1, 32, 12, 128, 4), (1, 4, 12, 1024, 4), (2, 4, 12, 1024, 4),
                               (1, 4, 12, 1024, 8)]:
        T = N + blocks * N * k
        g = torch.Generator(device="cuda").manual_seed(7)
        q, kk, v = (torch.randn(B, T, H, 64, device="cuda", generator=g).to(torch.bfloat16) for _ in range(3))
        out = torch.empty(B, T, H, 64, device="cuda")
        # visible pairs: context rows, then per block row its context prefix and windows
        ctx = N * (N + 1) // 2
        pairs = ctx + k * ctx + N * k * (k + 1) // 2
        if blocks == 2:
            pairs += k * ctx + N * k * k + N * k * (k + 1) // 2
        flops = 4.0 * 64 * pairs * B * H
        res = {}
        for dense in (0, 1):
            def call():
                lib.kf_op_train_attention(blocks, B, H, N, k, 0, T, q.data_ptr(), kk.data_ptr(),
                                          v.data_ptr(), out.data_ptr(), dense, None)
            for _ in range(max(3, args.warmup)):
                call()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(max(10, args.steps)):
                call()
            e1.record()
            torch.cuda.synchronize()
            res[dense] = e0.elapsed_time(e1) / max(10, args.steps)
        tf = flops / (res[0] / 1e3) / 1e12
        print(json.dumps({
            "metric": "training attention (App. C.2) TFLOP/s over the mask's pairs", "unit": "TFLOP/s",
            "value": tf, "ms": res[0], "dense_mask_ms": res[1], "speedup_vs_dense_mask": res[1] / res[0],
            "roofline": {"bound": "tensor", "achieved": tf, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": tf / pk["bf16_tflops"], "peak_source": peak_src},
            "config": {"mask": "SingleForward" if blocks == 1 else "DoubleForward", "batch": B, "heads": H,
                       "N": N, "k": k, "tokens": T, "visible_pairs_per_head": pairs},
            "data": "synthetic", "dtype": "bf16"}))
    return 0


def main():
    args = parse()
    if args.sweep:
        return run_sweep(args)
    if args.serving:
        return run_serving(args)
    if args.train_attention:
        return run_train_attention(args)
    if args.impl == "reference":
        return run_reference(args)
    import torch
    from paper_2606_10820_gb300 import build as kbuild
    from paper_2606_10820_gb300 import kforcing as kf
    from synth import make_weights, workload_prompts

    rank, world, dist = dist_init(args.gpus)
    dev = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(dev)
    if rank == 0:
        kbuild.build()
    if dist is not None:
        dist.barrier()
    kf.load_library()

    w, B, gen = workload_of(args)
    model = w.model
    k = args.k
    weights = make_weights(model)
    prompts = workload_prompts(w, B)
    stream = torch.cuda.Stream()
    max_k = max(k, 1)
    dec = kf.Decoder(model, weights, max_batch=B, max_k=max_k, stream=stream.cuda_stream)
    dec.prefill(prompts)
    pk, peak_src = peaks()

    def measure(kk, host=False):
        nout = max(kk, 1)
        calls = -(-gen // nout)
        rng = np.random.default_rng(2)
        z = rng.random((calls, B, nout), dtype=np.float32)
        if host:
            zbuf = torch.from_numpy(z).pin_memory()
            obuf = torch.zeros((calls, B, nout), dtype=torch.int32).pin_memory()
        else:
            zbuf = torch.from_numpy(z).cuda()
            obuf = torch.zeros((calls, B, nout), dtype=torch.int32, device="cuda")

        def one():
            dec.rewind()
            for i in range(calls):
                kf.kf_decode_step(dec.ctx, B, kk, zbuf[i], obuf[i])

        for _ in range(args.warmup):
            one()
        torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        e0.record(stream)
        for _ in range(args.steps):
            one()
        e1.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
        ms = e0.elapsed_time(e1) if not host else wall * 1000.0
        ms = max_over_ranks(ms, dist)
        tokens = world * args.steps * B * calls * nout
        return tokens / (ms / 1000.0), ms / args.steps, calls, z.nbytes // calls * calls

    clk = Clocks(dev)
    clk.start()
    val, ms_step, calls, _ = measure(k)
    clocks = clk.stop()
    e2e_val, e2e_ms, _, _ = measure(k, host=True)
    nout = max(k, 1)
    h2d = calls * B * nout * 4
    d2h = calls * B * nout * 4
    ar = None
    if not args.no_ar and k != 0:
        ar_val, ar_ms, ar_calls, _ = measure(0)
        ar = {"value": ar_val, "unit": "tokens/s", "ms_per_step": ar_ms, "calls_per_step": ar_calls}

    # per-kernel times over one profiled step (a graph with event nodes) near the middle of the generation
    dec.rewind()
    zmid = np.random.default_rng(5).random((B, nout), dtype=np.float32)
    out = np.zeros((B, nout), np.int32)
    launches_per_step = 0
    ms_kind = np.zeros(kf.KF_KIND_COUNT, np.float32)
    n_kind = np.zeros(kf.KF_KIND_COUNT, np.int32)
    ms_tot = np.zeros(kf.KF_KIND_COUNT, np.float64)
    n_tot = np.zeros(kf.KF_KIND_COUNT, np.int64)
    shape_launch = {}
    for i in range(calls):
        P = 1 if i == 0 else nout
        if i in (0, 1, calls // 2):
            lens = dec.lengths()
            kf.kf_profile_step(dec.ctx, B, k, zmid, out, ms_kind, n_kind)
            shape_launch[P] = int(n_kind.sum())
            if i == calls // 2:
                ms_tot += ms_kind
                n_tot += n_kind
                mid_lens = lens.copy()
        else:
            dec.step(k, zmid, out)
    launches_per_step = sum(shape_launch.get(1 if i == 0 else nout, 0) for i in range(calls))
    costs = kind_costs(model, B, nout, k, mid_lens)
    tot_ms = {kf.KIND_NAMES[i]: float(ms_tot[i]) for i in range(kf.KF_KIND_COUNT)}
    dom = max(costs, key=lambda n: tot_ms.get(n, 0.0))
    idx = kf.KIND_NAMES.index(dom)
    avg_ms = ms_tot[idx] / max(1, n_tot[idx])
    c = costs[dom]
    t_hbm = c["bytes"] / (pk["hbm_gbs"] * 1e9)
    t_tc = c["flops"] / (pk["bf16_tflops_sustained"] * 1e12)
    if t_tc > t_hbm:
        ach = c["flops"] / (avg_ms / 1e3) / 1e12
        roof = {"bound": "tensor", "achieved": ach, "peak": pk["bf16_tflops_sustained"],
                "unit": "TFLOP/s"}
    else:
        ach = c["bytes"] / (avg_ms / 1e3) / 1e9
        roof = {"bound": "hbm", "achieved": ach, "peak": pk["hbm_gbs"], "unit": "GB/s"}
    traffic = measured_traffic(dom, args.workload, B, k)
    roof.update({"frac": roof["achieved"] / roof["peak"], "traffic": traffic, "kernel": dom,
                 "launch_ms": avg_ms, "peak_source": peak_src,
                 "algorithmic_bytes": c["bytes"], "algorithmic_flops": c["flops"]})
    # whole-step roofline (slower of HBM bytes and tensor flops), over the generation
    t_roof = 0.0
    for i in range(calls):
        P = 1 if i == 0 else nout
        lens = np.array([len(p) - 1 + (0 if i == 0 else 1 + (i - 1) * nout) for p in prompts])
        byt, fl = step_bytes_flops(model, B, P, k, lens)
        t_roof += max(byt / (pk["hbm_gbs"] * 1e9), fl / (pk["bf16_tflops_sustained"] * 1e12))
    step_frac = (t_roof * 1e3) / ms_step

    cpu = None
    if rank == 0 and not args.no_cpu:
        Bs = min(B, 16)
        r, ncalls, el = cpu_oracle_rate(model, weights, prompts[:Bs], k, budget_s=15.0,
                                        max_calls=24)
        cpu = {"value": r, "unit": "tokens/s", "cores": cpu_threads(), "kind": "oracle",
               "sample": f"{Bs} of the {B} sequences, {ncalls} decode calls of k={k} "
                         f"after the prompt ({el:.1f} s, numpy fp64)"}
    dec.close()
    if rank == 0:
        line = {
            "metric": METRIC, "value": val, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": model.dtype, "data": "synthetic: seeded N(0,0.02) weights, uniform prompt ids, U[0,1) noise",
            "config": bench_config(w, B, gen, k),
            "k1": ar,
            "speedup_k_vs_k1": (val / ar["value"]) if ar else None,
            "step_roofline_frac": step_frac,
            "e2e": {"value": e2e_val, "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h},
            "roofline": roof,
            "cpu_baseline": cpu,
            "clocks": clocks,
            "gpu_launches": launches_per_step * args.steps,
            "kernel_ms_mid_step": {kn: round(v, 4) for kn, v in tot_ms.items() if v > 0},
        }
        print(json.dumps(line))
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
