#!/usr/bin/env python3
"""Throughput of speculative beam decoding with strict top-K verification on the 7B-shape workload.

One step = one recommendation list per user: prefill of the user history, then speculative steps
(gamma = 4 drafted beam-search steps of width N = 40 by the draft model, one verification call of
the 7B-shape target over the whole drafted tree, strict top-K verification with K = 10) until every
user holds K complete items.  Metric: rec lists/s (whole job), with the verification call's HBM
roofline fraction and the weight-streaming GEMM's achieved bandwidth measured live.

Weights are seeded random-init of the LLaMA-7B shape (the paper's trained LC-Rec / LLaMA-68M
weights and datasets are not available); inputs are synthetic (see synth/world.py).  Inputs are
larger than L2: every step streams the 13.5 GB of target weights several times.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--workload 7b]
                  [--mode strict|relaxed]
Under torchrun every rank decodes its own users (replicas, no collective on the data path).
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "rec lists/sec (7B-shape target); verify-call % of roofline"


# ---- multi-rank host logic (replicas: every rank decodes its own users, nothing is exchanged on
# the data path; only the timing is reduced)
def shard_users(all_prompts, rank, world):
    """This rank's users: an equal contiguous share of the job's users."""
    n = len(all_prompts) // world
    return all_prompts[rank * n:(rank + 1) * n]


def job_ms(ms, world, device=None):
    """Duration of the job's timed region: the slowest rank's (max over ranks)."""
    if world == 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(users_per_rank, world, steps, ms):
    """Whole-job throughput: the users of all ranks, steps lists each, over the job's duration."""
    return users_per_rank * world * steps / (ms / 1e3)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="7b")
    ap.add_argument("--mode", choices=["strict", "relaxed"], default="strict")
    ap.add_argument("--norm", choices=["masked", "full"], default="masked",
                    help="constrained log-softmax normaliser: the valid children (default) or the whole "
                         "vocabulary (the LM head then runs over all V rows)")
    ap.add_argument("--early-reject", action="store_true",
                    help="decide level 1 of depth-0 steps from the prefill logits and skip the tree forward "
                         "when every user rejects it (same outputs; not part of the paper's method)")
    ap.add_argument("--verify-only", type=int, default=0, metavar="R",
                    help="profiling aid: R verification calls of the workload, each in an NVTX range 'verify'")
    ap.add_argument("--layers", type=int, default=0, metavar="L",
                    help="profiling aid for --verify-only: cut the target to its first L layers (small ncu captures)")
    ap.add_argument("--kernel-probe", action="store_true",
                    help="profiling aid: the four layer GEMMs of the 7B shape at T=120 over 8 layers of weights")
    ap.add_argument("--sweep", action="store_true",
                    help="verification-call sweep on the 7B-shape target (512-token prompts, 50 000 items): "
                         "K in {1,5,10,20} x gamma in {1..4} x N in {K,2K,4K} x batch in {1,4,16}, strict and "
                         "relaxed; one JSON line per point")
    ap.add_argument("--sweep-batches", default="1,4,16", help="--sweep: the batch axis")
    ap.add_argument("--tree-vs-beam", action="store_true",
                    help="one target decoding step of beam width W: the W beams as one tree sharing the "
                         "user's history (tree attention) against W separate sequences, each with its own "
                         "copy of the history; one JSON line per W")
    return ap.parse_args()


# DRAM bytes per algorithmic byte of the batch-1 verification-call forward kernel (T = 120 tree
# tokens): dram__bytes_read.sum + dram__bytes_write.sum of one ncu capture of that kernel with the
# target cut to 2 layers (856.6 MB of traffic for 838.7 MB of algorithmic bytes).  Measured for the
# 128-token-tile schedule only: other workloads report no traffic figure.  TRAFFIC_CURRENT says
# whether the capture is of the kernel as built now; when it is not, the line reports no traffic.
TRAFFIC_PER_ALG_BYTE = 856.6 / 838.7
TRAFFIC_CURRENT = False   # captured before the residual-update sums went to one part in flight


def peaks():
    """(copy GB/s, bf16 TFLOP/s burst, bf16 TFLOP/s sustained, source)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return (float(p["hbm_gbs"]), float(p["bf16_tflops"]),
                float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured")
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def verify_bytes_flops(w, T, P_users, full=False):
    """Algorithmic bytes / FLOPs of one verification call: weights once, item-code LM-head rows (all
    V rows under FULL normalisation), every user's prefix KV read once, the tree's node KV written
    (bf16)."""
    t = w.target
    d, f, Lr = t.d_model, t.d_ffn, t.n_layers
    per_layer = 4 * d * d + 3 * d * f
    head = t.vocab if full else 1024
    B = 2 * Lr * per_layer + 2 * head * d + sum(P_users) * Lr * 2 * d * 2 + T * Lr * 2 * d * 2
    F = 2 * T * Lr * per_layer + sum(4 * (T / len(P_users)) * (P + 2) * d * Lr for P in P_users) + 2 * T * d * head
    return B, F


# ----------------------------------------------------------------------------------------------
# CPU oracle leg (bounded sample)
# ----------------------------------------------------------------------------------------------

def oracle_sample(w, mode, layers=1):
    """One recommendation list of the oracle with the target truncated to `layers` of its layers and
    the draft to one layer; returns (seconds for the sample, seconds scaled to the full model)."""
    from oracle.model import Model, PathEvaluator
    from oracle.sd import sd_decode
    from oracle.trie import Trie
    tspec = synth.ModelSpec(layers, w.target.d_model, w.target.n_heads, w.target.d_ffn, w.target.vocab)
    dspec = synth.ModelSpec(1, w.draft.d_model, w.draft.n_heads, w.draft.d_ffn, w.draft.vocab)
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    prompt = synth.make_prompts(1, w.prompt_len, w.target.vocab, w.seed)[0]
    tm = Model(tspec, synth.model_weights(tspec, w.seed, "target"), w.code_base)
    dm = Model(dspec, synth.model_weights(dspec, w.seed, "draft"), w.code_base)
    trie = Trie(items)
    t0 = time.perf_counter()
    te, de = PathEvaluator(tm, prompt), PathEvaluator(dm, prompt)

    def rows(ev):
        return lambda ps: [r[256 * len(p):256 * (len(p) + 1)].astype(np.float32) for p, r in zip(ps, ev.logits(ps))]
    sd_decode(rows(te), rows(de), trie, w.K, w.N, w.gamma, mode, seed=w.philox_seed)
    dt = time.perf_counter() - t0
    return dt, dt * w.target.n_layers / layers


def run_reference(args, w):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cores = os.cpu_count()
    times = []
    for i in range(args.warmup + args.steps):
        _, scaled = oracle_sample(w, args.mode)
        if i >= args.warmup:
            times.append(scaled)
    per_list = statistics.mean(times)
    value = 1.0 / per_list
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "rec lists/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_list * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": f"{w.name}: 7B-shape target, 4-layer d=768 draft, K={w.K}, N={w.N}, gamma={w.gamma}, "
                               f"P={w.prompt_len[0]}, {w.n_items} items, {args.mode} verification, batch 1"},
        "cpu_baseline": {"value": value, "unit": "rec lists/s", "cores": cores, "kind": "oracle",
                         "sample": "one rec list with the target cut to 1 of 32 layers and the draft to 1 layer, "
                                   "time x32"},
        "e2e": {"value": value, "unit": "rec lists/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------------------------
# GPU leg
# ----------------------------------------------------------------------------------------------

class Clocks:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu):
        self.gpu = gpu
        self.p = None
        self.f = tempfile.NamedTemporaryFile(mode="w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                       "-lms", "100", "-i", str(self.gpu)], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.p.terminate()
        self.p.wait()
        self.f.flush()
        self.f.seek(0)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.f.read().splitlines():
            t = [x.strip() for x in line.split(",")]
            if len(t) < 9:
                continue
            try:
                sm.append(float(t[1]))
                mx.append(float(t[2]))
            except ValueError:
                continue
            for n, v in zip(names, t[5:9]):
                if v.lower() in ("active", "0x1", "1"):
                    reasons.add(n)
        os.unlink(self.f.name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def run_ours(args, w):
    import torch
    import torch.distributed as dist

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    import paper_2410_05165_gb300 as ats
    try:
        ats.load()
    except RuntimeError:
        from paper_2410_05165_gb300.build import build
        build()
        ats.load()
    mode = ats.SD_STRICT if args.mode == "strict" else ats.SD_RELAXED
    vmode = ats.STRICT if args.mode == "strict" else ats.RELAXED

    def to_dev(spec, role):
        out = {}
        for name, arr in synth.iter_model_tensors(spec, w.seed, role):
            out[name] = torch.from_numpy(arr).to(device="cuda", dtype=torch.bfloat16)
        return out
    tw, dw = to_dev(w.target, "target"), to_dev(w.draft, "draft")
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    prompts = shard_users(synth.make_prompts(w.n_users * world, w.prompt_len, w.target.vocab, w.seed), rank, world)
    B = len(prompts)
    P_users = [len(p) for p in prompts]
    ctx = ats.Context(w.target, tw, w.draft, dw, items, w.code_base, max_users=B, max_prompt=max(P_users),
                      max_K=w.K, max_N=w.N, max_gamma=w.gamma)
    h_tok = torch.from_numpy(np.concatenate(prompts).astype(np.int32)).pin_memory()
    toks = h_tok.cuda()
    offsets = np.concatenate([[0], np.cumsum(P_users)]).astype(np.int32)
    o = ats.opts(w.K, w.N, w.gamma, w.philox_seed, norm=ats.NORM_FULL if args.norm == "full" else ats.NORM_MASKED)
    stream = torch.cuda.current_stream()

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()

    ctx.set_early_reject(args.early_reject)
    # ---- warm-up, then K timed steps (inputs resident in HBM)
    for _ in range(args.warmup):
        ctx.beam_search(toks, offsets, o, mode)
    barrier()
    clocks = Clocks(local)
    clocks.start()
    l0 = ctx.profile_read(-1)["launches"]
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    stats = None
    for _ in range(args.steps):
        _, _, stats = ctx.beam_search(toks, offsets, o, mode)
    e1.record(stream)
    barrier()
    clk = clocks.stop()
    launches = (ctx.profile_read(-1)["launches"] - l0) / args.steps
    ms = job_ms(e0.elapsed_time(e1), world, "cuda")
    value = job_rate(B, world, args.steps, ms)

    # ---- end to end through the C ABI: pinned host prompt -> device, decode, items -> host
    h_items = torch.empty(B, w.K, 4, dtype=torch.int32).pin_memory()
    h_sc = torch.empty(B, w.K, dtype=torch.float32).pin_memory()
    d_items = torch.empty(B, w.K, 4, dtype=torch.int32, device="cuda")
    d_sc = torch.empty(B, w.K, dtype=torch.float32, device="cuda")
    barrier()
    e0.record(stream)
    for _ in range(args.steps):
        toks.copy_(h_tok, non_blocking=True)
        ctx.beam_search(toks, offsets, o, mode, items_out=d_items, scores_out=d_sc)
        h_items.copy_(d_items, non_blocking=True)
        h_sc.copy_(d_sc, non_blocking=True)
    e1.record(stream)
    barrier()
    ms_e2e = job_ms(e0.elapsed_time(e1), world, "cuda")
    e2e = {"value": job_rate(B, world, args.steps, ms_e2e), "unit": "rec lists/s",
           "h2d_bytes_per_step": int(h_tok.numel() * 4), "d2h_bytes_per_step": int(h_items.numel() * 4 + h_sc.numel() * 4)}

    # ---- the verification call alone (first call of a decode: depth 0, T = 3 N tree tokens); always
    # the full call, whatever --early-reject says
    ctx.set_early_reject(False)
    hbm, tf, tf_sus, peak_kind = peaks()
    ver_ms, fk = [], {"ms": 0.0, "launches": 0}
    n_timed = max(3, args.steps)
    for rep in range(3 + n_timed + 2):
        ctx.prefill(toks, offsets)
        ctx.begin_step(o)
        for _ in range(w.gamma):
            ctx.draft_step(o, vmode)
        prof = rep >= 3 + n_timed
        if prof:
            ctx.profile(True)
        torch.cuda.synchronize()
        e0.record(stream)
        ctx.verify(o, vmode)
        e1.record(stream)
        torch.cuda.synchronize()
        if prof:
            r = ctx.profile_read(6)   # the persistent forward kernel of the verification call
            fk["ms"] += r["ms"]
            fk["launches"] += r["launches"]
            ctx.profile(False)
        elif rep >= 3:
            ver_ms.append(e0.elapsed_time(e1))
    T_first = min(w.gamma, 3) * w.N * B
    vb, vf = verify_bytes_flops(w, T_first, P_users, full=args.norm == "full")
    v_ms = statistics.median(ver_ms)
    t_roof = max(vb / (hbm * 1e9), vf / (tf * 1e12)) * 1e3
    k_ms = fk["ms"] / max(1, fk["launches"])
    # the kernel's bound: HBM when its algorithmic bytes take longer than its FLOPs at the tensor
    # peak (batch 1: T = 120 tree tokens), tensor otherwise (16 users: T = 3840); a launch of several
    # ms is a long kernel, so the tensor peak is the sustained one
    if vb / (hbm * 1e9) >= vf / (tf_sus * 1e12):
        roof = {"bound": "hbm", "achieved": vb / (k_ms / 1e3) / 1e9, "peak": hbm, "unit": "GB/s"}
    else:
        roof = {"bound": "tensor", "achieved": vf / (k_ms / 1e3) / 1e12, "peak": tf_sus, "unit": "TFLOP/s",
                "peak_note": "sustained bf16 (a launch of several ms)"}
    roof["frac"] = roof["achieved"] / roof["peak"]

    lo, hi = w.prompt_len
    p_label = str(lo) if lo == hi else f"U[{lo},{hi}] (mean {np.mean(P_users):.0f})"
    line = {
        "metric": METRIC, "value": value, "unit": "rec lists/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic (seeded random-init weights, synthetic items)",
        "config": {"workload": f"{w.name}: 7B-shape target (32L d4096 H32 ffn11008 V33024), draft 4L d768, "
                               f"K={w.K} N={w.N} gamma={w.gamma}, P={p_label}, {w.n_items} Zipf items, "
                               f"{args.mode} verification, {args.norm} normalisation, {B} user(s) per GPU"
                               + (", early rejection at depth 0" if args.early_reject else ""),
                   "l2": "inputs larger than L2 (13.5 GB of target weights per verification call)"},
        "roofline": dict(roof, **{
            "traffic": TRAFFIC_PER_ALG_BYTE * vb if T_first <= 128 and TRAFFIC_CURRENT else None,
            "traffic_source": ("dram__bytes_read.sum + dram__bytes_write.sum of one ncu capture of the same "
                               "kernel with the target cut to 2 layers, scaled by algorithmic bytes"
                               if T_first <= 128 and TRAFFIC_CURRENT else
                               "not captured for this build (the previous build's 2-layer capture: "
                               f"{TRAFFIC_PER_ALG_BYTE:.3f} x algorithmic bytes)" if T_first <= 128 else
                               "not captured at this tree size"),
            "kernel": f"fwd_kernel: persistent forward of the verification call (tcgen05 GEMMs, tree attention, "
                      f"norms; T={T_first} tree tokens)",
            "peak_source": peak_kind, "launches": fk["launches"], "avg_launch_ms": k_ms,
            "alg_bytes_per_launch": vb, "alg_flops_per_launch": vf}),
        "verify_call": {"ms": v_ms, "tree_tokens": T_first, "alg_bytes": vb, "alg_flops": vf,
                        "t_roof_ms": t_roof, "frac_of_roofline": t_roof / v_ms, "peak_source": peak_kind},
        "accepted_steps_per_list": float(np.mean(stats[:, 0])), "verify_calls_per_list": float(np.mean(stats[:, 1])),
        "tree_tokens_per_list": float(np.mean(stats[:, 2])),
        "e2e": e2e, "gpu_launches": int(launches), "clocks": clk,
    }
    if rank == 0 and world == 1:
        cores = os.cpu_count()
        samp, scaled = oracle_sample(w, args.mode, layers=4)
        line["cpu_baseline"] = {"value": 1.0 / scaled, "unit": "rec lists/s", "cores": cores, "kind": "oracle",
                                "sample": f"one rec list with the target cut to 4 of 32 layers (draft 1 layer), "
                                          f"{samp:.1f} s, time x8"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    ctx.close()
    if world > 1:
        dist.destroy_process_group()


def kernel_probe():
    """The weight-streaming GEMM alone at the verification call's shapes (T = 120 tree tokens),
    over 8 layers of distinct weights (3.2 GB, larger than L2), timed with CUDA events."""
    import torch
    import paper_2410_05165_gb300 as ats
    ats.load()
    d, f, T, nl = 4096, 11008, 120, 8
    shapes = {"qkv": (3 * d, d), "o": (d, d), "gate_up": (2 * f, d), "down": (d, f)}
    g = torch.Generator(device="cuda").manual_seed(0)
    Ws = {k: [(torch.randn(m, kk, device="cuda", generator=g) * 0.02).to(torch.bfloat16) for _ in range(nl)]
          for k, (m, kk) in shapes.items()}
    X = {kk: torch.randn(256, kk, device="cuda", generator=g).to(torch.bfloat16) for kk in (d, f)}
    out = {}
    for k, (m, kk) in shapes.items():
        Y = torch.zeros(T, m, device="cuda")
        ts = []
        for rep in range(3):
            for l in range(nl):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                ats.op_gemm(Ws[k][l], X[kk], T, Y=Y)
                e1.record()
                torch.cuda.synchronize()
                if rep:
                    ts.append(e0.elapsed_time(e1))
        t = statistics.median(ts)
        out[k] = {"M": m, "K": kk, "us": t * 1e3, "weight_GBps": m * kk * 2 / (t / 1e3) / 1e9}
    print(json.dumps({"kernel_probe": out}), flush=True)


def verify_only(w, mode, reps, layers=0):
    import dataclasses
    import torch
    import paper_2410_05165_gb300 as ats
    ats.load()
    if layers:
        w = dataclasses.replace(w, target=dataclasses.replace(w.target, n_layers=layers))
    tw = {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
          for n, a in synth.iter_model_tensors(w.target, w.seed, "target")}
    dw = {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
          for n, a in synth.iter_model_tensors(w.draft, w.seed, "draft")}
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    prompts = synth.make_prompts(w.n_users, w.prompt_len, w.target.vocab, w.seed)
    P = [len(p) for p in prompts]
    ctx = ats.Context(w.target, tw, w.draft, dw, items, w.code_base, max_users=len(prompts), max_prompt=max(P),
                      max_K=w.K, max_N=w.N, max_gamma=w.gamma)
    toks = torch.from_numpy(np.concatenate(prompts).astype(np.int32)).cuda()
    off = np.concatenate([[0], np.cumsum(P)]).astype(np.int32)
    o = ats.opts(w.K, w.N, w.gamma, w.philox_seed)
    vm = ats.STRICT if mode == "strict" else ats.RELAXED
    ms = []
    for r in range(reps):
        ctx.prefill(toks, off)
        ctx.begin_step(o)
        for _ in range(w.gamma):
            ctx.draft_step(o, vm)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.nvtx.range_push("verify")
        e0.record()
        ctx.verify(o, vm)
        e1.record()
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    print(json.dumps({"verify_ms": ms}), flush=True)
    ctx.close()


def sweep(batches, reps=2):
    """Verification-call sweep: for every (batch, K, gamma, N, mode) point, prefill the batch's
    512-token histories, draft gamma levels of width N and time the first verification call (median
    of `reps`), with its tree-token count, roofline fraction and accepted steps per user."""
    import torch
    import paper_2410_05165_gb300 as ats
    ats.load()
    w = synth.workload("7b")
    hbm, tf, _, src = peaks()
    tw = {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
          for n, a in synth.iter_model_tensors(w.target, w.seed, "target")}
    dw = {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
          for n, a in synth.iter_model_tensors(w.draft, w.seed, "draft")}
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    for B in batches:
        prompts = synth.make_prompts(B, w.prompt_len, w.target.vocab, w.seed)
        P = [len(p) for p in prompts]
        ctx = ats.Context(w.target, tw, w.draft, dw, items, w.code_base, max_users=B, max_prompt=max(P),
                          max_K=20, max_N=80, max_gamma=4)
        toks = torch.from_numpy(np.concatenate(prompts).astype(np.int32)).cuda()
        off = np.concatenate([[0], np.cumsum(P)]).astype(np.int32)
        for K in (1, 5, 10, 20):
            for gamma in (1, 2, 3, 4):
                for N in (K, 2 * K, 4 * K):
                    for mode in ("strict", "relaxed"):
                        o = ats.opts(K, N, gamma, w.philox_seed)
                        vm = ats.STRICT if mode == "strict" else ats.RELAXED
                        ms, acc_mean, T = [], 0.0, 0
                        for _ in range(reps):
                            ctx.prefill(toks, off)
                            ctx.begin_step(o)
                            for _ in range(gamma):
                                ctx.draft_step(o, vm)
                            # tree tokens of the call: the drafted levels 1 .. min(gamma, L - 1) (level-L
                            # nodes complete an item and are not forwarded; no incoming beams at depth 0)
                            cnt = ctx.debug_tree(gamma)["count"]
                            T = int(cnt[:, 1:1 + min(gamma, 3)].sum())
                            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                            e0.record()
                            acc, _, _, _ = ctx.verify(o, vm)
                            e1.record()
                            torch.cuda.synchronize()
                            ms.append(e0.elapsed_time(e1))
                            acc_mean = float(acc.float().mean())
                        vb, vf = verify_bytes_flops(w, T, P)
                        t_roof = max(vb / (hbm * 1e9), vf / (tf * 1e12)) * 1e3
                        v = float(np.median(ms))
                        print(json.dumps({"sweep": "verify", "batch": B, "K": K, "gamma": gamma, "N": N, "mode": mode,
                                          "tree_tokens": T, "verify_ms": round(v, 4),
                                          "bound": "hbm" if vb / (hbm * 1e9) >= vf / (tf * 1e12) else "tensor",
                                          "roofline_frac": round(t_roof / v, 4), "accepted_steps": acc_mean,
                                          "peak_source": src}), flush=True)
        ctx.close()


def tree_vs_beam(widths=(5, 10, 20, 40, 80), reps=3):
    """Cost of one target decoding step of beam search with W beams at depth 1 of the item (the
    analogue of the paper's tree-attention speedup, Sec. 4 / appendix): the W beams forwarded as
    one tree whose nodes share the user's 512-token history in the paged KV cache, against W
    independent sequences, each prefilled with its own copy of the history (W users of one beam).
    Both calls forward W tokens through the 7B-shape target; the first reads one history's K/V
    per layer, the second W of them."""
    import torch
    import paper_2410_05165_gb300 as ats
    ats.load()
    w = synth.workload("7b")
    tw = {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
          for n, a in synth.iter_model_tensors(w.target, w.seed, "target")}
    dw = {n: torch.from_numpy(a).to(device="cuda", dtype=torch.bfloat16)
          for n, a in synth.iter_model_tensors(w.draft, w.seed, "draft")}
    items = synth.make_items(w.n_items, w.code_dist, w.zipf_a, w.seed)
    prompt = synth.make_prompts(1, w.prompt_len, w.target.vocab, w.seed)[0]

    def call_ms(B, K):
        ctx = ats.Context(w.target, tw, w.draft, dw, items, w.code_base, max_users=B, max_prompt=len(prompt),
                          max_K=K, max_N=K, max_gamma=1)
        toks = torch.from_numpy(np.concatenate([prompt] * B).astype(np.int32)).cuda()
        off = (np.arange(B + 1) * len(prompt)).astype(np.int32)
        o = ats.opts(K, K, 1, w.philox_seed)
        ms, T = [], 0
        for _ in range(reps):
            ctx.prefill(toks, off)
            ctx.begin_step(o)
            ctx.draft_step(o, ats.STRICT)
            T = int(ctx.debug_tree(1)["count"][:, 1].sum())
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            ctx.verify(o, ats.STRICT)
            e1.record()
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        ctx.close()
        return float(np.median(ms)), T

    for W in widths:
        tree_ms, tree_T = call_ms(1, W)
        beam_ms, beam_T = call_ms(W, 1)
        print(json.dumps({"tree_vs_beam": W, "tree_tokens": tree_T, "tree_ms": round(tree_ms, 4),
                          "per_beam_tokens": beam_T, "per_beam_ms": round(beam_ms, 4),
                          "speedup": round(beam_ms / tree_ms, 3)}), flush=True)


def main():
    args = parse()
    w = synth.workload(args.workload)
    if args.tree_vs_beam:
        tree_vs_beam()
        return
    if args.sweep:
        sweep([int(b) for b in args.sweep_batches.split(",")])
        return
    if args.kernel_probe:
        kernel_probe()
        return
    if args.verify_only:
        verify_only(w, args.mode, args.verify_only, args.layers)
        return
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
