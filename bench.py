#!/usr/bin/env python
"""Benchmark of the budget-conditioned gated prefill on one GB300 per rank.

Workload: LLaVA-1.5-7B-shaped batch -- 16 samples of 576 CLIP ViT-L/14-336
visual tokens (dim 1024, low-rank + salient clusters) and 64 text tokens,
MLP projector 1024->4096->4096, 32-layer decoder (d 4096, 32 heads, SwiGLU
11008, vocab 32000), budgets 25/50/75/100% of full-prefill FLOPs. Weights
and inputs are synthetic (seeded), the paper's datasets and checkpoints are
not used.

A step is one pass of the whole path -- svl_score_select, svl_pack,
svl_gated_prefill -- over one batch; step i uses budget budgets[i % 4].
Reported value: input tokens per second (sum over samples of visual + text
tokens before selection) over the K timed steps, summed over ranks.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the CPU oracle (test infrastructure, float64
arithmetic) on a bounded sample of the same workload; it never touches the
GPU.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2607_20357_gb300 import synth  # noqa: E402

METRIC = "gated-prefill input tokens/sec and executed TFLOP/s (% of bf16 peak) vs budget"
WORKLOAD = "llava"
SEED = 1000


def rank_seed(rank: int) -> int:
    """Each rank runs its own batch (replicas over independent samples)."""
    return SEED + 17 * rank


def job_aggregate(max_part, sum_part, device="cpu"):
    """Whole-job figures over the ranks of the default process group: the
    maximum of each entry of `max_part` (times) and the sum of each entry of
    `sum_part` (tokens, FLOPs). Without a group of more than one rank the
    values come back as given. This is the only collective of the bench."""
    dist = torch.distributed
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in max_part], [float(v) for v in sum_part]
    mx = torch.tensor([float(v) for v in max_part], dtype=torch.float64, device=device)
    sm = torch.tensor([float(v) for v in sum_part], dtype=torch.float64, device=device)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return mx.tolist(), sm.tolist()


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=8)
    ap.add_argument("--warmup", type=int, default=4)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-hbm-sweep", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-fp8", action="store_true", help="skip the e4m3 (FP8 gated projections) pass")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the mixed / gating-sweep / video / Qwen passes")
    ap.add_argument("--decode-only", action="store_true",
                    help="profiling aid: only the decode measurement (bf16, and e4m3 unless --no-fp8)")
    ap.add_argument("--hbm-only", type=str, default="",
                    help="comma-separated batch multipliers: run only the token-controller/pack sweep "
                         "(for small profiler captures)")
    ap.add_argument("--workload", default=WORKLOAD, choices=["llava", "llava13b"],
                    help="llava (the benchmark line) or llava13b (the same batch on LLaVA-1.5-13B shapes)")
    ap.add_argument("--layers", type=int, default=0,
                    help="decoder layers (default: all 32). Fewer layers only for small profiler captures; "
                         "such a line is not the benchmark value")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as fh:
            p = json.load(fh)
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p.get("bf16_tflops_sustained", p["bf16_tflops"]), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def weight_count(d):
    dh = d.d_model // d.n_heads
    per = d.d_model * (d.n_heads * dh * 2 + 2 * d.n_kv_heads * dh) + 3 * d.d_model * d.d_ffn
    return d.n_layers * per + 2 * d.vocab * d.d_model


def workload_config(wl, batch):
    d = wl.dims
    name = "LLaVA-1.5-7B" if wl.name == "llava" else "LLaVA-1.5-13B"
    return {
        "workload": f"{name}-shaped gated prefill: B={batch}, 576 visual (C_v 1024, MLP projector) + 64 text "
                    f"tokens, {d.n_layers} layers d{d.d_model} h{d.n_heads} ffn{d.d_ffn} V{d.vocab}, "
                    f"G={d.n_groups} head groups, {d.n_prefix} prefix layers, budgets 0.25/0.5/0.75/1.0",
        "batch": batch, "n_vis": wl.n_vis[0], "s_text": wl.s_text[0], "budgets": list(wl.budgets),
        "layers": d.n_layers, "d_model": d.d_model, "heads": d.n_heads, "d_ffn": d.d_ffn, "vocab": d.vocab,
        "groups": d.n_groups, "gates": wl.gates,
        "l2": f"not flushed: each step streams {2 * weight_count(d) / 1e9:.0f} GB of weights through the 129 MB L2",
        "parallelism": "replicas (independent batches per GPU, no collective)",
    }


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "out", "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for n, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


class NvmlClock:
    """SM clock samples read through NVML (libnvidia-ml, read-only queries)
    by a background thread every few milliseconds, stamped with the host
    clock; `median(t0, t1)` is the median of the samples in a host-time
    window. Without NVML every median is None."""

    def __init__(self, index, period=0.003):
        import ctypes
        import threading
        self.samples, self.stop, self.thread = [], threading.Event(), None
        self.period = period
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            handle = ctypes.c_void_p()
            if lib.nvmlInit_v2() != 0 or lib.nvmlDeviceGetHandleByIndex_v2(int(index), ctypes.byref(handle)) != 0:
                lib = None
        except OSError:
            lib = None
        self.lib, self.handle = lib, (handle if lib is not None else None)
        if lib is None:
            return
        clock = ctypes.c_uint()

        def run():
            while not self.stop.is_set():
                if self.lib.nvmlDeviceGetClockInfo(self.handle, 1, ctypes.byref(clock)) == 0:  # NVML_CLOCK_SM
                    self.samples.append((time.perf_counter(), clock.value))
                time.sleep(self.period)

        self.thread = threading.Thread(target=run, daemon=True)
        self.thread.start()

    def median(self, t0, t1):
        v = [c for t, c in list(self.samples) if t0 <= t <= t1]
        return statistics.median(v) if v else None

    def close(self):
        if self.thread is not None:
            self.stop.set()
            self.thread.join(timeout=1.0)


# --------------------------------------------------------------------------- flops
def per_kind_flops(dims, k, s_text, lg, gg):
    """Algorithmic FLOPs per GEMM kind for one batch (executed work only)."""
    D, Di, G = dims.d_model, dims.d_ffn, dims.n_groups
    hq, dkv = dims.n_heads * dims.d_head, dims.d_kv
    f = {"qkv_gemm": 0.0, "o_gemm": 0.0, "gateup_gemm": 0.0, "down_gemm": 0.0, "attention": 0.0}
    for b in range(len(k)):
        S = int(k[b]) + int(s_text[b])
        for l in range(dims.n_layers):
            on = G if l < dims.n_prefix else int(lg[b, l] != 0) * int((gg[b, l] != 0).sum())
            a = on / G
            f["qkv_gemm"] += a * 2 * S * D * (hq + 2 * dkv)
            f["o_gemm"] += a * 2 * S * hq * D
            f["gateup_gemm"] += a * 2 * S * D * 2 * Di
            f["down_gemm"] += a * 2 * S * Di * D
            f["attention"] += a * 2 * D * S * (S + 1)
    return f


def executed_flops(svl, desc, k, s_text, n_vis, lg, gg):
    tot = 0.0
    for b in range(len(k)):
        _, ex = svl.svl_flops(desc, int(s_text[b]), int(k[b]), int(n_vis[b]), lg[b].contiguous(), gg[b].contiguous())
        tot += ex
    return tot


TRAFFIC_SOURCES = ("gemm.cu", "decoder.cu", "kernels.cuh", "api.cu")  # the GEMM and its tile order


def traffic_source_hash():
    h = hashlib.sha256()
    for f in TRAFFIC_SOURCES:
        with open(os.path.join(ROOT, "paper_2607_20357_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def gemm_traffic_record():
    """Per-launch DRAM bytes of the dominant GEMM from the committed ncu
    summary, if it was taken on the current source of the kernel and of the
    schedule that orders its tiles."""
    path = os.path.join(ROOT, "profiles", "gemm_traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as fh:
        rec = json.load(fh)
    return rec if rec.get("source_sha256_16") == traffic_source_hash() else None


# --------------------------------------------------------------------------- CPU oracle sample
def oracle_sample_seconds(dims, w_np, x, ids, budget, lg, gg, n_layers):
    """Seconds of the oracle on one sample: front (score/select/pack + final
    norm + LM head) and n_layers decoder layers."""
    from oracle import smartvl_oracle as O
    t0 = time.perf_counter()
    O.forward_sample(dims, w_np, x, ids, budget, lg, gg, mode="fp32", n_layers=0)
    t1 = time.perf_counter()
    O.forward_sample(dims, w_np, x, ids, budget, lg, gg, mode="fp32", n_layers=n_layers)
    t2 = time.perf_counter()
    front = t1 - t0
    return front, max(t2 - t1 - front, 0.0) / max(n_layers, 1), (t2 - t1)


def cpu_oracle_baseline(dims, weights_cpu_layers, weights_rest, batch_cpu, budget, n_layers):
    from oracle import smartvl_oracle as O
    w = O.to_numpy_weights(dict(weights_rest, layers=weights_cpu_layers))
    b = 0
    v0, v1 = int(batch_cpu["vis_off"][b]), int(batch_cpu["vis_off"][b + 1])
    t0, t1 = int(batch_cpu["text_off"][b]), int(batch_cpu["text_off"][b + 1])
    x = batch_cpu["vis"][v0:v1].double().numpy()
    ids = batch_cpu["text_ids"][t0:t1].numpy()
    lg, gg = batch_cpu["layer_gate"][b].numpy(), batch_cpu["group_gate"][b].numpy()
    front, per_layer, wall = oracle_sample_seconds(dims, w, x, ids, budget, lg, gg, n_layers)
    t_full = front + per_layer * dims.n_layers
    tokens = (v1 - v0) + (t1 - t0)
    return tokens / t_full, wall + front


# --------------------------------------------------------------------------- reference arm
def run_reference(args, rank, world):
    """The CPU oracle as the reference arm. One step is a bounded sample of
    the benchmark batch: one of its samples (they cycle through the batch
    and the budgets), its token controller, pack, final norm and LM head
    whole and decoder layers 0-1 of 32. ``ms_per_step`` is the time of that
    sample as measured; ``value`` is the sample's input tokens over the time
    the whole 32-layer path would take at the measured per-layer rate
    (front + 16 x two layers). Samples are independent, so the oracle's
    throughput on the batch is its per-sample throughput."""
    if rank != 0:
        return
    wl = synth.WORKLOADS[args.workload]
    dims = wl.dims
    nl = 2
    w = synth.make_weights(dims, SEED, device="cpu", layers=range(nl))
    from oracle import smartvl_oracle as O
    w_np = O.to_numpy_weights(w)
    bt = synth.make_batch(wl, SEED)  # the budgets below only change k; features are the same for each
    budgets = list(wl.budgets)
    measured, extrapolated, tokens = [], [], []
    for i in range(args.warmup + args.steps):
        budget = budgets[i % len(budgets)]
        b = (i // len(budgets)) % bt["B"]
        v0, v1 = int(bt["vis_off"][b]), int(bt["vis_off"][b + 1])
        t0, t1 = int(bt["text_off"][b]), int(bt["text_off"][b + 1])
        x = bt["vis"][v0:v1].double().numpy()
        ids = bt["text_ids"][t0:t1].numpy()
        front, per_layer, wall = oracle_sample_seconds(dims, w_np, x, ids, budget,
                                                       bt["layer_gate"][b].numpy(), bt["group_gate"][b].numpy(), nl)
        if i >= args.warmup:
            measured.append(wall + front)  # both forward_sample calls of the step
            extrapolated.append(front + per_layer * dims.n_layers)
            tokens.append(x.shape[0] + ids.shape[0])
    value = sum(tokens) / sum(extrapolated)
    cores = os.cpu_count()
    sample = (f"per step one sample of the B={wl.batch} batch (samples and budgets {list(wl.budgets)} cycle): "
              f"token controller, pack, final norm and LM head whole, decoder layers 0-{nl - 1} of "
              f"{dims.n_layers}; value = sample tokens / (front + {dims.n_layers // nl} x the two layers' time)")
    cfg = workload_config(wl, wl.batch)
    cfg["reference_step"] = f"one sample, front + {nl} of {dims.n_layers} layers (measured); throughput per sample"
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1000.0 * statistics.mean(measured), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": cfg, "impl": "reference",
        "ms_per_full_sample_extrapolated": 1000.0 * statistics.mean(extrapolated),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- our arm
def run_ours(args, rank, world, local_rank):
    from paper_2607_20357_gb300 import svl
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    wl = synth.WORKLOADS[args.workload]
    if args.layers:
        wl = synth.dataclasses.replace(wl, dims=synth.reduced(wl.dims, n_layers=args.layers))
    dims = wl.dims
    B = wl.batch
    pk = peaks()

    weights = synth.make_weights(dims, SEED, device=dev)
    max_seq = wl.n_vis[1] + wl.s_text[1] + 64
    if args.workload == "llava" and not args.no_workloads and not args.layers:
        # the mixed (576 + 256) and video (4608 + 64) batches run on this model too
        max_seq = max(max_seq, synth.WORKLOADS["video"].n_vis[1] + synth.WORKLOADS["video"].s_text[1] + 64)
    model = svl.GatedPrefill(dims, weights, max_seq=max_seq)
    if args.hbm_only:
        mults = tuple(int(x) for x in args.hbm_only.split(","))
        print(json.dumps({"hbm_kernels_sweep": run_hbm_sweep(svl, model, wl, dev, pk, mults=mults)}), flush=True)
        model.close()
        return
    seed = rank_seed(rank)
    batches = [synth.make_batch(wl, seed, budget=b, device=dev) for b in wl.budgets]
    if args.decode_only:
        out = {"decode": run_decode(svl, model, batches[1], dims, dev, pk)}
        model.close()
        if not args.no_fp8:
            m8 = svl.GatedPrefill(dims, weights, max_seq=max_seq, gemm_format=svl.SVL_GEMM_E4M3)
            out["fp8_decode"] = run_decode(svl, m8, batches[1], dims, dev, pk, layer_weight_bytes=1)
            m8.close()
        if rank == 0:
            print(json.dumps(out), flush=True)
        return
    outs = [model.alloc_outputs(bt) for bt in batches]
    stream = torch.cuda.current_stream()

    def step(i):
        model.run(batches[i % len(batches)], out=outs[i % len(batches)])

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    status = svl.svl_get_device_status(model.handle)
    if status:
        raise RuntimeError(f"device status {status:#x} after warm-up")

    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    launches0 = svl.svl_launch_count()
    # events only around the dominant kernel inside the timed region: events
    # between kernels would keep each launch from overlapping its predecessor
    live_tag = "gateup_gemm"
    svl.svl_profile_start(model.handle, tags=[live_tag])
    # the SM clock of each step: the host waits for each step, so the step
    # runs on the GPU within its host-time window, where NVML samples the clock
    nv = NvmlClock(local_rank)
    windows = []
    with ClockSampler(local_rank) as clk:
        t_wall0 = time.perf_counter()
        for i in range(args.steps):
            tw0 = time.perf_counter()
            ev[i][0].record(stream)
            step(i)
            ev[i][1].record(stream)
            torch.cuda.synchronize()
            windows.append((tw0, time.perf_counter()))
        t_wall = time.perf_counter() - t_wall0
    nv.close()
    step_mhz = [nv.median(a, b) for a, b in windows]
    kern_live = svl.svl_profile_stop(model.handle)
    launches = svl.svl_launch_count() - launches0
    # a second, untimed pass over the same steps with every kernel bracketed
    # by events: per-kernel shares and the per-budget breakdown
    svl.svl_profile_start(model.handle)
    for i in range(args.steps):
        step(i)
    kern = svl.svl_profile_stop(model.handle)
    per_launch = svl.svl_profile_launches(model.handle)
    if world > 1:
        torch.distributed.barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = sum(step_ms)

    # per-budget accounting (k read back after the timed region)
    desc = model.desc
    per_budget, tokens_total, fexec_total = [], 0, 0.0
    kind_flops = {}
    for j, bt in enumerate(batches):
        nsteps = len(range(j, args.steps, len(batches)))
        if nsteps == 0:
            continue
        k = outs[j]["k"].cpu().numpy()
        nv = (bt["vis_off"][1:] - bt["vis_off"][:-1]).cpu().numpy()
        st = (bt["text_off"][1:] - bt["text_off"][:-1]).cpu().numpy()
        lg, gg = bt["layer_gate"].cpu(), bt["group_gate"].cpu()
        toks = int(nv.sum() + st.sum())
        fex = executed_flops(svl, desc, k, st, nv, lg, gg)
        ms = statistics.mean(step_ms[i] for i in range(j, args.steps, len(batches)))
        mhz = [step_mhz[i] for i in range(j, args.steps, len(batches)) if step_mhz[i]]
        # SM cycles per step (time x median clock): the work in a unit that the
        # power cap's clock changes between steps do not move
        cyc = statistics.mean(step_ms[i] * step_mhz[i] * 1e3 for i in range(j, args.steps, len(batches))
                              if step_mhz[i]) if mhz else None
        per_budget.append({"budget": float(bt["budget"][0]), "k_mean": float(k.mean()), "ms_per_step": ms,
                           "sm_mhz": statistics.median(mhz) if mhz else None, "mcycles_per_step": cyc / 1e6 if cyc else None,
                           "tokens_per_s": toks / (ms / 1000.0), "exec_tflops": fex / (ms / 1000.0) / 1e12,
                           "exec_tflop_per_step": fex / 1e12})
        tokens_total += toks * nsteps
        fexec_total += fex * nsteps
        for kk, v in per_kind_flops(dims, k, st, lg.numpy(), gg.numpy()).items():
            kind_flops[kk] = kind_flops.get(kk, 0.0) + v * nsteps

    # device time per tag and budget (every step launches the same kernels)
    per_step = len(per_launch) // max(args.steps, 1)
    for p in per_budget:
        j = [q["budget"] for q in per_budget].index(p["budget"])
        agg = {}
        steps_j = list(range(j, args.steps, len(batches)))
        for i in steps_j:
            for tag, ms in per_launch[i * per_step:(i + 1) * per_step]:
                agg[tag] = agg.get(tag, 0.0) + ms / len(steps_j)
        p["kernel_ms"] = {t: round(v, 4) for t, v in sorted(agg.items(), key=lambda kv: -kv[1])}

    # linear-in-FLOPs check: t(b)/t(1) / (F(b)/F(1)) - 1
    full = [p for p in per_budget if abs(p["budget"] - 1.0) < 1e-6]
    if full:
        for p in per_budget:
            p["time_vs_flops_ratio_minus_1"] = (p["ms_per_step"] / full[0]["ms_per_step"]) / \
                (p["exec_tflop_per_step"] / full[0]["exec_tflop_per_step"]) - 1.0
            if p["mcycles_per_step"] and full[0]["mcycles_per_step"]:
                p["cycles_vs_flops_ratio_minus_1"] = (p["mcycles_per_step"] / full[0]["mcycles_per_step"]) / \
                    (p["exec_tflop_per_step"] / full[0]["exec_tflop_per_step"]) - 1.0

    # dominant kernel roofline (tensor-bound GEMM)
    gemm_tags = ["qkv_gemm", "o_gemm", "gateup_gemm", "down_gemm"]
    dom = max(gemm_tags, key=lambda t: kern.get(t, (0, 0.0))[1])
    n_l, t_l = kern_live[dom] if dom in kern_live else kern[dom]
    achieved = kind_flops[dom] / (t_l / 1000.0) / 1e12
    peak = pk["bf16_tflops_sustained"]
    traffic_rec = gemm_traffic_record()
    roofline = {"kernel": dom, "bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "peak_source": pk["source"] + " bf16 sustained",
                "timing": "CUDA events around each launch inside the timed region" if dom in kern_live
                else "CUDA events of the profiled pass",
                "launches": n_l, "avg_launch_ms": t_l / n_l,
                "flops_per_launch": kind_flops[dom] / n_l,
                "traffic": (traffic_rec["dram_bytes_per_launch"] * (kind_flops[dom] / n_l)
                            / traffic_rec["flops_per_launch_at_capture"])
                if traffic_rec and dom == "gateup_gemm" else None,
                "traffic_note": "DRAM bytes of one ncu capture (profiles/gemm_traffic.json, budget-1.0 launch) "
                                "scaled to this run's average launch by its FLOPs"}
    kernels = {t: {"launches": n, "total_ms": ms, "share": ms / max(sum(v[1] for v in kern.values()), 1e-9)}
               for t, (n, ms) in sorted(kern.items(), key=lambda kv: -kv[1][1])}
    for t in list(kind_flops):
        if t in kernels:
            kernels[t]["tflops"] = kind_flops[t] / (kernels[t]["total_ms"] / 1000.0) / 1e12

    # whole-job aggregate over ranks: max time, summed tokens
    (total_ms,), (tokens_total, fexec_total) = job_aggregate([total_ms], [tokens_total, fexec_total], dev)
    value = tokens_total / (total_ms / 1000.0)

    hbm = None
    if rank == 0 and not args.no_hbm_sweep:
        hbm = run_hbm_sweep(svl, model, wl, dev, pk)

    # e2e through the host-buffer entry point: H2D of inputs, D2H of logits
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, svl, model, batches, dims, world, dev)

    dec = None
    if rank == 0 and not args.no_decode:
        dec = run_decode(svl, model, batches[1], dims, dev, pk)

    gated = None
    if not args.no_workloads and not args.layers and args.workload == "llava":
        del outs
        torch.cuda.empty_cache()
        gated = run_gated_workloads(args, svl, model, dev, pk)

    fp8 = None
    if rank == 0 and not args.no_fp8:
        model.close()  # its workspace and outputs go; the e4m3 model holds its own weight codes
        fp8 = run_fp8(args, svl, wl, weights, batches, dev, pk, max_seq)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        nl = 16
        wl_cpu = [{k: v.cpu() for k, v in weights["layers"][l].items()} for l in range(nl)]
        rest = {k: (v.cpu() if isinstance(v, torch.Tensor) else v) for k, v in weights.items() if k != "layers"}
        b_cpu = {k: (v.cpu() if isinstance(v, torch.Tensor) else v) for k, v in batches[1].items()}
        tps, secs = cpu_oracle_baseline(dims, wl_cpu, rest, b_cpu, float(b_cpu["budget"][0]), nl)
        cpu = {"value": tps, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"sample 0 of the budget-{float(b_cpu['budget'][0])} batch: token controller, pack, "
                         f"final norm, LM head whole; decoder layers 0-{nl - 1} timed and scaled x"
                         f"{dims.n_layers // nl}; fp32 storage, float64 arithmetic; {secs:.1f} s of CPU time"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": dict(workload_config(wl, B), **({"profiling_only_layers": args.layers} if args.layers else {})),
            "exec_tflops": fexec_total / (total_ms / 1000.0) / 1e12,
            "exec_tflops_frac_of_peak": fexec_total / (total_ms / 1000.0) / 1e12 / peak,
            "per_budget": per_budget, "roofline": roofline, "kernels": kernels,
            "gpu_launches": int(launches), "gpu_launches_per_step": launches / args.steps,
            "wall_s_timed": t_wall, "clocks": clk.summary(), "e2e": e2e, "cpu_baseline": cpu,
            "hbm_kernels_sweep": hbm, "decode": dec, "fp8": fp8, "gated_workloads": gated,
        }
        # the full record first (no "metric" key), then the bench line:
        # required keys, roofline, clocks, e2e, CPU baseline and a compact
        # summary, short enough to survive a log tail
        print(json.dumps({"bench_details": line}), flush=True)
        keep = ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
                "vs_baseline", "dtype", "data", "gpu_launches", "roofline", "clocks", "e2e", "cpu_baseline")
        main_line = {k: line[k] for k in keep}
        main_line["summary"] = compact_summary(line, gated)
        main_line["exec_tflops"] = round(line["exec_tflops"], 1)
        main_line["config"] = {"workload": line["config"]["workload"], "batch": B,
                               "gates": line["config"]["gates"], "l2": line["config"]["l2"],
                               "parallelism": line["config"]["parallelism"]}
        main_line["roofline"] = {k: v for k, v in roofline.items() if k not in ("traffic_note", "timing")}
        main_line["cpu_baseline"] = dict(cpu, sample=cpu["sample"][:160]) if cpu else None
        print(json.dumps(main_line), flush=True)
    model.close()


def timed_steps(svl, model, batches, outs, steps, warmup, live_tags=("gateup_gemm",)):
    """`warmup` untimed steps, then `steps` steps cycling over `batches`,
    CUDA events around each step on the launching stream and around every
    launch of the kernels named in `live_tags` only. Fails on a non-zero
    device status word. Returns per-step ms, the live kernel times, the
    clock summary and the launch count of the timed steps."""
    stream = torch.cuda.current_stream()

    def step(i):
        model.run(batches[i % len(batches)], out=outs[i % len(batches)])

    for i in range(warmup):
        step(i)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    launches0 = svl.svl_launch_count()
    svl.svl_profile_start(model.handle, tags=list(live_tags))
    nv = NvmlClock(torch.cuda.current_device())
    windows = []
    with ClockSampler(torch.cuda.current_device()) as clk:
        for i in range(steps):
            tw0 = time.perf_counter()
            ev[i][0].record(stream)
            step(i)
            ev[i][1].record(stream)
            torch.cuda.synchronize()
            windows.append((tw0, time.perf_counter()))
    nv.close()
    live = svl.svl_profile_stop(model.handle)
    launches = svl.svl_launch_count() - launches0
    status = svl.svl_get_device_status(model.handle)
    if status:
        raise RuntimeError(f"device status {status:#x} in a timed pass")
    summary = clk.summary()
    summary["step_sm_mhz"] = [nv.median(a, b) for a, b in windows]
    return [a.elapsed_time(b) for a, b in ev], live, summary, launches


def batch_accounting(svl, model, dims, bt, out):
    """Input tokens, executed FLOPs (svl_flops: post-gating, causal
    attention, last-row LM head), per-kind FLOPs, mean k and the executed
    fraction alpha of the decoder's (layer, group) pairs of one batch."""
    k = out["k"].cpu().numpy()
    nv = (bt["vis_off"][1:] - bt["vis_off"][:-1]).cpu().numpy()
    st = (bt["text_off"][1:] - bt["text_off"][:-1]).cpu().numpy()
    lg, gg = bt["layer_gate"].cpu(), bt["group_gate"].cpu()
    on = effective_on(bt, dims)
    return {"tokens": int(nv.sum() + st.sum()), "fexec": executed_flops(svl, model.desc, k, st, nv, lg, gg),
            "kind": per_kind_flops(dims, k, st, lg.numpy(), gg.numpy()), "k_mean": float(k.mean()),
            "alpha": float(on.float().mean())}


def pass_summary(svl, model, dims, batches, outs, step_ms, live, pk, label_key=None, labels=None, step_mhz=None):
    """Per-batch rows (ms per step, tokens/s, executed TFLOP/s) and the
    whole pass: tokens/s, executed TFLOP/s and the gate/up GEMM's rate from
    the live events against the measured sustained bf16 peak."""
    peak = pk["bf16_tflops_sustained"]
    rows, tokens, fexec, kind = [], 0, 0.0, {}
    for j, bt in enumerate(batches):
        idx = list(range(j, len(step_ms), len(batches)))
        if not idx:
            continue
        acc = batch_accounting(svl, model, dims, bt, outs[j])
        ms = statistics.mean(step_ms[i] for i in idx)
        mhz = [step_mhz[i] for i in idx if step_mhz and step_mhz[i]]
        row = {"ms_per_step": round(ms, 3), "tokens_per_s": round(acc["tokens"] / (ms / 1e3), 1),
               "sm_mhz": statistics.median(mhz) if mhz else None,
               "mcycles_per_step": round(statistics.mean(step_ms[i] * step_mhz[i] / 1e3 for i in idx
                                                         if step_mhz[i]), 4) if mhz else None,
               "exec_tflops": round(acc["fexec"] / (ms / 1e3) / 1e12, 1),
               "exec_tflop_per_step": acc["fexec"] / 1e12, "k_mean": round(acc["k_mean"], 1),
               "alpha": round(acc["alpha"], 4)}
        if labels is not None:
            row[label_key] = labels[j]
        rows.append(row)
        tokens += acc["tokens"] * len(idx)
        fexec += acc["fexec"] * len(idx)
        for t, f in acc["kind"].items():
            kind[t] = kind.get(t, 0.0) + f * len(idx)
    total_s = sum(step_ms) / 1e3
    out = {"tokens_per_s": round(tokens / total_s, 1), "exec_tflops": round(fexec / total_s / 1e12, 1),
           "exec_frac_of_peak": round(fexec / total_s / 1e12 / peak, 4), "ms_per_step": sum(step_ms) / len(step_ms),
           "rows": rows}
    for tag in ("gateup_gemm", "attention"):
        if tag in live and kind.get(tag):
            n_l, t_l = live[tag]
            ach = kind[tag] / (t_l / 1e3) / 1e12
            out["roofline" if tag == "gateup_gemm" else "attention_roofline"] = {
                "kernel": tag, "bound": "tensor", "achieved": round(ach, 1), "peak": peak, "unit": "TFLOP/s",
                "frac": round(ach / peak, 4), "launches": n_l}
    return out


def scaling_vs(rows, key, ref_value):
    """t(x)/t(ref) / (F(x)/F(ref)) - 1 for each row, against the row whose
    `key` equals ref_value (linear scaling in executed FLOPs gives 0); the
    same with SM cycles (time x clock) in place of time when clocks exist."""
    ref = [r for r in rows if abs(r[key] - ref_value) < 1e-9]
    if not ref:
        return
    for r in rows:
        f = r["exec_tflop_per_step"] / ref[0]["exec_tflop_per_step"]
        r["time_vs_flops_ratio_minus_1"] = round((r["ms_per_step"] / ref[0]["ms_per_step"]) / f - 1.0, 4)
        if r.get("mcycles_per_step") and ref[0].get("mcycles_per_step"):
            r["cycles_vs_flops_ratio_minus_1"] = round((r["mcycles_per_step"] / ref[0]["mcycles_per_step"]) / f - 1.0,
                                                       4)


def gated_batch(wl, seed, dev, alpha=1.0, layer_skip=0.0, keep=288):
    """The mixed-serving batch shape (576 visual tokens, text U[16, 256]) at a
    fixed kept count, with exactly round(alpha * G) head groups on in every
    (sample, layer) -- which ones drawn at random -- and a fraction
    `layer_skip` of each sample's layers skipped (drawn at random)."""
    bt = synth.make_batch(wl, seed, budget=1.0, device="cpu")
    B, L, G = bt["B"], wl.dims.n_layers, wl.dims.n_groups
    g = torch.Generator().manual_seed(seed + 5)
    n_on = max(1, round(alpha * G))
    order = torch.rand(B, L, G, generator=g).argsort(dim=2)
    gg = (order < n_on).to(torch.uint8)
    lg = torch.ones(B, L, dtype=torch.uint8)
    n_skip = round(layer_skip * L)
    if n_skip:
        skip = torch.rand(B, L, generator=g).argsort(dim=1) < n_skip
        lg[skip] = 0
    bt["group_gate"], bt["layer_gate"] = gg, lg
    bt["keep_count"] = torch.full((B,), keep, dtype=torch.int32)
    return {k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in bt.items()}


def run_gated_workloads(args, svl, llava_model, dev, pk):
    """The other configurations of the benchmark suite, each with its own
    warm-up and timed steps (CUDA events, clocks sampled):

    * mixed serving (B = 64, text U[16, 256], per-sample budgets U[0.1, 1],
      head gates Bern(sqrt(b)) and layer skips, LLaVA-7B decoder);
    * a gating sweep on the mixed shape at a fixed kept count (288 of 576):
      head-group density alpha = 1, 0.75, 0.5, 0.25, and half the layers
      skipped -- wall time against executed FLOPs, which shows that gated-off
      heads, channels and layers are never issued;
    * video (B = 2, 8 x 576 visual tokens, budgets 0.1 / 0.25 / 0.5);
    * Qwen2-VL-7B shapes (B = 8, 256..2048 visual tokens, GQA 28/4, vocab
      152,064, per-sample budgets U[0.2, 1]), its own weights.
    """
    res = {}
    w_steps, t_steps = max(3, min(args.warmup, 3)), max(4, min(args.steps, 6))
    dims = llava_model.dims
    wl_m = synth.WORKLOADS["mixed"]
    bts = [synth.make_batch(wl_m, SEED + 301 + i, device=dev) for i in range(2)]
    outs = [llava_model.alloc_outputs(bt) for bt in bts]
    ms, live, clk, _ = timed_steps(svl, llava_model, bts, outs, t_steps, w_steps)
    res["mixed"] = dict(pass_summary(svl, llava_model, dims, bts, outs, ms, live, pk,
                                     step_mhz=clk.pop("step_sm_mhz")), clocks=clk)
    del outs
    # gating sweep at fixed k
    points = [("alpha", 1.0, 0.0), ("alpha", 0.75, 0.0), ("alpha", 0.5, 0.0), ("alpha", 0.25, 0.0),
              ("layer_skip", 1.0, 0.5)]
    rows = []
    for kind, alpha, skip in points:
        bt = gated_batch(wl_m, SEED + 401, dev, alpha=alpha, layer_skip=skip)
        out = [llava_model.alloc_outputs(bt)]
        ms, live, clk, _ = timed_steps(svl, llava_model, [bt], out, max(3, t_steps // 2), 2)
        r = pass_summary(svl, llava_model, dims, [bt], out, ms, live, pk, step_mhz=clk.pop("step_sm_mhz"))["rows"][0]
        r["point"] = f"{kind} {alpha if kind == 'alpha' else skip}"
        rows.append(r)
    ref = rows[0]
    for r in rows:
        r["t_over_t1"] = round(r["ms_per_step"] / ref["ms_per_step"], 4)
        r["f_over_f1"] = round(r["exec_tflop_per_step"] / ref["exec_tflop_per_step"], 4)
        r["time_vs_flops_ratio_minus_1"] = round(r["t_over_t1"] / r["f_over_f1"] - 1.0, 4)
        if r.get("mcycles_per_step") and ref.get("mcycles_per_step"):
            r["cycles_vs_flops_ratio_minus_1"] = round(
                (r["mcycles_per_step"] / ref["mcycles_per_step"]) / r["f_over_f1"] - 1.0, 4)
    res["gating_sweep"] = {"batch": "mixed shape, B=64, keep 288 of 576, layer gates on unless skipped",
                           "rows": rows}
    # video
    wl_v = synth.WORKLOADS["video"]
    bts = [synth.make_batch(wl_v, SEED + 501, budget=b, device=dev) for b in wl_v.budgets]
    outs = [llava_model.alloc_outputs(bt) for bt in bts]
    ms, live, clk, _ = timed_steps(svl, llava_model, bts, outs, 2 * len(bts), w_steps,
                                   live_tags=("gateup_gemm", "attention"))
    v = pass_summary(svl, llava_model, dims, bts, outs, ms, live, pk, "budget", list(wl_v.budgets),
                     step_mhz=clk.pop("step_sm_mhz"))
    scaling_vs(v["rows"], "budget", 0.5)
    v["clocks"] = clk
    res["video"] = v
    del outs
    # Qwen2-VL-7B shapes
    wl_q = synth.WORKLOADS["qwen"]
    wq = synth.make_weights(wl_q.dims, SEED + 7, device=dev)
    mq = svl.GatedPrefill(wl_q.dims, wq, max_seq=wl_q.n_vis[1] + wl_q.s_text[1] + 64)
    bts = [synth.make_batch(wl_q, SEED + 601 + i, device=dev) for i in range(2)]
    outs = [mq.alloc_outputs(bt) for bt in bts]
    ms, live, clk, _ = timed_steps(svl, mq, bts, outs, t_steps, w_steps)
    res["qwen"] = dict(pass_summary(svl, mq, wl_q.dims, bts, outs, ms, live, pk, step_mhz=clk.pop("step_sm_mhz")),
                       clocks=clk)
    mq.close()
    del wq, outs, mq
    torch.cuda.empty_cache()
    return res


def compact_summary(line, gated):
    """The figures a reader needs first, small enough for a log tail."""
    s = {"per_budget": [[p["budget"], round(p["ms_per_step"], 2), round(p.get("time_vs_flops_ratio_minus_1", 0), 4),
                         p.get("sm_mhz"), round(p["cycles_vs_flops_ratio_minus_1"], 4)
                         if p.get("cycles_vs_flops_ratio_minus_1") is not None else None]
                        for p in line["per_budget"]],
         "per_budget_cols": ["budget", "ms_per_step", "t_vs_F_minus_1", "sm_mhz", "cycles_vs_F_minus_1"]}
    kern = line.get("kernels", {})
    s["tflops"] = {t: round(kern[t]["tflops"]) for t in ("qkv_gemm", "o_gemm", "gateup_gemm", "down_gemm", "attention")
                   if t in kern and "tflops" in kern[t]}
    if line.get("hbm_kernels_sweep"):
        s["hbm_frac"] = {f"B{r['batch']}": {n: r[n]["frac_of_measured_hbm"] for n in ("score", "select", "pack")
                                            if n in r} for r in line["hbm_kernels_sweep"]}
    if gated:
        m = gated["mixed"]
        s["mixed"] = [m["tokens_per_s"], m["exec_tflops"], m.get("roofline", {}).get("frac")]
        s["gating_sweep"] = [[r["point"], r["t_over_t1"], r["f_over_f1"], r["time_vs_flops_ratio_minus_1"],
                              r.get("cycles_vs_flops_ratio_minus_1")] for r in gated["gating_sweep"]["rows"]]
        v = gated["video"]
        s["video"] = [[r["budget"], r["ms_per_step"], r.get("time_vs_flops_ratio_minus_1"),
                       r.get("cycles_vs_flops_ratio_minus_1")] for r in v["rows"]]
        s["video_attention_tflops"] = v.get("attention_roofline", {}).get("achieved")
        q = gated["qwen"]
        s["qwen"] = [q["tokens_per_s"], q["exec_tflops"], q.get("roofline", {}).get("frac")]
    if line.get("fp8"):
        f = line["fp8"]
        s["fp8"] = [round(f["value"]), round(f["exec_tflops"]), round(f["gateup_gemm"]["frac"], 3)]
    if line.get("decode"):
        s["decode"] = [round(line["decode"]["tokens_per_s"]), round(line["decode"]["frac_of_measured_hbm"], 3)]
    return s


def run_fp8(args, svl, wl, weights, batches, dev, pk, max_seq):
    """The same workload with SVL_GEMM_E4M3: the four gated projections on
    e4m3 operands (per-channel weight and per-row activation scales). Not the
    headline (reduced precision): its own tokens/s, executed TFLOP/s against
    the fp8 peak (measured bf16 sustained peak x 2, the nominal fp8/bf16
    ratio), the per-kernel breakdown including the activation quantisation,
    and e4m3 decode."""
    dims = wl.dims
    model = svl.GatedPrefill(dims, weights, max_seq=max_seq, gemm_format=svl.SVL_GEMM_E4M3)
    outs = [model.alloc_outputs(bt) for bt in batches]
    stream = torch.cuda.current_stream()

    def step(i):
        model.run(batches[i % len(batches)], out=outs[i % len(batches)])

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    status = svl.svl_get_device_status(model.handle)
    if status:
        raise RuntimeError(f"device status {status:#x} in the e4m3 pass")
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    svl.svl_profile_start(model.handle, tags=["gateup_gemm"])
    with ClockSampler(torch.cuda.current_device()) as clk:
        for i in range(args.steps):
            ev[i][0].record(stream)
            step(i)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
    live = svl.svl_profile_stop(model.handle)
    svl.svl_profile_start(model.handle)
    for i in range(args.steps):
        step(i)
    kern = svl.svl_profile_stop(model.handle)
    step_ms = [a.elapsed_time(b) for a, b in ev]
    tokens, fexec, kind = 0, 0.0, {}
    per_budget = []
    for j, bt in enumerate(batches):
        idx = list(range(j, args.steps, len(batches)))
        if not idx:
            continue
        k = outs[j]["k"].cpu().numpy()
        nv = (bt["vis_off"][1:] - bt["vis_off"][:-1]).cpu().numpy()
        st = (bt["text_off"][1:] - bt["text_off"][:-1]).cpu().numpy()
        lg, gg = bt["layer_gate"].cpu(), bt["group_gate"].cpu()
        toks = int(nv.sum() + st.sum())
        fex = executed_flops(svl, model.desc, k, st, nv, lg, gg)
        ms = statistics.mean(step_ms[i] for i in idx)
        per_budget.append({"budget": float(bt["budget"][0]), "ms_per_step": ms, "tokens_per_s": toks / (ms / 1e3),
                           "exec_tflops": fex / (ms / 1e3) / 1e12})
        tokens += toks * len(idx)
        fexec += fex * len(idx)
        for kk, v in per_kind_flops(dims, k, st, lg.numpy(), gg.numpy()).items():
            kind[kk] = kind.get(kk, 0.0) + v * len(idx)
    total_ms = sum(step_ms)
    peak8 = 2.0 * pk["bf16_tflops_sustained"]
    n_l, t_l = live["gateup_gemm"]
    gu = kind["gateup_gemm"] / (t_l / 1e3) / 1e12
    tot_k = max(sum(v[1] for v in kern.values()), 1e-9)
    kernels = {t: {"launches": n, "total_ms": ms, "share": ms / tot_k}
               for t, (n, ms) in sorted(kern.items(), key=lambda kv: -kv[1][1])}
    for t in kind:
        if t in kernels:
            kernels[t]["tflops"] = kind[t] / (kernels[t]["total_ms"] / 1e3) / 1e12
    dec = None
    if not args.no_decode:
        dec = run_decode(svl, model, batches[1], dims, dev, pk, layer_weight_bytes=1)
    model.close()
    return {"gemm_format": "e4m3 (gated projections; projector, token controller, attention, LM head bf16)",
            "value": tokens / (total_ms / 1e3), "unit": "tokens/s", "ms_per_step": total_ms / args.steps,
            "exec_tflops": fexec / (total_ms / 1e3) / 1e12,
            "exec_tflops_frac_of_fp8_peak": fexec / (total_ms / 1e3) / 1e12 / peak8,
            "fp8_peak_tflops": peak8, "fp8_peak_source": pk["source"] + " bf16 sustained x 2 (nominal fp8/bf16)",
            "gateup_gemm": {"launches": n_l, "avg_launch_ms": t_l / n_l, "tflops": gu, "frac": gu / peak8},
            "per_budget": per_budget, "kernels": kernels, "clocks": clk.summary(), "decode": dec}


def run_decode(svl, model, bt, dims, dev, pk, steps=16, warm=3, layer_weight_bytes=2):
    """Gated decode after a KV-cache prefill of the budget-0.5 batch: tokens
    per second over `steps` teacher-forced steps (CUDA events) and the bytes
    each step must read -- every weight of the active groups once plus the
    cached keys and values of the active heads -- against the measured HBM
    bandwidth (decode is bound by streaming them)."""
    B = bt["B"]
    nv, nt = int(bt["vis"].shape[0]), int(bt["text_ids"].shape[0])
    out = model.run(bt, stages=("select", "pack"))
    max_len = nv // B + nt // B + steps + warm + 8
    ws, wsb = model.workspace(B, nv, nt, dev, ("prefill",))
    kv = torch.empty(svl.svl_kv_cache_size(model.handle, B, max_len), dtype=torch.uint8, device=dev)
    cache_len = torch.zeros(B, dtype=torch.int32, device=dev)
    svl.svl_gated_prefill_kv(model.handle, B, nv + nt, out["X"], out["cu_seqlens"], out["pos"], bt["layer_gate"],
                             bt["group_gate"], svl.SVL_LOGITS_LAST, out["logits"], kv, max_len, cache_len, ws, wsb)
    dws = torch.empty(svl.svl_decode_workspace_size(model.handle, B), dtype=torch.uint8, device=dev)
    g = torch.Generator(device=dev).manual_seed(SEED + 99)
    fed = torch.randint(0, dims.vocab, (warm + steps, B), generator=g, device=dev, dtype=torch.int32)
    logits = torch.empty(B, dims.vocab, dtype=torch.float32, device=dev)
    nxt = torch.empty(B, dtype=torch.int32, device=dev)
    for t in range(warm):
        svl.svl_decode_step(model.handle, B, fed[t], kv, max_len, cache_len, bt["layer_gate"], bt["group_gate"],
                            logits, nxt, dws, dws.numel())
    torch.cuda.synchronize()
    len0 = cache_len.clone()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for t in range(warm, warm + steps):
        svl.svl_decode_step(model.handle, B, fed[t], kv, max_len, cache_len, bt["layer_gate"], bt["group_gate"],
                            logits, nxt, dws, dws.numel())
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    # device time per kernel kind over a few more steps (events around every launch)
    svl.svl_profile_start(model.handle)
    for t in range(warm):
        svl.svl_decode_step(model.handle, B, fed[t], kv, max_len, cache_len, bt["layer_gate"], bt["group_gate"],
                            logits, nxt, dws, dws.numel())
    kern = svl.svl_profile_stop(model.handle)
    kernel_ms = {k: round(v[1] / warm, 4) for k, v in sorted(kern.items(), key=lambda kv: -kv[1][1])}
    d = dims
    dh = d.d_model // d.n_heads
    on = effective_on(bt, d)  # active (layer, group) pairs per sample
    per_group = d.d_model * (d.n_heads * dh * 2 + 2 * d.n_kv_heads * dh) // d.n_groups + 3 * d.d_model * d.d_ffn // d.n_groups
    # groups active in any sample (e4m3 models: one byte per gated-projection weight)
    w_bytes = layer_weight_bytes * int(on.any(dim=0).sum()) * per_group + 2 * d.vocab * d.d_model
    ctx = float((len0.double() + steps / 2).mean())
    kv_bytes = 2 * 2 * float(on.sum()) * (d.n_kv_heads // d.n_groups) * dh * ctx
    nbytes = w_bytes + kv_bytes
    return {"batch": B, "steps": steps, "ms_per_step": ms, "tokens_per_s": B / (ms / 1000.0),
            "context_mean": ctx, "bytes_per_step": nbytes, "gb_s": nbytes / (ms / 1000.0) / 1e9,
            "frac_of_measured_hbm": nbytes / (ms / 1000.0) / 1e9 / pk["hbm_gbs"],
            "kernel_ms_per_step_profiled": kernel_ms,
            "note": "teacher-forced, budget-0.5 batch, prefill gates; bytes = active-group weights once "
                    "(shared by the batch) + cached K/V of the active heads"}


def effective_on(bt, d):
    """[B, L, G] bool: group j of layer l runs for sample b (prefix layers always)."""
    lg = bt["layer_gate"].bool()[:, :, None]
    gg = bt["group_gate"].bool()
    on = lg & gg
    on[:, :d.n_prefix, :] = True
    return on.cpu()


def run_hbm_sweep(svl, model, wl, dev, pk, reps=5, mults=(1, 4, 16)):
    """Token controller and pack alone at 1x, 4x and 16x the benchmark batch
    (budget 0.5): achieved bandwidth of the HBM-bound kernels from their
    algorithmic bytes and CUDA-event times."""
    d = wl.dims
    out = []
    for mult in mults:
        B = wl.batch * mult
        bt = synth.make_batch(wl, SEED + 7 + mult, budget=0.5, batch=B, device=dev)
        o = model.alloc_outputs(bt)
        for _ in range(2):
            model.run(bt, out=o, stages=("select", "pack"))
        torch.cuda.synchronize()
        svl.svl_profile_start(model.handle)
        for _ in range(reps):
            model.run(bt, out=o, stages=("select", "pack"))
        kern = svl.svl_profile_stop(model.handle)
        nv = int(bt["vis"].shape[0])
        nt = int(bt["text_ids"].shape[0])
        k = int(o["k"].sum())
        rows = {
            # visual features read + logits written
            "score": (2 * nv * d.c_vis + 4 * nv, kern.get("score")),
            # logits read + kept indices written
            "select": (4 * nv + 4 * k + 4 * B, kern.get("select")),
            # kept features gathered to the projector staging rows, text embedding rows copied
            "pack": (2 * (2 * k * d.c_vis) + 2 * (2 * nt * d.d_model) + 4 * nt + 8 * (nv + nt), kern.get("pack")),
        }
        line = {"batch": B, "visual_tokens": nv, "kept": k}
        for name, (nbytes, km) in rows.items():
            if km is None:
                continue
            ms = km[1] / reps
            gbs = nbytes / (ms / 1000.0) / 1e9
            line[name] = {"ms": round(ms, 4), "bytes": nbytes, "gb_s": round(gbs, 1),
                          "frac_of_measured_hbm": round(gbs / pk["hbm_gbs"], 3),
                          "launches": km[0] // reps}
        out.append(line)
        del bt, o
        torch.cuda.empty_cache()
    return out


def run_e2e(args, svl, model, batches, dims, world, dev):
    stream = torch.cuda.current_stream()
    hosts = []
    for bt in batches:
        h = {k: (v.cpu().pin_memory() if isinstance(v, torch.Tensor) else v) for k, v in bt.items()}
        h["logits"] = torch.empty(bt["B"], dims.vocab, dtype=torch.float32).pin_memory()
        h["k"] = torch.empty(bt["B"], dtype=torch.int32).pin_memory()
        hosts.append(h)
    nv = batches[0]["vis"].shape[0]
    nt = int(batches[0]["text_ids"].shape[0])
    B = batches[0]["B"]
    need = svl.svl_host_workspace_size(model.handle, B, nv, nt)
    ws = torch.empty(need, dtype=torch.uint8, device=dev)

    def step(i):
        h = hosts[i % len(hosts)]
        svl.svl_prefill_from_host(model.handle, B, nv, nt, h["vis"], h["vis_off"], h["text_ids"], h["text_off"],
                                  h["budget"], h["keep_count"], h["layer_gate"], h["group_gate"], h["logits"],
                                  h["k"], ws, need, stream)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for i in range(args.steps):
        step(i)
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b)
    tokens = sum(int(hosts[i % len(hosts)]["vis"].shape[0] + hosts[i % len(hosts)]["text_ids"].shape[0])
                 for i in range(args.steps))
    h0 = hosts[0]
    h2d = sum(int(h0[k].numel() * h0[k].element_size()) for k in
              ("vis", "vis_off", "text_ids", "text_off", "budget", "keep_count", "layer_gate", "group_gate"))
    d2h = int(h0["logits"].numel() * 4 + h0["k"].numel() * 4)
    (ms,), (tokens,) = job_aggregate([ms], [tokens], dev)
    return {"value": tokens / (ms / 1000.0), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "entry_point": "svl_prefill_from_host (pinned host buffers)"}


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    try:
        run_ours(args, rank, world, local_rank)
    finally:
        if world > 1:
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
