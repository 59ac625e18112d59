"""Benchmark of the budget-routed decode step (one JSON line on stdout).

python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                [--workload NAME] [--no-graph]

Default workload: Llama-3-8B shape, bf16, batch 1, context 2048, budget k = 15
of 30 middle layers (the configuration the headline metric is quoted on).  The
default run also times the other bf16 workloads (Llama-3-8B B=64 mixed
budgets, Llama-2-13B B=32, Qwen2.5-7B B=256), each over its own step count,
and reports them under "per_config".
A step = one budget-routed decode step of the whole batch (layer 0, router,
compaction, the selected middle layers on their sub-batches, last layer).
Inputs (weights 14 GB, KV cache) are resident in HBM and larger than L2.

For N > 1 (torchrun) every rank runs an independent replica of the workload on
its own GPU (weak scaling); the only cross-rank traffic is a barrier and the
max-over-ranks of the timed region.  `--impl reference` times the CPU oracle
on the host cores instead (rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "budget-routed decode tokens/s at 1 GB300 per budget; % of HBM/tensor roofline"
# ncu dram bytes (read + write) per launch of the dominant kernel, from the
# committed ncu summary of the gate/up GEMM (3-layer model with the same layer
# shapes as the 32-layer bench workload); absent for kernels not captured
NCU_TRAFFIC_PER_LAUNCH = {("llama3-8b-b1", "gemm_gate_up"): 238031616}
# DRAM traffic per algorithmic byte where the capture was a smaller case of
# the same kernel whose traffic grows with the bytes it processes: the
# attention of the 3-layer Qwen2.5-7B B=256 model (1,200,036,736 bytes of
# traffic for 1,192,611,840 algorithmic bytes per launch)
NCU_TRAFFIC_RATIO = {("qwen2.5-7b-b256", "attention"): 1200036736 / 1192611840}


def _ncu_traffic(workload, kernel, bytes_per_launch):
    if (workload, kernel) in NCU_TRAFFIC_PER_LAUNCH:
        return NCU_TRAFFIC_PER_LAUNCH[(workload, kernel)]
    if (workload, kernel) in NCU_TRAFFIC_RATIO:
        return int(round(NCU_TRAFFIC_RATIO[(workload, kernel)] * bytes_per_launch))
    return None
DEFAULT_WORKLOAD = "llama3-8b-b1"
PER_CONFIG = ["llama3-8b-b64-mixed", "llama2-13b-b32", "qwen2.5-7b-b256"]
PREFILL_WORKLOAD = "llama3-8b-prefill-b16"


def _peak_tflops_burst():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"])
    except Exception:
        return 1900.0


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "20"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for line in (self.out or "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append((float(f[1]), float(f[2]), f[5:9]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        mx = max(r[1] for r in rows)
        load = [r for r in rows if r[0] > 0.5 * mx] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for r in rows for j in range(4) if r[2][j].lower() == "active"})
        return {"sm_mhz": float(np.median([r[0] for r in load])), "sm_max_mhz": mx,
                "reasons": reasons, "samples": len(rows)}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _max_over_ranks(x: float, ws: int, device) -> float:
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(local_ms: float, tokens_per_rank: int, ws: int, device="cpu"):
    """Whole-job throughput of independent replicas: every rank processed
    `tokens_per_rank` tokens; the job took the slowest rank's time."""
    ms = _max_over_ranks(local_ms, ws, device)
    return ms, ws * tokens_per_rank / (ms / 1e3)


def _barrier(ws: int):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------------------
# CPU oracle sample (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------
def oracle_sample(w, n_layers_sample=None, steps=1, device="cuda"):
    """Times the oracle on one sequence of the workload for `steps` decode
    steps.  Weights/KV come from the shared generator (generated on `device`
    and copied to host; that preparation is excluded).  If n_layers_sample is
    given, each step runs layer 0, the router, the first n_layers_sample
    selected middle layers and the last layer: a step then counts as the
    fraction (executed blocks of the sample) / (executed blocks of the full
    routed step) of a token."""
    import torch

    from oracle import adapter as A
    from oracle import buddy_oracle as O
    from workloads import synth

    s = w.shape
    seq = 0
    prep = {"t": 0.0}

    def src(l):
        t0 = time.perf_counter()
        out = {k: v.cpu() for k, v in synth.layer_weights(s, w.seed, l, device).items()}
        prep["t"] += time.perf_counter() - t0
        return out

    model = A.build_model(s, w.seed, layer_source=src,
                          dm_source=lambda: {k: v.cpu() for k, v in synth.dm_weights(s, w.seed, device).items()},
                          cache_layers=2)
    t0 = time.perf_counter()
    st = A.build_state(s, w.seed, [int(w.contexts()[seq])], seqs=[0], gen_device=device)
    prep["t"] += time.perf_counter() - t0
    k = [int(w.budgets()[seq])]
    seconds, tokens, per_step = 0.0, 0.0, []
    for t in range(steps):
        h = A.to_f64(synth.h_in(s, w.seed, t, [seq], device))
        prep0 = prep["t"]
        info = {}

        def truncate(rr):
            info["full"] = len(rr.sel[0])
            keep = rr.sel[0][:n_layers_sample]
            info["keep"] = len(keep)
            return [keep]

        t0 = time.perf_counter()
        O.decode_step(model, st, h, k, override_sel=truncate if n_layers_sample is not None else None)
        dt = time.perf_counter() - t0 - (prep["t"] - prep0)
        frac = 1.0 if n_layers_sample is None else (info["keep"] + 2) / (info["full"] + 2)
        seconds += dt
        tokens += frac
        per_step.append(dt)
    return {"seconds": seconds, "tokens": tokens, "per_step": per_step, "cores": os.cpu_count()}


def class_bytes(s, masks, ctxs, B):
    """Algorithmic bytes per kernel class over the profiled steps: weights of
    every launched layer, activations in and out, KV read by attention."""
    esz = s.elem_bytes
    d, F, qd, kvd, N = s.d_model, s.ffn_dim, s.q_dim, s.kv_dim, s.qkv_dim
    out = {"gemm_gate_up": 0, "gemm_down": 0, "gemm_qkv": 0, "gemm_o": 0, "attention": 0, "rmsnorm": 0}
    for m_, n_ in zip(masks, ctxs):
        rows = m_.sum(axis=0)
        for l in range(s.n_layers):
            m = int(rows[l])
            if m == 0:
                continue
            out["gemm_gate_up"] += 2 * F * d * esz + m * (d + F) * esz
            out["gemm_down"] += F * d * esz + m * (F * esz + 8 * d)
            out["gemm_qkv"] += N * d * esz + m * (d * esz + 4 * N)
            out["gemm_o"] += qd * d * esz + m * (qd * esz + 8 * d)
            sel = np.nonzero(m_[:, l])[0]
            out["attention"] += int(2 * kvd * esz * (n_[:B][sel] + 1).sum()) + m * qd * (4 + esz)
            out["rmsnorm"] += 2 * m * d * (4 + esz)
    return out


# ---------------------------------------------------------------------------
# Our arm
# ---------------------------------------------------------------------------
NOMINAL_HBM_GBS = 7900.0   # GB300 HBM3e, nominal (context for the measured-peak fractions)


def measure(w, K, W, dev, ws, local, use_graph=True, e2e=True):
    """Times K budget-routed decode steps of workload w (after W warm-up
    steps) on device `dev`, then profiles kernel classes over a few more
    direct-launch steps and (optionally) times the host-buffer entry point."""
    import torch

    from workloads import cost
    from workloads import device as D
    from workloads import synth

    s = w.shape
    B = w.batch
    prof_steps = min(K, 8)
    e2e_steps = K if e2e else 0
    extra = W + K + prof_steps + e2e_steps + 2
    dw = D.build(w, device=dev, extra_steps=extra, use_graph=use_graph)
    ctx, kv = dw.ctx, dw.kv
    n_steps_total = W + K + prof_steps + e2e_steps
    h_all = [synth.h_in(s, w.seed, t, range(B), dev) for t in range(n_steps_total)]
    # the step input lives in one resident buffer (as a serving loop would keep
    # it); each step's new hidden states are copied into it inside the step
    h_buf = torch.empty(B, s.d_model, device=dev)
    h_out = torch.empty(B, s.d_model, device=dev)
    count = torch.empty(s.n_layers, dtype=torch.int32, device=dev)
    mask = torch.empty(B, s.n_layers, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    # warm-up (also captures the graph)
    step = 0
    for _ in range(W):
        h_buf.copy_(h_all[step], non_blocking=True)
        ctx.buddy_decode_step(kv, h_buf, dw.k, h_out, mask, None, count)
        step += 1
    torch.cuda.synchronize(dev)
    if ctx.buddy_device_status() != 0:
        raise RuntimeError("device error flag during warm-up")

    # timed region: K steps, positions advancing
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        _barrier(ws)
        torch.cuda.synchronize(dev)
        start.record(stream)
        for t in range(K):
            h_buf.copy_(h_all[step], non_blocking=True)
            ctx.buddy_decode_step(kv, h_buf, dw.k, h_out, mask, None, count)
            step += 1
        end.record(stream)
        torch.cuda.synchronize(dev)
        _barrier(ws)
    ms = start.elapsed_time(end)
    ms_max, value = aggregate(ms, B * K, ws, dev)
    if ctx.buddy_device_status() != 0:
        raise RuntimeError("device error flag in timed region")

    # instrumented pass: per-kernel-class CUDA events (direct launches)
    ctx.buddy_set_options(False)
    ctx.buddy_set_profiling(True)
    ctx.buddy_profile_read()
    prof_masks, prof_ctx = [], []
    for t in range(prof_steps):
        prof_ctx.append(kv.len.cpu().numpy().copy())
        h_buf.copy_(h_all[step], non_blocking=True)
        ctx.buddy_decode_step(kv, h_buf, dw.k, h_out, mask, None, count)
        torch.cuda.synchronize(dev)
        prof_masks.append(mask.cpu().numpy().copy())
        step += 1
    prof = ctx.buddy_profile_read()
    ctx.buddy_set_profiling(False)
    ctx.buddy_set_options(use_graph)

    e2e_out = None
    if e2e:
        # end to end through the host-buffer entry point (pinned buffers)
        h_host = [h.cpu().pin_memory() for h in h_all[step:step + e2e_steps]]
        k_host = dw.k.cpu().pin_memory()
        o_host = torch.empty(B, s.d_model).pin_memory()
        m_host = torch.empty(B, s.n_layers, dtype=torch.uint8).pin_memory()
        ctx.buddy_decode_step_host(kv, h_host[0], k_host, o_host, m_host)   # graph for the staging buffers
        step += 1
        _barrier(ws)
        t0 = time.perf_counter()
        for t in range(1, e2e_steps):
            ctx.buddy_decode_step_host(kv, h_host[t], k_host, o_host, m_host)
        e2e_s = time.perf_counter() - t0
        e2e_s = _max_over_ranks(e2e_s, ws, dev)
        e2e_out = {"value": round(ws * B * (e2e_steps - 1) / e2e_s, 2), "unit": "tokens/s",
                   "h2d_bytes_per_step": B * s.d_model * 4 + B * 4,
                   "d2h_bytes_per_step": B * s.d_model * 4 + B * s.n_layers}

    # algorithmic cost of the profiled steps (realised masks and lengths)
    hbm, tflops, peak_src = _peaks()
    c_sum = {"bytes": 0, "flops": 0, "weight_bytes": 0, "kv_read_bytes": 0}
    for m_, n_ in zip(prof_masks, prof_ctx):
        c = cost.step_cost(s, m_, n_[:B])
        for key in c_sum:
            c_sum[key] += c[key]
    # dominant kernel class and its algorithmic bytes (summed over the profiled steps)
    dom = max(prof, key=lambda k: prof[k][0])
    per_class_bytes = class_bytes(s, prof_masks, prof_ctx, B)
    roof = None
    if dom in per_class_bytes and prof[dom][1] > 0:
        launches = prof[dom][1]
        bytes_per_launch = per_class_bytes[dom] / launches
        avg_s = prof[dom][0] / 1e3 / launches
        ach = bytes_per_launch / avg_s / 1e9
        roof = {"bound": "hbm", "kernel": dom, "achieved": round(ach, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(ach / hbm, 4), "traffic": _ncu_traffic(w.name, dom, bytes_per_launch),
                "bytes_per_launch": int(bytes_per_launch), "avg_launch_us": round(avg_s * 1e6, 2),
                "launches": launches, "peak_source": f"{peak_src} hbm_gbs",
                "frac_of_nominal": round(ach / NOMINAL_HBM_GBS, 4)}
    t_roof = max(c_sum["bytes"] / (hbm * 1e9), c_sum["flops"] / (tflops * 1e12)) / prof_steps
    t_roof_nom = max(c_sum["bytes"] / (NOMINAL_HBM_GBS * 1e9), c_sum["flops"] / (tflops * 1e12)) / prof_steps
    step_ms = ms_max / K
    # router + compaction per step (direct-launch events) over the graph step time
    route_ms = (prof["route"][0] + prof["compact"][0]) / prof_steps
    launches_per_step = sum(v[1] for v in prof.values()) / prof_steps
    # the timed steps launch every routed layer (a layer no row selected exits
    # at once); the profiled steps launch only the selected ones
    per_layer = ("rmsnorm", "gemm_qkv", "qkv_finalize", "attention", "gemm_o", "gemm_gate_up", "gemm_down",
                 "gemm_fixup")
    exec_layers = prof.get("attention", (0, 0))[1] / prof_steps
    per_layer_kernels = sum(prof.get(k, (0, 0))[1] for k in per_layer) / max(exec_layers * prof_steps, 1)
    graph_extra = max(s.n_layers - exec_layers, 0) * per_layer_kernels
    out = {
        "value": round(value, 2), "unit": "tokens/s", "ms_per_step": round(step_ms, 4), "steps": K,
        "warmup": W, "dtype": s.dtype,
        "config": {"workload": w.name, "model": s.name, "batch": B, "ctx": w.ctx_args,
                   "k": w.k_args, "layers": s.n_layers, "parallelism": f"replicas x{ws}", "graph": use_graph,
                   "l2": "inputs larger than L2 (per-step weight stream %.1f GB)"
                         % (c_sum["weight_bytes"] / prof_steps / 1e9)},
        "paths": ctx.buddy_get_paths(),
        "roofline": roof,
        "step_roofline": {"t_roof_ms": round(t_roof * 1e3, 4), "frac": round(t_roof * 1e3 / step_ms, 4),
                          "frac_of_nominal_hbm": round(t_roof_nom * 1e3 / step_ms, 4),
                          "bytes_per_step": int(c_sum["bytes"] / prof_steps),
                          "flops_per_step": int(c_sum["flops"] / prof_steps), "peak_gbs": hbm,
                          "nominal_gbs": NOMINAL_HBM_GBS, "peak_source": peak_src},
        "route_compact_ms_per_step": round(route_ms, 4),
        "route_compact_frac": round(route_ms / step_ms, 4),
        "kernel_ms_per_step": {k: round(v[0] / prof_steps, 4) for k, v in prof.items() if v[1] > 0},
        "kernel_gbs": {k: round(per_class_bytes[k] / (prof[k][0] / 1e3) / 1e9, 1)
                       for k in per_class_bytes if prof[k][0] > 0},
        "e2e": e2e_out,
        "gpu_launches": int(round((launches_per_step + graph_extra) * K)),
        "clocks": clk.summary(),
    }
    ctx.close()
    del dw, kv, ctx, h_all
    torch.cuda.empty_cache()
    return out


def measure_prefill(w, K, W, dev, ws, local):
    """Times K routed prefill calls of workload w's prompts (fresh sequences:
    positions are reset before each call, as a server reuses a slot) after W
    warm-up calls, then one profiled call for the kernel classes."""
    import torch

    from workloads import configs as C
    from workloads import cost
    from workloads import device as D
    from workloads import synth

    s = w.shape
    lengths = [int(v) for v in C.prompt_lengths(w)]
    T = int(sum(lengths))
    dw = D.build(w, device=dev, extra_steps=max(lengths) + 2, max_prefill_tokens=T)
    ctx, kv = dw.ctx, dw.kv
    x = synth.prompt_inputs(s, w.seed, lengths, dev)
    h_out = torch.empty(T, s.d_model, device=dev)
    mask = torch.empty(w.batch, s.n_layers, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def call():
        kv.len.zero_()
        ctx.buddy_prefill(kv, lengths, x, dw.k, h_out, mask)

    for _ in range(W):
        call()
    torch.cuda.synchronize(dev)
    if ctx.buddy_device_status() != 0:
        raise RuntimeError("device error flag during prefill warm-up")
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        _barrier(ws)
        torch.cuda.synchronize(dev)
        start.record(stream)
        for _ in range(K):
            call()
        end.record(stream)
        torch.cuda.synchronize(dev)
        _barrier(ws)
    ms = start.elapsed_time(end)
    ms_max, value = aggregate(ms, T * K, ws, dev)
    ctx.buddy_set_profiling(True)
    ctx.buddy_profile_read()
    call()
    torch.cuda.synchronize(dev)
    prof = ctx.buddy_profile_read()
    ctx.buddy_set_profiling(False)
    m = mask.cpu().numpy()
    c = cost.prefill_cost(s, m, lengths, [0] * w.batch)
    hbm, _, _ = _peaks()
    burst = _peak_tflops_burst()
    call_ms = ms_max / K
    gemm_ms = prof["pf_gemm"][0]
    out = {"workload": w.name, "value": round(value, 1), "unit": "tokens/s", "ms_per_call": round(call_ms, 3),
           "calls": K, "warmup": W, "prompts": w.batch, "tokens_per_call": T,
           "prompt_lengths": lengths, "k": w.k_args,
           "tflops_per_call": round(c["flops"] / 1e12, 3),
           "achieved_tflops": round(c["flops"] / (call_ms / 1e3) / 1e12, 1),
           "roofline": {"bound": "tensor", "kernel": "pf_gemm",
                        "achieved": round(c["gemm_flops"] / (gemm_ms / 1e3) / 1e12, 1) if gemm_ms > 0 else None,
                        "peak": burst, "unit": "TFLOP/s",
                        "frac": round(c["gemm_flops"] / (gemm_ms / 1e3) / 1e12 / burst, 4) if gemm_ms > 0 else None,
                        "traffic": None, "flops_per_call": c["gemm_flops"], "peak_source": "measured bf16_tflops"},
           "call_roofline_frac": round(max(c["flops"] / (burst * 1e12), c["bytes"] / (hbm * 1e9)) * 1e3 / call_ms, 4),
           "kernel_ms_per_call": {k: round(v[0], 4) for k, v in prof.items() if v[1] > 0},
           "paths": ctx.buddy_get_paths(), "clocks": clk.summary()}
    ctx.close()
    del dw, kv, ctx, x, h_out
    torch.cuda.empty_cache()
    return out


def run_ours(args, ws, rank, local):
    import torch

    from workloads import configs as C

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    w = C.BY_NAME[args.workload]
    if args.prefill_only:
        # the routed prefill alone (a prefill workload): one JSON line
        r = measure_prefill(w, args.steps, args.warmup, dev, ws, local)
        out = {"metric": "routed prefill tokens/s at 1 GB300", "value": r["value"], "unit": "tokens/s",
               "n_gpus": ws, "steps": args.steps, "warmup": args.warmup, "ms_per_step": r["ms_per_call"],
               "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.shape.dtype,
               "data": "synthetic (seeded counter-based generator)", "config": {"workload": w.name}}
        out.update({k: v for k, v in r.items() if k not in ("value", "unit")})
        if rank == 0:
            print(json.dumps(out), flush=True)
        if ws > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    head = measure(w, args.steps, args.warmup, dev, ws, local, use_graph=not args.no_graph)
    out = {"metric": METRIC, "value": head["value"], "unit": "tokens/s", "n_gpus": ws, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": head["ms_per_step"], "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": head["dtype"],
           "data": "synthetic (seeded counter-based generator)"}
    out.update({k: v for k, v in head.items() if k not in ("value", "unit", "ms_per_step", "steps", "warmup",
                                                           "dtype")})
    if args.workload == DEFAULT_WORKLOAD and not args.headline_only:
        # the other bf16 workloads, each over its own step count, on the same box
        out["per_config"] = {}
        for name in PER_CONFIG:
            wc = C.BY_NAME[name]
            r = measure(wc, wc.steps, args.warmup, dev, ws, local, use_graph=not args.no_graph, e2e=False)
            out["per_config"][name] = r
        # routed prefill (the paper's other speed column)
        out["prefill"] = measure_prefill(C.BY_NAME[PREFILL_WORKLOAD], 5, 3, dev, ws, local)
    if rank == 0 and not args.no_cpu:
        o = oracle_sample(w, n_layers_sample=None, steps=1, device=dev)
        out["cpu_baseline"] = {"value": round(o["tokens"] / o["seconds"], 5), "unit": "tokens/s",
                               "cores": o["cores"], "kind": "oracle",
                               "sample": f"1 decode step of sequence 0 of {w.name} (numpy float64; "
                                         f"weight generation and host copy excluded)"}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_reference(args, ws, rank, local):
    if rank != 0:
        return
    import torch
    from workloads import configs as C
    w = C.BY_NAME[args.workload]
    dev = torch.device("cuda", local) if torch.cuda.is_available() else "cpu"
    # bounded per-step sample: layer 0, router, 1 selected middle layer, last
    # layer; warm-up steps untimed, then the timed steps (their measured time)
    oracle_sample(w, n_layers_sample=1, steps=args.warmup, device=dev)
    o = oracle_sample(w, n_layers_sample=1, steps=args.steps, device=dev)
    value = o["tokens"] / o["seconds"]
    out = {"metric": METRIC, "value": round(value, 5), "unit": "tokens/s", "n_gpus": 1, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": round(o["seconds"] / args.steps * 1e3, 2),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "impl": "reference",
           "config": {"workload": w.name, "model": w.shape.name, "batch": w.batch},
           "cpu_baseline": {"value": round(value, 5), "unit": "tokens/s", "cores": o["cores"], "kind": "oracle",
                            "sample": "per step: sequence 0 through layer 0, the router, the first selected "
                                      "middle layer and the last layer (numpy float64); a step counts as the "
                                      "fraction of a token's executed blocks it ran "
                                      f"({o['tokens'] / args.steps:.3f} tokens per step)"},
           "e2e": {"value": round(value, 5), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=64)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--headline-only", action="store_true", help="skip the per_config workloads")
    ap.add_argument("--prefill-only", action="store_true",
                    help="time the routed prefill of --workload (a prefill workload) alone")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-cpu", action="store_true", help="skip the cpu_baseline oracle sample")
    args = ap.parse_args()
    ws, rank, local = _dist()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args, ws, rank, local)
    else:
        run_ours(args, ws, rank, local)


if __name__ == "__main__":
    main()
