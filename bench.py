"""Benchmark of the AVTP pruning stage on GB300.

One step = one avtp_prune call (validate -> score -> allocate -> select ->
compact) over the Qwen3-VL-8B-shaped multi-image request: 16 images of
256..1024 visual tokens, 256 text tokens, hidden 4096, M-RoPE position ids
(3 planes), keep ratio 0.33, criterion = hidden-state variation (paper §3.3.1).
Inputs are synthetic and resident in HBM before the timed region; L2 is flushed
(256 MiB write) before every timed step, outside the step's own events.

Prints one JSON line. ``--impl reference`` times the fp64 CPU oracle on the
host instead (the reference arm of this build: the paper ships no code).

Multi-GPU (torchrun): every rank runs an independent replica of the workload
(the stage shards by request with no exchange); ``value`` sums all ranks'
visual tokens over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "pruning-stage latency (µs) and visual tokens/s on 1 GB300; % of HBM roofline"
UNIT = "visual tokens/s"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
STEP_NAMES = ("validate", "score", "allocate_select", "compact")
SCORE_KERNELS = {"hidden_variation": ["k_score_hvar"],
                 "text_attention": ["k_attn_lse", "k_attn_mass", "k_attn_pack", "k_attn_finalize"]}


# ---------------------------------------------------------------- helpers
def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, "fallback"


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def reduce_max(value: float, world: int, device=None) -> float:
    """Max over ranks (timing only; not on the data path)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_step: int, steps: int, total_ms: float, world: int, device=None):
    """Every rank's units over the slowest rank's time: (units/s, ms per step of the slowest rank).

    Each rank runs its own replica of the workload (weak scaling), so the job's units
    are world x units_per_step x steps."""
    total_ms_max = reduce_max(total_ms, world, device)
    return units_per_step * steps * world / (total_ms_max * 1e-3), total_ms_max / steps


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


class ClockSampler:
    """Samples SM clock and throttle reasons with nvidia-smi while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, period_ms: int = 50):
        self.gpu_index = gpu_index
        self.period_ms = period_ms
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-i",
                 str(self.gpu_index), "-lms", str(self.period_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(self.period_ms / 1000.0 * 2)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for _, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for name, flag in zip(names, parts[4:8]):
                if flag.lower() in ("active", "1", "0x1"):
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if the kernel's sources are unchanged since."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        entry = json.load(f).get(f"{kernel}@{workload}")
    if not entry:
        return None
    csrc = os.path.join(ROOT, "paper_2608_26806_gb300", "csrc")
    h = hashlib.sha256()
    for fn in entry["source_files"]:
        with open(os.path.join(csrc, fn), "rb") as f:
            h.update(f.read())
    if h.hexdigest()[:16] != entry["source_sha"]:
        return None
    return float(entry["dram_bytes_per_launch"])


class L2Flush:
    """Makes L2 cold before a timed step: writes a 256 MiB buffer (twice the L2),
    then reads another 256 MiB buffer so that the lines left in L2 are clean and
    unrelated to the step's inputs (otherwise the step would pay for writing the
    flush data back). Runs outside the step's timed events."""

    def __init__(self, dev):
        import torch

        self.w = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)
        self.r = torch.ones(64 * 1024 * 1024, dtype=torch.float32, device=dev)
        self.sink = torch.empty((), dtype=torch.float32, device=dev)

    def __call__(self):
        import torch

        self.w.zero_()
        torch.amax(self.r, dim=0, out=self.sink)


# ---------------------------------------------------------------- workload accounting
def stage_roofline(acct, ms_step, hbm_gbs, bf16_tflops, peak_kind):
    """The slower of the stage's compulsory bytes at HBM bandwidth and its FLOPs at the
    bf16 tensor peak, as a fraction of the measured step time."""
    t_hbm = acct["stage_bytes"] / (hbm_gbs * 1e9)
    t_tensor = acct["flops"] / (bf16_tflops * 1e12)
    out = {"bound": "hbm" if t_hbm >= t_tensor else "tensor", "algorithmic_bytes": acct["stage_bytes"],
           "algorithmic_flops": acct["flops"], "bound_us": round(max(t_hbm, t_tensor) * 1e6, 2),
           "achieved_gbs": round(acct["stage_bytes"] / (ms_step * 1e-3) / 1e9, 1), "peak_gbs": hbm_gbs,
           "peak_tflops": bf16_tflops, "frac": round(max(t_hbm, t_tensor) / (ms_step * 1e-3), 4),
           "peak_kind": peak_kind}
    return out


def stage_accounting(wl, criterion, n_kept, lse=False, query_set="text"):
    lay = wl.layout
    n_vis = int(lay.n_visual_per_request().sum())
    n_txt = lay.n_tokens - n_vis
    D = wl.hidden
    pos_bytes = wl.pos_planes * 4
    gather = n_kept * D * 2 * 2 + n_kept * pos_bytes * 2  # read + write of every kept row
    if criterion == "hidden_variation":
        score_bytes = 2 * n_vis * D * 2
        # compulsory: both visual rows once, text rows once (kept), kept rows written, positions
        stage_bytes = score_bytes + n_txt * D * 2 + n_kept * D * 2 + n_kept * pos_bytes * 2
        flops = 0
    elif query_set == "last":
        # the request's last token as the only query (CUDA-core path): every key once, the
        # last token's query rows; FMAs, not tensor-core work, so the stage is HBM-bound
        Hq, Hkv, d = wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        R = lay.n_requests
        score_bytes = lay.n_tokens * Hkv * d * 2 + R * Hq * d * 2
        stage_bytes = score_bytes + n_txt * D * 2 + n_kept * D * 2 + n_kept * pos_bytes * 2
        fma_flops = 0
        for r in range(R):
            T_r = int(lay.cu_seqlens[r + 1]) - int(lay.cu_seqlens[r])
            fma_flops += 2 * Hq * d * T_r + 2 * Hq * d * int(lay.n_visual_per_request()[r])
        return {"n_vis": n_vis, "n_txt": n_txt, "score_bytes": int(score_bytes), "stage_bytes": int(stage_bytes),
                "gather_bytes": int(gather), "flops": 0, "fma_flops": int(fma_flops)}
    else:
        Hq, Hkv, d = wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        if lse:  # supplied LSE: visual keys, text queries and the text rows' LSE only
            score_bytes = n_vis * Hkv * d * 2 + n_txt * Hq * d * 2 + n_txt * Hq * 4
        else:
            score_bytes = lay.n_tokens * Hkv * d * 2 + n_txt * Hq * d * 2
        stage_bytes = score_bytes + n_txt * D * 2 + n_kept * D * 2 + n_kept * pos_bytes * 2
        flops = 0
        vis = lay.visual_mask()
        for r in range(lay.n_requests):
            a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
            v = vis[a:b]
            text_pos = np.nonzero(~v)[0]
            vis_prefix = np.concatenate([[0], np.cumsum(v)])
            for p in text_pos:
                if not lse:
                    flops += 2 * Hq * d * (p + 1)          # pass 1: every visible key
                flops += 2 * Hq * d * int(vis_prefix[p + 1])  # pass 2: visible visual keys
    return {"n_vis": n_vis, "n_txt": n_txt, "score_bytes": int(score_bytes), "stage_bytes": int(stage_bytes),
            "gather_bytes": int(gather), "flops": int(flops)}


# ---------------------------------------------------------------- our arm
def run_ours(args, world, rank, local):
    import torch

    from paper_2608_26806_gb300 import avtp, synth

    import __graft_entry__

    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    __graft_entry__.build()
    crit = args.criterion
    second = None if args.no_secondary or crit != "hidden_variation" else "text_attention"
    parts = ("A", "pos") if (crit == "hidden_variation" and second is None) else ("A", "B", "V", "pos")
    wl = synth.make_workload(args.config, parts=parts)
    lay = wl.layout

    def bf16(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)

    L = avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)
    h_cur, h_prior = bf16(wl.h_cur), bf16(wl.h_prior)
    pos = torch.from_numpy(wl.pos).to(dev)
    kr = torch.from_numpy(wl.keep_ratio).to(dev)
    score_tensors = dict(h_cur=h_cur, h_prior=h_prior)
    if crit == "text_attention":
        score_tensors = dict(q=bf16(wl.q), k=bf16(wl.k), softmax_scale=wl.softmax_scale)
    call = avtp.PruneCall(L, crit, keep_ratio=kr, keep_ratio_host=wl.keep_ratio, rows={"hidden": h_cur},
                          planes={"pos": pos}, **score_tensors)
    n_kept = call.buffers.n_kept
    acct = stage_accounting(wl, crit, n_kept)
    stream = torch.cuda.current_stream()
    flush = L2Flush(dev)
    K, W = args.steps, args.warmup
    n_ev = avtp.N_STEP_EVENTS
    outer = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    inner = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ev)] for _ in range(K)]
    for evs in inner:  # create the driver events before they are handed to the library
        for e in evs:
            e.record(stream)
    for _ in range(W):
        flush()
        call.run(stream)
    torch.cuda.synchronize()
    st = avtp.read_device_status(call.buffers.workspace)
    if st != avtp.OK:
        raise RuntimeError(f"device status after warm-up: {avtp.status_string(st)}")

    # timed region 1 (the headline): whole avtp_prune calls, kernels chained by
    # programmatic dependent launch, L2 flushed before each step outside its events
    sampler = ClockSampler(torch.cuda.current_device()) if not args.no_clocks else None
    barrier(world)
    torch.cuda.synchronize()
    if sampler:
        sampler.start()
        time.sleep(0.3)
    for i in range(K):
        flush()
        outer[i][0].record(stream)
        call.run(stream)
        outer[i][1].record(stream)
    torch.cuda.synchronize()
    # timed region 2: the same steps with an event after every kernel, for per-kernel durations
    for i in range(K):
        flush()
        call.run(stream, step_events=inner[i])
    torch.cuda.synchronize()
    # the other scoring criterion (text-to-visual attention), timed the same way on the
    # same workload, for a secondary object of the line
    sec = sec_lse = sec_last = prog = fwd = None
    if second is not None:
        sec = time_secondary(args, wl, L, kr, h_cur, pos, bf16, stream, flush, torch, avtp, world, dev)
        lse = fa_lse(wl, bf16(wl.q), bf16(wl.k), torch)
        torch.cuda.synchronize()
        sec_lse = time_secondary(args, wl, L, kr, h_cur, pos, bf16, stream, flush, torch, avtp, world, dev, lse=lse)
        del lse
        sec_last = time_secondary(args, wl, L, kr, h_cur, pos, bf16, stream, flush, torch, avtp, world, dev,
                                  query_set="last")
        prog = time_progressive(args, wl, L, h_cur, h_prior, pos, stream, flush, torch, avtp, world, dev)
        fwd = time_forward(args, wl, L, bf16, stream, flush, torch, avtp, world, dev)
    variants = time_variants(args, call, stream, flush, torch, avtp, 4 if crit == "hidden_variation" else 7)
    clocks = sampler.stop() if sampler else None
    barrier(world)
    step_ms = [a.elapsed_time(b) for a, b in outer]
    per_step = {name: [inner[i][j].elapsed_time(inner[i][j + 1]) for i in range(K)]
                for j, name in enumerate(STEP_NAMES)}
    serial_ms = [inner[i][0].elapsed_time(inner[i][n_ev - 1]) for i in range(K)]
    total_ms = sum(step_ms)
    value, ms_step = whole_job_rate(acct["n_vis"], K, total_ms, world, dev)

    # end to end through the public API: pinned host inputs -> device -> prune -> host outputs,
    # with the process (and so the pinned buffers it touches first) on the GPU's NUMA node
    numa, prev_cpus = bind_to_gpu_numa_node(dev.index if dev.index is not None else 0)
    e2e = run_e2e(args, wl, crit, L, call, dev, stream, torch, avtp)
    e2e_pipe = run_e2e_pipelined(args, wl, crit, L, call, dev, torch, avtp)
    e2e["numa"] = numa
    os.sched_setaffinity(0, prev_cpus)

    if rank != 0:
        return None
    hbm, bf16_tf, peak_kind = measured_peaks()
    score_ms = statistics.mean(per_step["score"])
    dominant = SCORE_KERNELS[crit][0]
    if crit == "hidden_variation":
        achieved = acct["score_bytes"] / (score_ms * 1e-3) / 1e9
        roof = {"bound": "hbm", "kernel": dominant, "achieved": round(achieved, 1), "peak": hbm, "unit": "GB/s",
                "frac": round(achieved / hbm, 4), "peak_kind": peak_kind,
                "algorithmic_bytes_per_launch": acct["score_bytes"],
                "avg_launch_us": round(score_ms * 1e3, 2),
                "traffic": recorded_traffic(dominant, args.config)}
    else:
        achieved = acct["flops"] / (score_ms * 1e-3) / 1e12
        roof = {"bound": "tensor", "kernel": "score (lse + mass + finalize)", "achieved": round(achieved, 2),
                "peak": bf16_tf, "unit": "TFLOP/s", "frac": round(achieved / bf16_tf, 4), "peak_kind": peak_kind,
                "algorithmic_flops_per_launch": acct["flops"], "avg_launch_us": round(score_ms * 1e3, 2),
                "traffic": None}
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world, "steps": K, "warmup": W,
        "ms_per_step": round(ms_step, 5), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": args.config, "criterion": crit, "global_batch": lay.n_requests,
                   "seq_len": lay.n_tokens, "visual_tokens": acct["n_vis"], "kept_tokens": n_kept,
                   "hidden": wl.hidden, "images": lay.n_images, "keep_ratio": float(wl.keep_ratio[0]),
                   "parallelism": f"replicas{world}", "l2": "flushed before every timed step: 256 MiB write, then 256 MiB read (clean), outside the step's events"},
        "latency_us": _latency(step_ms),
        "warm_l2": variants["warm_l2"],
        "graph": variants["graph"],
        "steps_us": {k: round(statistics.mean(v) * 1e3, 2) for k, v in per_step.items()},
        "serialized_step_us": round(statistics.mean(serial_ms) * 1e3, 2),
        "stage_roofline": stage_roofline(acct, ms_step, hbm, bf16_tf, peak_kind),
        "roofline": roof,
        "e2e": e2e,
        "e2e_pipelined": e2e_pipe,
        "gpu_launches": K * (4 if crit == "hidden_variation" else 7) + variants["launches"],
        "clocks": clocks,
    }
    hbm_s, bf16_s, _ = measured_peaks()
    for key, res, label in (("text_attention", sec, "score (pack + lse + mass + finalize)"),
                            ("text_attention_lse", sec_lse, "score with a supplied LSE (pack + mass + finalize)")):
        if res is None:
            continue
        ms2 = res["ms_per_step"]
        score_us = res["steps_us"]["score"]
        line[key] = {
            "criterion": "text_attention", "lse": "supplied" if key.endswith("lse") else "computed",
            "value": round(res["acct"]["n_vis"] / (ms2 * 1e-3), 1), "unit": UNIT,
            "ms_per_step": round(ms2, 5), "steps": res["steps"], "latency_us": res["latency_us"],
            "steps_us": res["steps_us"],
            "stage_roofline": stage_roofline(res["acct"], ms2, hbm_s, bf16_s, peak_kind),
            "score_roofline": {"bound": "tensor", "kernel": label,
                               "achieved": round(res["acct"]["flops"] / (score_us * 1e-6) / 1e12, 2),
                               "peak": bf16_s, "unit": "TFLOP/s",
                               "frac": round(res["acct"]["flops"] / (score_us * 1e-6) / 1e12 / bf16_s, 4),
                               "algorithmic_flops_per_launch": res["acct"]["flops"]},
            "gpu_launches": res["launches"]}
        line["gpu_launches"] += res["launches"]
    if sec_last is not None:
        ms3 = sec_last["ms_per_step"]
        score_us = sec_last["steps_us"]["score"]
        a3 = sec_last["acct"]
        line["text_attention_last"] = {
            "criterion": "text_attention", "query_set": "last (the request's last token, §4.1)",
            "path": "CUDA cores", "value": round(a3["n_vis"] / (ms3 * 1e-3), 1), "unit": UNIT,
            "ms_per_step": round(ms3, 5), "steps": sec_last["steps"], "latency_us": sec_last["latency_us"],
            "steps_us": sec_last["steps_us"],
            "stage_roofline": stage_roofline(a3, ms3, hbm_s, bf16_s, peak_kind),
            "score_roofline": {"bound": "hbm", "kernel": "score (logits + mass)",
                               "achieved": round(a3["score_bytes"] / (score_us * 1e-6) / 1e9, 1), "peak": hbm_s,
                               "unit": "GB/s",
                               "frac": round(a3["score_bytes"] / (score_us * 1e-6) / 1e9 / hbm_s, 4),
                               "algorithmic_bytes_per_launch": a3["score_bytes"],
                               "fma_flops_per_launch": a3["fma_flops"]},
            "gpu_launches": sec_last["launches"]}
        line["gpu_launches"] += sec_last["launches"]
    if prog is not None:
        line["progressive"] = prog
        line["gpu_launches"] += prog["gpu_launches"]
    if fwd is not None:
        res, Kf = fwd
        flops = forward_flops(wl)
        plain, with_b = res["plain"]["ms"], res["with_scores"]["ms"]
        achieved = flops / (plain * 1e-3) / 1e12
        line["attn_forward"] = {
            "what": "the pruning layer's causal attention forward (O fp32, natural-log LSE) through "
                    "avtp_attn_forward, plain and with criterion B's scores from the forward's LSE",
            "steps": Kf, "l2": "flushed before every timed call",
            "plain_us": round(plain * 1e3, 2), "plain_p50_us": res["plain"]["p50_us"],
            "with_scores_us": round(with_b * 1e3, 2), "with_scores_p50_us": res["with_scores"]["p50_us"],
            "criterion_b_marginal_us": round((with_b - plain) * 1e3, 2),
            "criterion_b_marginal_frac": round((with_b - plain) / plain, 4),
            "roofline": {"bound": "tensor", "kernel": "forward (query tiles + value transpose + k_attn_fwd)",
                         "achieved": round(achieved, 2), "peak": bf16_s, "unit": "TFLOP/s",
                         "frac": round(achieved / bf16_s, 4), "peak_kind": peak_kind,
                         "algorithmic_flops_per_launch": flops},
            "gpu_launches": res["plain"]["launches"] + res["with_scores"]["launches"]}
        line["gpu_launches"] += line["attn_forward"]["gpu_launches"]
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, crit, args.cpu_seconds)
        if not args.no_all_core_baseline:
            n_img = int(wl.layout.img_cu[1])
            line["cpu_baseline"]["all_cores"] = cpu_baseline_all_cores(args.config, crit, n_img,
                                                                       min(10.0, args.cpu_seconds))
    return line


def _latency(ms):
    srt = sorted(ms)
    return {"p50": round(srt[len(srt) // 2] * 1e3, 2), "p90": round(srt[int(len(srt) * 0.9)] * 1e3, 2),
            "mean": round(statistics.mean(ms) * 1e3, 2)}


def time_variants(args, call, stream, flush, torch, avtp, per_step):
    """The headline step two more ways: with L2 left warm between steps (stream
    launches, back to back), and replayed from a CUDA graph (L2 flushed, then warm)."""
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]

    def loop(launch, flushed):
        for i in range(K):
            if flushed:
                flush()
            ev[i][0].record(stream)
            launch()
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        return _latency([a.elapsed_time(b) for a, b in ev])

    for _ in range(3):
        call.run(stream)
    torch.cuda.synchronize()
    out = {"warm_l2": {"latency_us": loop(lambda: call.run(stream), False), "steps": K, "launch": "stream"},
           "launches": K * per_step}
    try:
        side = torch.cuda.Stream()
        side.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=side):
            call.run(side)
        torch.cuda.synchronize()
        for _ in range(3):
            flush()
            graph.replay()
        torch.cuda.synchronize()
        cold = loop(graph.replay, True)
        warm = loop(graph.replay, False)
        st = avtp.read_device_status(call.buffers.workspace)
        if st != avtp.OK:
            raise RuntimeError(f"device status after graph replays: {avtp.status_string(st)}")
        out["graph"] = {"latency_us": cold, "warm_l2_latency_us": warm, "steps": K,
                        "l2": "flushed before every replay (cold), then back to back (warm)"}
        out["launches"] += 2 * K * per_step
    except Exception as e:  # a capture the runtime refuses: report it, keep the stream numbers
        out["graph"] = {"unavailable": f"{type(e).__name__}: {str(e)[:200]}"}
    return out


def fa_lse(wl, q, k, torch):
    """Natural-log LSE of every (head, text query) over its causally visible keys, [Hq, T] fp32.

    This stands in for the normaliser a FlashAttention forward of the pruning layer
    keeps; it is an input of the stage in that mode, computed here once with plain
    torch before any timing."""
    lay = wl.layout
    Hq, Hkv = wl.n_q_heads, wl.n_kv_heads
    G = Hq // Hkv
    out = torch.zeros(Hq, lay.n_tokens, dtype=torch.float32, device=q.device)
    vis = lay.visual_mask()
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        tp = torch.from_numpy(np.nonzero(~vis[a:b])[0]).to(q.device)
        if tp.numel() == 0:
            continue
        keys = torch.arange(b - a, device=q.device)
        mask = keys[None, :] > tp[:, None]
        for h in range(Hq):
            z = (q[a + tp, h].float() @ k[a:b, h // G].float().T) * wl.softmax_scale
            out[h, a + tp] = torch.logsumexp(z.masked_fill(mask, float("-inf")), dim=1)
    return out


def time_secondary(args, wl, L, kr, h_cur, pos, bf16, stream, flush, torch, avtp, world, dev, lse=None,
                   query_set="text"):
    """The attention criterion on the same workload: whole-call latency and per-step times."""
    crit = "text_attention"
    extra = {} if lse is None else {"lse": lse}
    call = avtp.PruneCall(L, crit, keep_ratio=kr, keep_ratio_host=wl.keep_ratio, rows={"hidden": h_cur},
                          planes={"pos": pos}, q=bf16(wl.q), k=bf16(wl.k), softmax_scale=wl.softmax_scale,
                          query_set=query_set, **extra)
    acct = stage_accounting(wl, crit, call.buffers.n_kept, lse=lse is not None, query_set=query_set)
    K = max(10, min(args.steps, 300))
    n_ev = avtp.N_STEP_EVENTS
    outer = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    inner = [[torch.cuda.Event(enable_timing=True) for _ in range(n_ev)] for _ in range(K)]
    for evs in inner:
        for e in evs:
            e.record(stream)
    for _ in range(max(3, args.warmup)):
        flush()
        call.run(stream)
    torch.cuda.synchronize()
    st = avtp.read_device_status(call.buffers.workspace)
    if st != avtp.OK:
        raise RuntimeError(f"device status after warm-up (attention criterion): {avtp.status_string(st)}")
    barrier(world)
    torch.cuda.synchronize()
    for i in range(K):
        flush()
        outer[i][0].record(stream)
        call.run(stream)
        outer[i][1].record(stream)
    torch.cuda.synchronize()
    for i in range(K):
        flush()
        call.run(stream, step_events=inner[i])
    torch.cuda.synchronize()
    step_ms = sorted(a.elapsed_time(b) for a, b in outer)
    ms = reduce_max(sum(step_ms), world, dev) / K
    per_step = {name: statistics.mean(inner[i][j].elapsed_time(inner[i][j + 1]) for i in range(K))
                for j, name in enumerate(STEP_NAMES)}
    return {"acct": acct, "steps": K, "ms_per_step": ms,
            "latency_us": {"p50": round(step_ms[len(step_ms) // 2] * 1e3, 2),
                           "p90": round(step_ms[int(len(step_ms) * 0.9)] * 1e3, 2)},
            "steps_us": {k: round(v * 1e3, 2) for k, v in per_step.items()},
            # k_prep, k_attn_pack, k_attn_lse (computed LSE only), k_attn_mass, k_attn_finalize,
            # k_alloc_select, k_compact; the last-token set: k_prep, k_narrow_logits,
            # k_narrow_mass, k_alloc_select, k_compact
            "launches": K * ((7 if lse is None else 6) if query_set == "text" else 5)}


def forward_flops(wl):
    """Causal attention forward FLOPs: every visible (query, key) pair of every query head
    costs d multiply-adds in Q K^T and d in P V."""
    cu = wl.layout.cu_seqlens
    pairs = sum(int(n) * (int(n) + 1) // 2 for n in np.diff(cu))
    return 4 * pairs * wl.n_q_heads * wl.head_dim


def time_forward(args, wl, L, bf16, stream, flush, torch, avtp, world, dev):
    """The layer's attention forward (avtp_attn_forward) on the same workload, plain and
    with criterion B's scores from its own LSE: B's marginal cost is the difference."""
    q, k, v = bf16(wl.q), bf16(wl.k), bf16(wl.v)
    K = max(5, min(args.steps, 100))
    out = {}
    for key, with_scores in (("plain", False), ("with_scores", True)):
        call = avtp.ForwardCall(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale, scores=with_scores)
        for _ in range(max(3, args.warmup)):
            flush()
            call.run(stream)
        torch.cuda.synchronize()
        st = avtp.read_device_status(call.workspace)
        if st != avtp.OK:
            raise RuntimeError(f"device status after warm-up (attention forward): {avtp.status_string(st)}")
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
        barrier(world)
        torch.cuda.synchronize()
        for i in range(K):
            flush()
            ev[i][0].record(stream)
            call.run(stream)
            ev[i][1].record(stream)
        torch.cuda.synchronize()
        ms = sorted(a.elapsed_time(b) for a, b in ev)
        out[key] = {"ms": reduce_max(sum(ms), world, dev) / K, "p50_us": round(ms[len(ms) // 2] * 1e3, 2),
                    "launches": K * (7 if with_scores else 4)}  # k_prep, qtiles, transpose, forward (+ pack, mass, finalize)
        del call
    return out, K


def time_progressive(args, wl, L, h_cur, h_prior, pos, stream, flush, torch, avtp, world, dev, stages=3):
    """Progressive pruning (paper §3.3.2): the stage three times on a shrinking batch.

    Each step prunes with criterion A at a per-stage keep ratio of 0.5^(1/3) (half of the
    visual tokens survive the three stages). After each stage the next layout is built
    on the device (avtp_pruned_layout) and the compacted h_cur becomes the next h_prior;
    the next layer's hidden states are fixed synthetic inputs of the shrunk size."""
    ratio = np.full(wl.layout.n_requests, np.float32(0.5 ** (1.0 / 3.0)), dtype=np.float32)
    kr = torch.from_numpy(ratio).to(dev)
    calls, layouts, bytes_total = [], [], 0
    cur_L, cur_cur, cur_prior, cur_pos = L, h_cur, h_prior, pos
    gen = torch.Generator(device=dev)
    gen.manual_seed(7)
    for s_i in range(stages):
        call = avtp.PruneCall(cur_L, "hidden_variation", keep_ratio=kr, keep_ratio_host=ratio, h_cur=cur_cur,
                              h_prior=cur_prior, rows={"hidden": cur_cur}, planes={"pos": cur_pos})
        n_vis = int(cur_L.n_vis_per_request.astype(np.int64).sum())
        n_txt = cur_L.n_tokens - n_vis
        D = cur_cur.shape[1]
        bytes_total += 2 * n_vis * D * 2 + n_txt * D * 2 + call.buffers.n_kept * (D * 2 + cur_pos.shape[0] * 4 * 2)
        calls.append(call)
        call.run(stream)
        if s_i + 1 < stages:
            ws = avtp.new_workspace(avtp.workspace_size(cur_L), dev)
            nxt = avtp.pruned_layout(cur_L, ratio, call.buffers.budgets, call.buffers.out_cu_seqlens, workspace=ws,
                                     stream=stream)
            layouts.append((cur_L, call, nxt, ws))
            cur_prior = call.buffers.outputs["hidden"]
            cur_cur = (cur_prior.float() + 0.5 * torch.randn(cur_prior.shape, generator=gen, device=dev)).to(torch.bfloat16)
            cur_pos = call.buffers.outputs["pos"]
            cur_L = nxt
    torch.cuda.synchronize()

    def step():
        for s_i, call in enumerate(calls):
            call.run(stream)
            if s_i + 1 < stages:
                prev_L, prev_call, nxt, ws = layouts[s_i]
                avtp.pruned_layout(prev_L, ratio, prev_call.buffers.budgets, prev_call.buffers.out_cu_seqlens,
                                   workspace=ws, stream=stream, into=nxt)

    K = max(10, min(args.steps, 300))
    for _ in range(max(3, args.warmup)):
        flush()
        step()
    torch.cuda.synchronize()
    for c in calls:
        st = avtp.read_device_status(c.buffers.workspace)
        if st != avtp.OK:
            raise RuntimeError(f"device status after warm-up (progressive): {avtp.status_string(st)}")
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    barrier(world)
    torch.cuda.synchronize()
    for i in range(K):
        flush()
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    ms = sorted(a.elapsed_time(b) for a, b in ev)
    p50 = ms[len(ms) // 2]
    hbm, _, peak_kind = measured_peaks()
    bound_us = bytes_total / (hbm * 1e9) * 1e6
    return {"stages": stages, "keep_ratio_per_stage": round(float(ratio[0]), 6), "criterion": "hidden_variation",
            "visual_tokens": [int(c.layout.n_vis_per_request.astype(np.int64).sum()) for c in calls],
            "tokens": [int(c.layout.n_tokens) for c in calls], "steps": K,
            "latency_us": {"p50": round(p50 * 1e3, 2), "p90": round(ms[int(len(ms) * 0.9)] * 1e3, 2)},
            "stage_roofline": {"bound": "hbm", "algorithmic_bytes": int(bytes_total), "bound_us": round(bound_us, 2),
                               "frac": round(bound_us / (p50 * 1e3), 4), "peak_gbs": hbm, "peak_kind": peak_kind},
            "gpu_launches": K * (4 * stages + (stages - 1))}  # each boundary: one k_prep (it builds the spans)


def run_e2e(args, wl, crit, L, call, dev, stream, torch, avtp):
    """Same metric through the public API with host buffers: H2D inputs, prune, D2H outputs, all timed."""
    b = call.buffers
    host_in = {"h_cur": torch.from_numpy(np.ascontiguousarray(wl.h_cur).view(np.int16)).pin_memory(),
               "pos": torch.from_numpy(wl.pos).pin_memory()}
    if crit == "hidden_variation":
        host_in["h_prior"] = torch.from_numpy(np.ascontiguousarray(wl.h_prior).view(np.int16)).pin_memory()
    else:
        host_in["q"] = torch.from_numpy(np.ascontiguousarray(wl.q).view(np.int16)).pin_memory()
        host_in["k"] = torch.from_numpy(np.ascontiguousarray(wl.k).view(np.int16)).pin_memory()
    for name in ("cu_seqlens", "img_cu", "img_start", "img_len"):
        host_in["lay_" + name] = torch.from_numpy(L.host[name].copy()).pin_memory()
    host_in["keep_ratio"] = torch.from_numpy(wl.keep_ratio.copy()).pin_memory()
    # device destinations: the very tensors the prepared call reads
    dev_dst = {"h_cur": call._keep_alive[1]["hidden"], "pos": call._keep_alive[2]["pos"],
               "lay_cu_seqlens": L.cu_seqlens, "lay_img_cu": L.img_cu, "lay_img_start": L.img_start,
               "lay_img_len": L.img_len, "keep_ratio": call._keep_alive[0]}
    st = call._keep_alive[3]
    if crit == "hidden_variation":
        dev_dst["h_prior"] = st["h_prior"]
    else:
        dev_dst["q"], dev_dst["k"] = st["q"], st["k"]
    outs = [b.kept_idx[:b.n_kept], b.budgets, b.out_cu_seqlens] + list(b.outputs.values())
    host_out = [torch.empty(o.shape, dtype=o.dtype).pin_memory() for o in outs]
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(o.numel() * o.element_size() for o in outs)
    steps = max(3, min(50, args.e2e_steps))
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def one():
        for k, h in host_in.items():
            dst = dev_dst[k]
            dst.view(torch.int16 if dst.dtype == torch.bfloat16 else dst.dtype).copy_(
                h.view(torch.int16) if dst.dtype == torch.bfloat16 else h, non_blocking=True)
        call.run(stream)
        for o, h in zip(outs, host_out):
            h.copy_(o, non_blocking=True)

    for _ in range(3):
        one()
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(steps):
        one()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / steps
    n_vis = int(wl.layout.n_visual_per_request().sum())
    return {"value": round(n_vis / (ms * 1e-3), 1), "unit": UNIT, "ms_per_step": round(ms, 4),
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": steps}


def run_e2e_pipelined(args, wl, crit, L, call, dev, torch, avtp):
    """The same end-to-end metric with consecutive steps overlapped, as a serving loop
    would run them: step i + 1's inputs are copied in while step i computes and copies
    its outputs out. Each step still copies all its inputs in and all its outputs out.
    Two prepared calls with their own device inputs and outputs alternate, and three
    streams (copy in, compute, copy out) are ordered by events."""
    from paper_2608_26806_gb300 import avtp as A

    calls = [call]
    # a second call on its own copies of every device input
    L2 = A.Layout.from_host(L.host["cu_seqlens"], L.host["img_cu"], L.host["img_start"], L.host["img_len"],
                            device=dev)
    st0 = call._keep_alive[3]
    kr2 = call._keep_alive[0].clone()
    h_cur2 = call._keep_alive[1]["hidden"].clone()
    pos2 = call._keep_alive[2]["pos"].clone()
    if crit == "hidden_variation":
        st2 = dict(h_cur=h_cur2, h_prior=st0["h_prior"].clone())
    else:
        st2 = dict(q=st0["q"].clone(), k=st0["k"].clone(), softmax_scale=st0["softmax_scale"])
    calls.append(A.PruneCall(L2, crit, keep_ratio=kr2, keep_ratio_host=wl.keep_ratio, rows={"hidden": h_cur2},
                             planes={"pos": pos2}, **st2))
    layouts = [L, L2]

    host_in = {"h_cur": torch.from_numpy(np.ascontiguousarray(wl.h_cur).view(np.int16)).pin_memory(),
               "pos": torch.from_numpy(wl.pos).pin_memory()}
    if crit == "hidden_variation":
        host_in["h_prior"] = torch.from_numpy(np.ascontiguousarray(wl.h_prior).view(np.int16)).pin_memory()
    else:
        host_in["q"] = torch.from_numpy(np.ascontiguousarray(wl.q).view(np.int16)).pin_memory()
        host_in["k"] = torch.from_numpy(np.ascontiguousarray(wl.k).view(np.int16)).pin_memory()
    for name in ("cu_seqlens", "img_cu", "img_start", "img_len"):
        host_in["lay_" + name] = torch.from_numpy(L.host[name].copy()).pin_memory()
    host_in["keep_ratio"] = torch.from_numpy(wl.keep_ratio.copy()).pin_memory()

    def dests(c, lay):
        d = {"h_cur": c._keep_alive[1]["hidden"], "pos": c._keep_alive[2]["pos"], "lay_cu_seqlens": lay.cu_seqlens,
             "lay_img_cu": lay.img_cu, "lay_img_start": lay.img_start, "lay_img_len": lay.img_len,
             "keep_ratio": c._keep_alive[0]}
        sc = c._keep_alive[3]
        if crit == "hidden_variation":
            d["h_prior"] = sc["h_prior"]
        else:
            d["q"], d["k"] = sc["q"], sc["k"]
        return d

    dst = [dests(c, lay) for c, lay in zip(calls, layouts)]
    outs = []
    for c in calls:
        b = c.buffers
        outs.append([b.kept_idx[:b.n_kept], b.budgets, b.out_cu_seqlens] + list(b.outputs.values()))
    host_out = [[torch.empty(o.shape, dtype=o.dtype).pin_memory() for o in outs[j]] for j in range(2)]
    s_in, s_comp, s_out = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    in_done = [torch.cuda.Event() for _ in range(2)]
    comp_done = [torch.cuda.Event() for _ in range(2)]
    out_done = [torch.cuda.Event() for _ in range(2)]
    for j in range(2):  # every buffer starts free
        comp_done[j].record(s_comp)
        out_done[j].record(s_out)

    def step(i):
        j = i & 1
        s_in.wait_event(comp_done[j])  # step i - 2 has read these inputs
        with torch.cuda.stream(s_in):
            for k, h in host_in.items():
                d = dst[j][k]
                d.view(torch.int16 if d.dtype == torch.bfloat16 else d.dtype).copy_(
                    h.view(torch.int16) if d.dtype == torch.bfloat16 else h, non_blocking=True)
        in_done[j].record(s_in)
        s_comp.wait_event(in_done[j])
        s_comp.wait_event(out_done[j])  # step i - 2's outputs have been copied out
        calls[j].run(s_comp)
        comp_done[j].record(s_comp)
        s_out.wait_event(comp_done[j])
        with torch.cuda.stream(s_out):
            for o, h in zip(outs[j], host_out[j]):
                h.copy_(o, non_blocking=True)
        out_done[j].record(s_out)

    steps = max(4, min(50, args.e2e_steps))
    for i in range(4):
        step(i)
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(s_in)
    s_comp.wait_stream(s_in)
    s_out.wait_stream(s_in)
    for i in range(steps):
        step(i)
    s_out.wait_stream(s_comp)
    s_out.wait_stream(s_in)
    ev1.record(s_out)
    torch.cuda.synchronize()
    for c in calls:
        st = A.read_device_status(c.buffers.workspace)
        if st != A.OK:
            raise RuntimeError(f"device status after the pipelined steps: {A.status_string(st)}")
    # the last step's outputs equal those of the serial path
    for o, h in zip(outs[(steps - 1) & 1], host_out[(steps - 1) & 1]):
        if not torch.equal(o.cpu(), h):
            raise RuntimeError("pipelined end-to-end outputs differ from the device outputs")
    ms = ev0.elapsed_time(ev1) / steps
    n_vis = int(wl.layout.n_visual_per_request().sum())
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(o.numel() * o.element_size() for o in outs[0])
    return {"value": round(n_vis / (ms * 1e-3), 1), "unit": UNIT, "ms_per_step": round(ms, 4),
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": steps,
            "launch": "two prepared calls alternating; copy-in, compute and copy-out streams overlap consecutive steps"}


# ---------------------------------------------------------------- CPU oracle (baseline / reference arm)
def _sub_workload(wl, n_images):
    """The first n_images images of request 0 with their surrounding text: a bounded sample."""
    from paper_2608_26806_gb300 import synth

    lay = wl.layout
    i_end = min(n_images, int(lay.img_cu[1]))
    if i_end < int(lay.img_cu[1]):
        end_tok = int(lay.img_start[i_end])  # stop before the next image
    else:
        end_tok = int(lay.cu_seqlens[1])
    sub = synth.Layout(cu_seqlens=np.array([0, end_tok], dtype=np.int32), img_cu=np.array([0, i_end], dtype=np.int32),
                       img_start=lay.img_start[:i_end].copy(), img_len=lay.img_len[:i_end].copy())
    t = {k: v[:end_tok] for k, v in wl.tensors.items() if k in ("h_cur", "h_prior", "q", "k")}
    if "pos" in wl.tensors:
        t["pos"] = wl.tensors["pos"][:, :end_tok]
    return sub, t


def _oracle_step(O, sub, t, wl, crit):
    kw = dict(keep_ratio=wl.keep_ratio[:1], rows={"hidden": t["h_cur"]}, planes={"pos": t["pos"]})
    if crit == "hidden_variation":
        return O.prune(sub, h_cur=t["h_cur"], h_prior=t["h_prior"], **kw)
    return O.prune(sub, criterion="text_attention", q=t["q"], k=t["k"], n_q_heads=wl.n_q_heads,
                   n_kv_heads=wl.n_kv_heads, scale=wl.softmax_scale, **kw)


def _oracle_threads():
    try:
        import threadpoolctl

        info = threadpoolctl.threadpool_info()
        return max([int(i.get("num_threads", 1)) for i in info] or [1])
    except Exception:  # noqa: BLE001
        return 1


def cpu_baseline(wl, crit, seconds):
    from oracle import avtp_oracle as O

    lay = wl.layout
    n_img = int(lay.img_cu[1])
    sub, t = _sub_workload(wl, n_img)
    t0 = time.perf_counter()
    done_tokens = 0
    runs = 0
    while True:
        _oracle_step(O, sub, t, wl, crit)
        runs += 1
        done_tokens += int(sub.img_len.sum())
        if time.perf_counter() - t0 > seconds:
            break
    el = time.perf_counter() - t0
    cores = 1 if crit == "hidden_variation" else _oracle_threads()
    return {"value": round(done_tokens / el, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{runs} full pass(es) of the oracle pipeline over request 0 ({n_img} images, "
                      f"{int(sub.img_len.sum())} visual tokens), criterion {crit}, {el:.1f} s"}


def _oracle_worker(config, crit, n_img, seconds, start_at):
    """One process of the all-core oracle baseline: the same bounded sample, run from a
    common start time for `seconds`; returns (visual tokens done, seconds)."""
    from oracle import avtp_oracle as O
    from paper_2608_26806_gb300 import synth

    parts = ("A", "pos") if crit == "hidden_variation" else ("A", "B", "pos")
    wl = synth.make_workload(config, parts=parts)
    sub, t = _sub_workload(wl, n_img)
    while time.time() < start_at:
        time.sleep(0.005)
    t0 = time.perf_counter()
    runs = 0
    while True:
        _oracle_step(O, sub, t, wl, crit)
        runs += 1
        if time.perf_counter() - t0 > seconds:
            break
    return runs * int(sub.img_len.sum()), time.perf_counter() - t0


def cpu_baseline_all_cores(config, crit, n_img, seconds):
    """The oracle on every host core: one process per core (spawned, one BLAS thread each),
    all running the same bounded sample over a common window."""
    import multiprocessing as mp

    cores = len(os.sched_getaffinity(0))
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(cores) as pool:
            start_at = time.time() + 25.0  # every worker has built its sample by then
            res = pool.starmap(_oracle_worker, [(config, crit, n_img, seconds, start_at)] * cores)
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    tokens = sum(r[0] for r in res)
    window = max(r[1] for r in res)
    return {"value": round(tokens / window, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{cores} processes, each the oracle pipeline over the same request-0 sample "
                      f"({n_img} images) for {seconds:.0f} s from a common start, criterion {crit}"}


def bind_to_gpu_numa_node(dev_index):
    """Pin this process to the CPUs of the GPU's NUMA node (when the platform reports one),
    so that pinned host buffers allocated afterwards sit on that node (first touch).
    Returns (what was done, the previous CPU set to restore)."""
    prev = os.sched_getaffinity(0)
    info = {"gpu_numa_node": None, "bound": False, "process_cpus": len(prev)}
    try:
        import subprocess

        bus = subprocess.run(["nvidia-smi", "--query-gpu=pci.bus_id", "--format=csv,noheader", "-i",
                              str(dev_index)], capture_output=True, text=True, timeout=20).stdout.strip()
        dom, rest = bus.split(":", 1)
        path = f"/sys/bus/pci/devices/{dom[-4:].lower()}:{rest.lower()}/numa_node"
        node = int(open(path).read().strip())
        info["gpu_numa_node"] = node
        if node >= 0:
            cpulist = open(f"/sys/devices/system/node/node{node}/cpulist").read().strip()
            cpus = set()
            for part in cpulist.split(","):
                if part:
                    a, _, b = part.partition("-")
                    cpus.update(range(int(a), int(b or a) + 1))
            cpus &= prev
            if cpus:
                os.sched_setaffinity(0, cpus)
                info.update(bound=True, process_cpus=len(cpus), node_cpulist=cpulist)
    except Exception as e:  # noqa: BLE001 - a platform without the information keeps the default placement
        info["note"] = f"no NUMA binding: {type(e).__name__}"
    return info, prev


def run_reference(args, world, rank):
    if rank != 0:
        return None
    from oracle import avtp_oracle as O
    from paper_2608_26806_gb300 import synth

    crit = args.criterion
    parts = ("A", "pos") if crit == "hidden_variation" else ("A", "B", "pos")
    wl = synth.make_workload(args.config, parts=parts)
    n_img = int(wl.layout.img_cu[1])
    # size each step's sample so that warm-up + timed steps stay within ~2 minutes
    sub, t = _sub_workload(wl, 1)
    t0 = time.perf_counter()
    _oracle_step(O, sub, t, wl, crit)
    per_img = max(time.perf_counter() - t0, 1e-3)
    budget = 120.0 / max(1, args.steps + args.warmup)
    k_img = int(max(1, min(n_img, budget // per_img)))
    sub, t = _sub_workload(wl, k_img)
    for _ in range(args.warmup):
        _oracle_step(O, sub, t, wl, crit)
    times = []
    for _ in range(args.steps):
        s = time.perf_counter()
        _oracle_step(O, sub, t, wl, crit)
        times.append(time.perf_counter() - s)
    toks = int(sub.img_len.sum())
    total = sum(times)
    value = toks * args.steps / total
    cores = 1 if crit == "hidden_variation" else _oracle_threads()
    sample = (f"each step: the oracle's full pipeline on the first {k_img} of {n_img} images of the "
              f"{args.config} request ({toks} visual tokens), criterion {crit}")
    return {"impl": "reference", "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.config, "criterion": crit, "parallelism": "host cores"},
            "cpu_baseline": {"value": round(value, 1), "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


# ---------------------------------------------------------------- phase timeline (diagnostic)
def run_timeline(args):
    """The headline stage in the timeline build (-DAVTP_TIMELINE): per phase, the earliest
    and latest global-timer stamp over the CTAs that reached it, in microseconds after the
    validation kernel starts (median over the steps after a few warm-up calls), with L2
    flushed before each call (the host enqueues the call while the flush runs) and, for
    comparison, back to back. Not a bench line: the stamps add atomics to the kernels."""
    os.environ["AVTP_TIMELINE"] = "1"
    import torch

    from paper_2608_26806_gb300 import avtp, build, synth

    build.build(timeline=True)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = synth.make_workload(args.config, parts=("A", "B", "pos") if args.criterion == "text_attention" else ("A", "pos"))
    lay = wl.layout

    def bf16(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)

    L = avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)
    h_cur = bf16(wl.h_cur)
    kr = torch.from_numpy(wl.keep_ratio).to(dev)
    if args.criterion == "hidden_variation":
        score = dict(h_cur=h_cur, h_prior=bf16(wl.h_prior))
    else:
        score = dict(q=bf16(wl.q), k=bf16(wl.k), softmax_scale=wl.softmax_scale)
    call = avtp.PruneCall(L, args.criterion, keep_ratio=kr, keep_ratio_host=wl.keep_ratio, rows={"hidden": h_cur},
                          planes={"pos": torch.from_numpy(wl.pos).to(dev)}, **score)
    flush = L2Flush(dev)
    out = {"config": args.config, "criterion": args.criterion, "unit": "us after the validation kernel starts"}
    for mode in ("flushed", "back_to_back"):
        runs = []
        for i in range(max(args.steps, 8)):
            torch.cuda.synchronize()
            if mode == "flushed":
                flush()
            else:
                call.run()
            call.run()
            torch.cuda.synchronize()
            tl = avtp.timeline(call.buffers.workspace)
            t0 = tl["prep_begin"][0]
            runs.append({k: ((v[0] - t0) / 1e3, (v[1] - t0) / 1e3) for k, v in tl.items()})
        keep = runs[3:]
        out[mode] = {k: [round(float(np.median([r[k][j] for r in keep])), 2) for j in (0, 1)] for k in keep[-1]}
    return out


# ---------------------------------------------------------------- forward timeline (diagnostic)
def run_timeline_forward(args):
    """The attention forward in the timeline build (-DAVTP_TIMELINE): clock stamps per key
    block of the CTA with the most key blocks (head 0), medians over its steady blocks and
    over calls, in SM cycles: the block period, the softmax's phases and the MMA-issuing
    thread's. Not a bench line: the stamps add stores to the kernel."""
    os.environ["AVTP_TIMELINE"] = "1"
    import torch

    from paper_2608_26806_gb300 import avtp, build, synth

    build.build(timeline=True)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = synth.make_workload(args.config, parts=("B", "V"))
    lay = wl.layout

    def bf16(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)

    L = avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)
    call = avtp.ForwardCall(L, q=bf16(wl.q), k=bf16(wl.k), v=bf16(wl.v), softmax_scale=wl.softmax_scale,
                            scores=False)
    # the first CTA runs the last query tile of the last request: its key blocks
    cu = lay.cu_seqlens
    a, b = int(cu[-2]), int(cu[-1])
    nblk = (b - 1) // 128 - a // 128 + 1
    n = min(nblk, 256)  # the timeline build keeps the first 256 blocks
    flush = L2Flush(dev)
    per_call = []
    for i in range(max(args.steps, 8)):
        flush()
        call.run()
        torch.cuda.synchronize()
        if i >= 3:
            per_call.append(avtp.forward_timeline(n))
    st = avtp.read_device_status(call.workspace)
    if st != avtp.OK:
        raise RuntimeError(f"device status (forward timeline): {avtp.status_string(st)}")
    S = {n: i for i, n in enumerate(avtp.FORWARD_TIMELINE_SLOTS)}

    def med(f):
        vals = []
        for t in per_call:
            vals += [f(t, j) for j in range(2, n - 1)]
        return round(float(np.median(vals)), 1)

    return {"config": args.config, "blocks": nblk, "blocks_stamped": n, "unit": "SM cycles per 128-key block (median)",
            "period": med(lambda t, j: t[j, S["p_handed"]] - t[j - 1, S["p_handed"]]),
            "softmax": {"wait_for_S": med(lambda t, j: t[j, S["s_ready"]] - t[j, S["top"]]),
                        "load_mask_max_exchange": med(lambda t, j: t[j, S["exchanged"]] - t[j, S["s_ready"]]),
                        "exponentials": med(lambda t, j: t[j, S["exp_done"]] - t[j, S["exchanged"]]),
                        "p_handover": med(lambda t, j: t[j, S["p_handed"]] - t[j, S["exp_done"]])},
            "mma_thread": {"S_waits_and_issue": med(lambda t, j: t[j, S["mma_s_issued"]] - t[j, S["mma_s_entry"]]),
                           "PV_waits": med(lambda t, j: t[j, S["mma_pv_ready"]] - t[j, S["mma_pv_entry"]]),
                           "PV_issue": med(lambda t, j: t[j, S["mma_pv_issued"]] - t[j, S["mma_pv_ready"]])}}


# ---------------------------------------------------------------- single-step entry points (diagnostic)
def run_standalone(args):
    """The steps as separate calls (avtp_score, avtp_allocate, avtp_select, avtp_compact) on
    the workload, and the pruning-layer statistic (avtp_layer_attention for every layer of a
    36-layer model, then avtp_layer_select over 256 samples): event-timed calls, L2 flushed
    before each, medians in microseconds. Not a bench line: each call also runs the
    validation kernel, and nothing is chained."""
    import torch

    from paper_2608_26806_gb300 import avtp, synth

    import __graft_entry__

    __graft_entry__.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = synth.make_workload(args.config, parts=("A", "pos"))
    lay = wl.layout

    def bf16(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)

    L = avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)
    h_cur, h_prior = bf16(wl.h_cur), bf16(wl.h_prior)
    pos = torch.from_numpy(wl.pos).to(dev)
    kr = torch.from_numpy(wl.keep_ratio).to(dev)
    n_kept = avtp.kept_count_host({"cu_seqlens": lay.cu_seqlens, "img_cu": lay.img_cu, "img_len": lay.img_len},
                                  wl.keep_ratio)
    ws = avtp.new_workspace(avtp.workspace_size(L, "hidden_variation", h_cur=h_cur, h_prior=h_prior), dev)
    scores = torch.zeros(lay.n_tokens, dtype=torch.float32, device=dev)
    sums = torch.empty(max(lay.n_images, 1), dtype=torch.int64, device=dev)
    budgets = torch.empty(max(lay.n_images, 1), dtype=torch.int32, device=dev)
    ocu = torch.empty(lay.n_requests + 1, dtype=torch.int32, device=dev)
    kept = torch.empty(max(n_kept, 1), dtype=torch.int32, device=dev)
    hid_out = torch.empty(max(n_kept, 1), h_cur.shape[1], dtype=torch.bfloat16, device=dev)
    pos_out = torch.empty(pos.shape[0], max(n_kept, 1), dtype=pos.dtype, device=dev)
    rows = [(h_cur, hid_out)] + [(pos[p_], pos_out[p_]) for p_ in range(pos.shape[0])]
    n_layers, n_samples = 36, 256
    A = torch.zeros(n_samples, n_layers, dtype=torch.int64, device=dev)
    A.copy_(torch.randint(0, 1 << 40, (n_samples, n_layers), generator=torch.Generator().manual_seed(3)).to(dev))
    A1 = torch.zeros(lay.n_requests, n_layers, dtype=torch.int64, device=dev)
    steps = {
        "score": lambda: avtp.score(L, "hidden_variation", h_cur=h_cur, h_prior=h_prior, scores=scores,
                                    img_sums=sums, workspace=ws),
        "allocate": lambda: avtp.allocate(L, sums, kr, budgets=budgets, out_cu_seqlens=ocu, workspace=ws),
        "select": lambda: avtp.select(L, scores, budgets, ocu, n_kept, kept_idx=kept, workspace=ws),
        "compact": lambda: avtp.compact(kept[:n_kept], lay.n_tokens, [(a_, b_[:n_kept]) for a_, b_ in rows],
                                        workspace=ws),
        "layer_attention_36_layers": lambda: [avtp.layer_attention(L, sums, A1, l_, workspace=ws)
                                              for l_ in range(n_layers)],
        "layer_select_256_samples": lambda: avtp.layer_select(A, 3),
    }
    flush = L2Flush(dev)
    K = max(10, min(args.steps, 100))
    out = {"config": args.config, "unit": "us per call (median, L2 flushed before each)", "calls": K}
    for name, fn in steps.items():
        for _ in range(3):
            flush()
            fn()
        torch.cuda.synchronize()
        ms = []
        for _ in range(K):
            flush()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
        out[name] = round(float(np.median(ms)) * 1e3, 2)
    st = avtp.read_device_status(ws)
    if st != avtp.OK:
        raise RuntimeError(f"device status (standalone steps): {avtp.status_string(st)}")
    return out


# ---------------------------------------------------------------- criterion-B pass timelines (diagnostic)
def run_timeline_attn(args):
    """Criterion B's tensor-core passes in the timeline build (-DAVTP_TIMELINE): clock stamps
    per step of each pass's first CTA, medians over its steps after the first and over calls,
    in SM cycles: the step period, the MMA thread's wait for its operands and accumulators,
    its issue, the epilogue's hold of the accumulators, and the time from a key tile's load
    to the MMA thread finding it ready. Not a bench line: the stamps add stores."""
    os.environ["AVTP_TIMELINE"] = "1"
    import torch

    from paper_2608_26806_gb300 import avtp, build, synth

    build.build(timeline=True)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = synth.make_workload(args.config, parts=("B",))
    lay = wl.layout

    def bf16(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)

    L = avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)
    q, k = bf16(wl.q), bf16(wl.k)
    ws = avtp.new_workspace(avtp.workspace_size(L, "text_attention", q=q, k=k, path="tensor"), dev)
    flush = L2Flush(dev)
    S = {n: i for i, n in enumerate(avtp.SCORE_TIMELINE_SLOTS)}
    stamps = {1: [], 2: []}
    for i in range(max(args.steps, 8)):
        flush()
        avtp.score(L, "text_attention", q=q, k=k, softmax_scale=wl.softmax_scale, path="tensor", workspace=ws)
        torch.cuda.synchronize()
        if i >= 3:
            for p in (1, 2):
                stamps[p].append(avtp.score_timeline(p, 64))
    st = avtp.read_device_status(ws)
    if st != avtp.OK:
        raise RuntimeError(f"device status (criterion-B timeline): {avtp.status_string(st)}")
    out = {"config": args.config, "unit": "SM cycles per step (median)"}
    for p in (1, 2):
        def med(f):
            vals = []
            for t in stamps[p]:
                n = int(np.count_nonzero(t[:, S["mma_issued"]]))  # steps the first CTA ran
                vals += [f(t, j) for j in range(1, n)]
            return round(float(np.median(vals)), 1) if vals else None
        out[f"pass{p}"] = {
            "steps_stamped": int(np.count_nonzero(stamps[p][-1][:, S["mma_issued"]])),
            "period": med(lambda t, j: t[j, S["mma_issued"]] - t[j - 1, S["mma_issued"]]),
            "mma_wait_for_operands": med(lambda t, j: t[j, S["mma_ready"]] - t[j, S["mma_step"]]),
            "mma_issue": med(lambda t, j: t[j, S["mma_issued"]] - t[j, S["mma_ready"]]),
            "epilogue_hold": med(lambda t, j: t[j, S["acc_released"]] - t[j, S["acc_ready"]]),
            "load_to_ready": med(lambda t, j: t[j, S["mma_ready"]] - t[j, S["load_issued"]])}
    return out


# ---------------------------------------------------------------- path crossover (diagnostic)
def run_crossover(args):
    """Criterion-B scoring on both paths as the query set widens: one request of four
    640-token images followed by n text tokens, Qwen3-shaped heads (32 query heads, 8 KV
    groups, d = 128), rows per KV group = 4n. Each avtp_score call is event-timed with L2
    flushed before it (the host enqueues the call while the flush runs); the median of 30
    calls per point. Not a bench line."""
    import torch

    from paper_2608_26806_gb300 import avtp, synth

    import __graft_entry__

    __graft_entry__.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    flush = L2Flush(dev)

    def bf16(x):
        return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).to(dev).view(torch.bfloat16)

    out = []
    texts = [args.crossover_text] if args.crossover_text else [1, 2, 4, 8, 16, 32, 64, 128]
    paths = [args.crossover_path] if args.crossover_path else ["tensor", "cuda"]
    for n_text in texts:
        wl = synth.make_custom([[("i", 640)] * 4 + [("t", n_text)]], hidden=128, n_q_heads=32, n_kv_heads=8,
                               head_dim=128, seed=3, parts=("B",))
        lay = wl.layout
        L = avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)
        st = dict(q=bf16(wl.q), k=bf16(wl.k), softmax_scale=wl.softmax_scale)
        row = {"text_tokens": n_text, "rows_per_kv_group": 4 * n_text}
        for path in paths:
            ws = avtp.new_workspace(avtp.workspace_size(L, "text_attention", path=path, **st))
            sc = torch.zeros(lay.n_tokens, device=dev)
            sums = torch.zeros(lay.n_images, dtype=torch.int64, device=dev)
            for _ in range(5):
                avtp.score(L, "text_attention", path=path, scores=sc, img_sums=sums, workspace=ws, **st)
            torch.cuda.synchronize()
            ts = []
            for _ in range(30):
                flush()
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record()
                avtp.score(L, "text_attention", path=path, scores=sc, img_sums=sums, workspace=ws, **st)
                b.record()
                torch.cuda.synchronize()
                ts.append(a.elapsed_time(b) * 1e3)
            row[path + "_us"] = round(float(np.median(ts)), 2)
        out.append(row)
    return {"crossover": out, "unit": "us per avtp_score call (event-timed, L2 flushed)"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="qwen3_vl_8b")
    ap.add_argument("--criterion", default="hidden_variation", choices=["hidden_variation", "text_attention"])
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-all-core-baseline", action="store_true",
                    help="skip the oracle timed on every host core (about 35 s)")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-secondary", action="store_true",
                    help="skip the attention-criterion object (timed after the headline criterion)")
    ap.add_argument("--timeline", action="store_true",
                    help="print the phase timeline of the headline stage (timeline build) instead of the bench line")
    ap.add_argument("--timeline-forward", action="store_true",
                    help="per-block phase timings of the attention forward (timeline build), not a bench line")
    ap.add_argument("--standalone", action="store_true",
                    help="time the single-step entry points and the layer statistic, not the bench line")
    ap.add_argument("--timeline-attn", action="store_true",
                    help="per-step phase timings of criterion B's tensor-core passes (timeline build), not a bench line")
    ap.add_argument("--crossover", action="store_true",
                    help="print criterion-B scoring times of both paths as the query set widens, not the bench line")
    ap.add_argument("--crossover-text", type=int, default=0, help="--crossover: only this many text tokens")
    ap.add_argument("--crossover-path", default="", choices=["", "tensor", "cuda"], help="--crossover: only this path")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.timeline:
        print(json.dumps(run_timeline(args)), flush=True)
        return
    if args.timeline_forward:
        print(json.dumps(run_timeline_forward(args)), flush=True)
        return
    if args.timeline_attn:
        print(json.dumps(run_timeline_attn(args)), flush=True)
        return
    if args.standalone:
        print(json.dumps(run_standalone(args)), flush=True)
        return
    if args.crossover:
        print(json.dumps(run_crossover(args)), flush=True)
        return
    world, rank, local = dist_env()
    if args.impl == "reference":
        line = run_reference(args, world, rank)
    else:
        line = run_ours(args, world, rank, local)
    if line is not None:
        print(json.dumps(line), flush=True)
    if world > 1 and args.impl == "ours":
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
