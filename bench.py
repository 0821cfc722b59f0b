"""Benchmark of Conduit's hot path on GB300: one step = scoring pass, selection,
gather, scatter and refresh attention over one batch of a synthetic workload.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl conduit|reference]
                  [--config batched|single|multi|longdoc|tiny]

The default workload is batched serving (16 requests x 8 192 tokens, paged
cache, refresh and scatter included): the largest single-GPU configuration.

Prints one JSON line. ``value`` is cached visual tokens passed through the
whole step per second (device time, inputs resident in HBM, L2 flushed
between steps); ``metric_parts`` splits it into the metric's two halves
(tokens scored and selected per second, refresh-pass µs) from per-call
times; ``e2e`` is the same through the public step with the cache,
queries and fresh rows copied from pinned host memory each step and the
selection and refresh output copied back, over back-to-back steps of two
pipelines that alternate (one step's copies overlap the previous step's
kernels). Under torchrun every rank runs its
own replica on its own GPU (the path has no collective step); the step time is
the maximum over ranks.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

_CORES = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(_CORES))

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "cached visual tokens scored+selected/sec and refresh-pass µs; % of HBM roofline"
UNIT = "tokens/s"
DESCR = {
    "tiny": "tiny single-image: 1 layer, 1 image x 256 visual tokens, 16 query-prefix tokens, 4/2 heads, head_dim 64, fp32, budget 10%",
    "single": "single high-res image: 28 layers, 28/4 heads, head_dim 128, bf16 cache [28,4,1024,128], 32 query-prefix tokens, budget 10%",
    "multi": "multi-image: 8 images x 1024 tokens, 28 layers, 28/4 heads, head_dim 128, bf16, 64 query-prefix tokens, budget 10%",
    "longdoc": "long document: 32 pages x 1296 tokens, 36 layers, 32/8 heads, head_dim 128, bf16, 48 query-prefix tokens, budget 10%",
    "batched": "batched serving: 16 requests x 4 images x 2048 tokens, 28 layers, 28/4 heads, head_dim 128, bf16 paged (16-token pages), 32-128 query tokens, budgets 5/10/20%",
}
L2_FLUSH_BYTES = 256 << 20


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# fp32 CUDA-core peak: 152 SMs x 128 FMA lanes x 2 FLOP x 2.07 GHz (max SM clock)
ALU_FP32_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi samples every 50 ms while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.proc, self.lines = index, None, []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self._t = threading.Thread(target=self._read, daemon=True)
            self._t.start()
            t_end = time.time() + 5.0  # the timed region starts once sampling runs
            while not self.lines and time.time() < t_end and self.proc.poll() is None:
                time.sleep(0.02)
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc is not None:
            n0, t_end = len(self.lines), time.time() + 1.0  # one sample after the region
            while len(self.lines) == n0 and time.time() < t_end:
                time.sleep(0.02)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------ distributed
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def reduce_max(value: float, world: int) -> float:
    """Maximum of a float over ranks (identity on one rank)."""
    if world == 1:
        return value
    import torch.distributed as dist
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------ work models
def work_model(pipe, idx_sets=None) -> dict:
    """Algorithmic bytes / FLOPs of one step, per C-ABI call. The refresh
    figures depend on the selected positions, which change from step to step
    (each step's exchange rewrites the cache the next step scores): with
    `idx_sets` (the selections of the timed calls) they are the mean over
    those selections, else those of the selection now in `pipe.idx`."""
    kv, b = pipe.kv, pipe.batch
    esz = pipe.kv.k.element_size()
    L = kv.num_layers if pipe.layers is None else len(pipe.layers)
    Lall, Hq, Hkv, d = kv.num_layers, kv.num_q_heads, kv.num_kv_heads, kv.head_dim
    tok, qo = b.tok_off.tolist(), b.q_off.tolist()
    R, K = b.num_requests, b.num_images
    n_tot = tok[-1]
    # K read once, the queries, s and attn_sum written, g; then the value-norm source:
    # V read once, or one stored fp32 per token and scored layer, or nothing
    score_bytes = L * Hkv * n_tot * d * esz + L * Hq * qo[-1] * d * esz + 8 * n_tot + 4 * K
    score_bytes += {"v": L * Hkv * n_tot * d * esz, "side_cache": 4 * L * n_tot, "none": 0}[pipe.value_norm]
    if pipe.extra_lse is not None:  # one fp32 per scoring row
        score_bytes += 4 * L * Hq * qo[-1]
    score_flops = sum(2 * L * Hq * (qo[r + 1] - qo[r]) * (tok[r + 1] - tok[r]) * d for r in range(R))
    k_sel = pipe.n_sel
    sel_bytes = 4 * n_tot + 4 * K + 4 * n_tot + n_tot + 4 * k_sel + 4 * K
    if pipe.selection == "quota":  # coefficients, quotas and offsets through the workspace
        sel_bytes += 2 * 12 * K
    copy_bytes = 2 * 2 * Lall * k_sel * Hkv * d * esz
    if not idx_sets:
        idx_sets = [pipe.idx[:k_sel].cpu().tolist()]
    off = pipe.idx_off.tolist()
    ref_flops, ref_bytes = 0, 0
    for idx in idx_sets:
        for r in range(R):
            ps = idx[off[r]:off[r + 1]]
            ref_flops += sum(4 * Hq * d * (p + 1) for p in ps) * Lall
            if ps:
                ref_bytes += 2 * Lall * Hkv * (max(ps) + 1) * d * esz
    ref_flops /= len(idx_sets)
    ref_bytes /= len(idx_sets)
    ref_bytes += 2 * Lall * k_sel * Hq * d * esz  # the query rows in, the output out
    out = {
        "score": {"bytes": score_bytes, "flops": score_flops},
        "select": {"bytes": sel_bytes, "flops": 0},
        "exchange": {"bytes": 2 * copy_bytes, "flops": 0},
        "refresh": {"bytes": ref_bytes, "flops": ref_flops},
    }
    if pipe.vnorm is not None:  # re-read the rewritten value rows, write their norms
        out["norm_update"] = {"bytes": Lall * k_sel * Hkv * d * esz + 4 * Lall * k_sel, "flops": 0}
    return out


def side_cache_bytes(pipe) -> int:
    """conduit_value_norms: every value row read once, one fp32 per token and layer written."""
    kv = pipe.kv
    n_tot = pipe.batch.n_tot
    return kv.num_layers * n_tot * (kv.num_kv_heads * kv.head_dim * kv.k.element_size() + 4)


def call_kernels(pipe) -> dict:
    """Kernels behind each C-ABI call for this cache, their binding unit and source file.

    bf16 caches with head_dim 128 take the tensor-core kernels; other shapes
    the CUDA-core ones (the library makes the same choice).
    """
    tc = pipe.kv.k.dtype == torch.bfloat16 and pipe.kv.head_dim == 128
    tail = ["finalize_tokens_kernel", "image_means_kernel"]
    if tc:  # hbm or tensor: run_conduit keeps whichever ideal time is longer for the workload
        score = (["score_tc_kernel"] + tail, "hbm", "score_tc.cu")
        refresh = (["refresh_tc_kernel"], "tensor", "refresh_tc.cu")
    else:
        score = (["value_sumsq_kernel", "rowstats_kernel", "colsum_kernel"] + tail, "alu", "score_simt.cu")
        refresh = (["refresh_simt_kernel"], "alu", "refresh_simt.cu")
    norms = (["vnorm_halves_kernel" if tc else "vnorm_rows_kernel"], "hbm", "vnorm.cu")
    if pipe.value_norm != "v" and not tc:  # no separate value pass
        score = (["rowstats_kernel", "colsum_kernel"] + tail, "alu", "score_simt.cu")
    sel = ["quota_kernel", "select_kernel"] if pipe.selection == "quota" else ["select_kernel"]
    # conduit_score_select_topk: the scoring kernels, then one launch for the
    # tail and the selection when every request holds at most 8192 tokens
    tok = pipe.batch.tok_off.tolist()
    max_tok = max(b - a for a, b in zip(tok[:-1], tok[1:]))
    sms = torch.cuda.get_device_properties(pipe.device).multi_processor_count
    fused = (score[0][:-len(tail)] + ["finalize_select_kernel"] if max_tok <= 8192 and tok[-1] <= 32 * sms
             else score[0] + ["select_kernel" if max_tok <= 8192 or max_tok > 65536 else "select_cluster_kernel"])
    return {"score": score, "select": (sel, "hbm", "select.cu"),
            "score_select": (fused, score[1], score[2]),
            "exchange": (["kv_copy_kernel"], "hbm", "kvcopy.cu"), "refresh": refresh,
            "norm_update": norms, "side_cache": norms}


def _src_hash(src: str) -> str:
    with open(os.path.join(ROOT, "paper_2609_05821_gb300", "csrc", src), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()[:12]


def _traffic(call: str, workload: str, src: str):
    """DRAM bytes per launch from a committed ncu summary, if the kernel source is unchanged.

    profiles/traffic.txt lines: <call> <workload> <bytes per launch> <sha256[:12] of the source>;
    the workload is the config name, with @<ratio> when the run overrides the ratio.
    """
    p = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(p):
        return None
    for line in open(p):
        f = line.split()
        if len(f) >= 4 and not line.startswith("#") and f[0] == call and f[1] == workload:
            return float(f[2]) if f[3] == _src_hash(src) else None
    return None


# -------------------------------------------------------------- our arm
def run_config(args, n_tok: int, budget_total: int, layers: int) -> dict:
    """The workload and run settings of a bench line; both arms print this dict."""
    return {"workload": DESCR[args.config], "name": args.config, "tokens_per_step": n_tok,
            "budget_total": budget_total, "layers": layers,
            "ratio_override": args.ratio,
            "l2": f"flushed between timed steps ({L2_FLUSH_BYTES >> 20} MB write)",
            "cuda_graph": not args.no_graph, "parallelism": f"replicas x{int(os.environ.get('WORLD_SIZE', '1'))}",
            "statistic": args.statistic,
            "value_norms": {"v": "read from V inside the scoring pass",
                            "side_cache": "side cache: built once per cache outside the step, "
                                          "updated for the rewritten rows inside it",
                            "none": "not used (attention alone)"}[args.value_norm],
            "softmax": ("full context (seeded outside-key log-sum-exps)" if args.full_context
                        else "visual keys"),
            "selection": {"global": "one global top-k (Eq. 11)",
                          "quota": "per-image quotas (App. D.3)"}[args.selection]}


def build_pipeline(cfg: str, device, ratio=None, statistic="mean", value_norm="v",
                   full_context=False, selection="global", num_requests=None):
    from paper_2609_05821_gb300 import pipeline, synth
    w = synth.workload(cfg) if num_requests is None else synth.workload(cfg, num_requests=num_requests)
    inputs = synth.make_inputs(w, device=device)
    _with_ratio(inputs, ratio)  # one refresh ratio for every request (e.g. the long-document budgets)
    extra = synth.make_extra_lse(inputs) if full_context else None
    return pipeline.from_inputs(inputs, statistic=statistic, value_norm=value_norm,
                                extra_lse=extra, selection=selection), w


def time_steps(fn, steps: int, flush=None):
    """Per-step device time (ms) with CUDA events on the current stream."""
    stream = torch.cuda.current_stream()
    times = []
    for _ in range(steps):
        if flush is not None:
            flush()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        b.synchronize()
        times.append(a.elapsed_time(b))
    return times


def run_conduit(args):
    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_05821_gb300 import conduit as C

    pipe, w = build_pipeline(args.config, dev, args.ratio, args.statistic, args.value_norm,
                             args.full_context, args.selection)
    n_tok = pipe.batch.n_tot
    flush_buf = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flush = lambda: flush_buf.zero_()

    # warm-up (eager), then one graph of the whole step
    for _ in range(args.warmup):
        pipe.step()
    torch.cuda.synchronize()
    launches0 = C.conduit_launch_count()
    pipe.step()
    torch.cuda.synchronize()
    launches_per_step = C.conduit_launch_count() - launches0
    if not args.no_graph:
        pipe.capture()
        for _ in range(max(1, args.warmup)):
            pipe.step()
    torch.cuda.synchronize()

    # timed region: K whole steps
    hbm, tc, tc_sus, peak_src = _peaks()
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0 = time.perf_counter()
        step_ms = time_steps(pipe.step, args.steps, flush)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    barrier(world)
    mean_ms = sum(step_ms) / len(step_ms)
    max_ms = reduce_max(mean_ms, world)

    # per-call breakdown over K eager steps (events on the launching stream)
    graph, pipe.graph = pipe.graph, None
    from paper_2609_05821_gb300 import conduit as CC
    seq = [("score", pipe.score), ("select", pipe.select), ("exchange", pipe.exchange)]
    if pipe.vnorm is not None:
        seq.append(("norm_update", pipe.norm_update))
    seq.append(("refresh", pipe.refresh_attn))
    calls = {name: [] for name, _ in seq}
    stream = torch.cuda.current_stream()
    idx_sets = []  # each timed refresh call's selection, read back after its events
    for _ in range(args.steps):
        flush()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(seq) + 1)]
        ev[0].record(stream)
        for i, (_, fn) in enumerate(seq):
            fn()
            ev[i + 1].record(stream)
        ev[-1].synchronize()
        for i, (name, _) in enumerate(seq):
            calls[name].append(ev[i].elapsed_time(ev[i + 1]))
        idx_sets.append(pipe.idx[:pipe.n_sel].cpu().tolist())
    # the step runs scoring and selection as one call (conduit_score_select_topk)
    # under the global rule: timed the same way, on its own
    fused_ms = None
    if pipe.selection == "global":
        ts = []
        for _ in range(args.steps):
            flush()
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            ev[0].record(stream)
            pipe.score_select()
            ev[1].record(stream)
            ev[1].synchronize()
            ts.append(ev[0].elapsed_time(ev[1]))
        fused_ms = sum(ts) / len(ts)
    side_cache = None
    if pipe.vnorm is not None:  # built once per cache (outside the step): timed on its own
        scratch = torch.empty_like(pipe.vnorm)
        ts = []
        for _ in range(max(3, args.steps)):
            flush()
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            ev[0].record(stream)
            CC.conduit_value_norms(pipe.kv, pipe.batch, scratch)
            ev[1].record(stream)
            ev[1].synchronize()
            ts.append(ev[0].elapsed_time(ev[1]))
        sc_ms = sum(ts) / len(ts)
        sc_bytes = side_cache_bytes(pipe)
        side_cache = {"us": round(sc_ms * 1e3, 2), "bytes": sc_bytes,
                      "GB_per_s": round(sc_bytes / (sc_ms / 1e3) / 1e9, 1),
                      "hbm_frac": round(sc_bytes / (sc_ms / 1e3) / 1e9 / hbm, 4),
                      "kernels": call_kernels(pipe)["side_cache"][0]}
    pipe.graph = graph
    call_ms = {k: sum(v) / len(v) for k, v in calls.items()}
    status = C.conduit_read_status(pipe.status)

    # roofline of the dominant call
    model = work_model(pipe, idx_sets)
    dom = max(call_ms, key=call_ms.get)
    kernels, bound, src = call_kernels(pipe)[dom]
    if bound in ("hbm", "tensor"):
        # the unit whose ideal time is longer binds: bytes / HBM peak vs FLOPs / tensor peak
        bound = "tensor" if model[dom]["flops"] / (tc * 1e12) > model[dom]["bytes"] / (hbm * 1e9) else "hbm"
    sec = call_ms[dom] / 1e3
    if bound == "hbm":
        achieved, peak, unit = model[dom]["bytes"] / sec / 1e9, hbm, "GB/s"
        peak_note = f"HBM copy, {peak_src}"
    elif bound == "tensor":
        achieved, peak, unit = model[dom]["flops"] / sec / 1e12, tc, "TFLOP/s"
        peak_note = f"bf16 dense burst, {peak_src}"
    else:
        achieved, peak, unit = model[dom]["flops"] / sec / 1e12, ALU_FP32_TFLOPS, "TFLOP/s"
        peak_note = "fp32 FMA: 152 SMs x 128 lanes x 2 FLOP x 2.07 GHz"
    # committed ncu traffic covers the default scoring pass only
    # the workload key carries a ratio override (long document at r = 0.05 / 0.10 / 0.20)
    wkey = args.config + (f"@{args.ratio:g}" if args.ratio is not None else "")
    traffic = _traffic(dom, wkey, src) if pipe.plain and pipe.selection == "global" else None
    roofline = {"bound": bound, "achieved": round(achieved, 3), "peak": round(peak, 1), "unit": unit,
                "frac": round(achieved / peak, 4), "traffic": traffic, "kernel": dom,
                "kernels": kernels, "peak_source": peak_note,
                "hbm_frac": round(model[dom]["bytes"] / sec / 1e9 / hbm, 4)}
    breakdown = {}
    for name, ms in call_ms.items():
        s_ = ms / 1e3
        by, fl = model[name]["bytes"], model[name]["flops"]
        kern_bound = call_kernels(pipe)[name][1]
        if kern_bound in ("hbm", "tensor"):  # the longer ideal time binds
            kern_bound = "tensor" if fl / (tc * 1e12) > by / (hbm * 1e9) else "hbm"
        frac = (fl / s_ / 1e12 / (tc if kern_bound == "tensor" else ALU_FP32_TFLOPS)
                if kern_bound in ("tensor", "alu") else by / s_ / 1e9 / hbm)
        breakdown[name] = {"us": round(ms * 1e3, 2),
                           "GB_per_s": round(by / s_ / 1e9, 1),
                           "hbm_frac": round(by / s_ / 1e9 / hbm, 4),
                           "bound": kern_bound, "frac_of_bound": round(frac, 4)}
        if fl:
            breakdown[name]["TFLOP_per_s"] = round(fl / s_ / 1e12, 2)
        if name in ("score", "select", "exchange"):
            # the scoring, selection and scatter kernels are to sustain 70 % of
            # the peak of their binding unit
            breakdown[name]["target_0_7"] = "pass" if frac >= 0.7 else "fail"

    # end to end through the public step with host buffers: two pipelines of
    # the batch stepped alternately (one step's copies overlap the previous
    # step's kernels), K steps back to back between two events on the
    # launching stream; every step's copies are ordered after the first event
    from paper_2609_05821_gb300 import pipeline
    twin, _ = build_pipeline(args.config, dev, args.ratio, args.statistic, args.value_norm,
                             args.full_context, args.selection)
    if not args.no_graph:
        twin.capture()
    stepper = pipeline.DoubleBuffered(pipe, twin)
    host = pipe.host_buffers()
    for _ in range(4):
        stepper.step_from_host(host)
    torch.cuda.synchronize()
    n_e2e = max(4, min(args.steps, 10))
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    stepper.start_after(a)
    for _ in range(n_e2e):
        stepper.step_from_host(host)
    b.record(stream)
    b.synchronize()
    e2e_mean = reduce_max(a.elapsed_time(b) / n_e2e, world)
    del stepper, twin

    score_select_ms = fused_ms if fused_ms else call_ms["score"] + call_ms["select"]
    out = {
        "metric": METRIC, "value": round(world * n_tok / (max_ms / 1e3), 1), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(max_ms, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if pipe.kv.k.dtype == torch.bfloat16 else "f32",
        "data": "synthetic (seeded; shapes and value laws of the paper's workloads)",
        "config": run_config(args, n_tok, pipe.n_sel, pipe.kv.num_layers),
        "score_select_tokens_per_s": round(n_tok / (score_select_ms / 1e3), 1),
        **({"score_select_call": {"us": round(fused_ms * 1e3, 2),
                                  "kernels": call_kernels(pipe)["score_select"][0]}} if fused_ms else {}),
        "refresh_pass_us": round((call_ms["exchange"] + call_ms.get("norm_update", 0.0)
                                  + call_ms["refresh"]) * 1e3, 2),
        "breakdown": breakdown,
        # the metric's two halves from the eager per-call times: tokens scored and
        # selected per second, and the refresh pass (K/V exchange, the norm update
        # when the side cache is kept, refresh attention)
        "metric_parts": {
            "scored_selected_tokens_per_s": round(world * n_tok / (score_select_ms / 1e3), 1),
            "refresh_pass_us": round(1e3 * sum(call_ms[k] for k in ("exchange", "norm_update", "refresh")
                                               if k in call_ms), 2),
        },
        **({"side_cache_build": side_cache} if side_cache else {}),
        "roofline": roofline,
        "e2e": {"value": round(world * n_tok / (e2e_mean / 1e3), 1), "unit": UNIT,
                "h2d_bytes_per_step": pipe.h2d_bytes(), "d2h_bytes_per_step": pipe.d2h_bytes(),
                "steps": n_e2e, "pipelines": 2},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk.summary(),
        "status": status,
        "wall_s_timed": round(wall, 3),
    }
    default = pipe.plain and pipe.selection == "global"
    if rank == 0 and world == 1 and not args.no_cpu_baseline and default:  # the oracle arm times the default pass
        out["cpu_baseline"] = cpu_baseline(args.config, args.cpu_seconds, args.ratio)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(out), flush=True)


# ------------------------------------------------------- CPU oracle arm
def oracle_step_sample(cfg: str, budget_seconds: float, seed_inputs=None):
    """Time the CPU oracle on a bounded sample of one step of the workload.

    Scoring runs layer by layer over all of request 0's tokens until about
    60 % of the budget is spent; selection runs once on the sample's scores;
    refresh attention runs for a few selected rows of the sampled layers.
    Returns (estimated seconds per full step, description).
    """
    from oracle import conduit_oracle as O
    from paper_2609_05821_gb300 import synth
    w = synth.workload(cfg)
    inputs = seed_inputs or synth.make_inputs(w, device="cpu")
    tok, qo = inputs["tok_off"].tolist(), inputs["q_off"].tolist()
    R, L = len(tok) - 1, w.num_layers
    t0, t1, q0, q1 = tok[0], tok[1], qo[0], qo[1]
    spans = [x - t0 for x in inputs["img_off"].tolist()[: inputs["req_img_off"].tolist()[1] + 1]]
    ql = lambda l: inputs["q"][l, :, q0:q1].double().numpy()
    kl = lambda l: inputs["k"][l, :, t0:t1].double().numpy()
    vl = lambda l: inputs["v"][l, :, t0:t1].double().numpy()
    a, vn, layer_t = [], [], []
    start = time.perf_counter()
    for l in range(L):
        ts = time.perf_counter()
        a.append(O.head_query_mean_attention(ql(l), kl(l)))
        vn.append(O.value_norms(vl(l)))
        layer_t.append(time.perf_counter() - ts)
        if time.perf_counter() - start > 0.6 * budget_seconds:
            break
    ts = time.perf_counter()
    a_, vn_ = np.stack(a), np.stack(vn)
    s = O.throughput_score(a_, vn_)
    g = O.image_mean_attention(a_, spans)
    c = O.image_coefficients(g, 1.0)
    kk = O.budget(inputs["ratios"][0], t1 - t0)
    idx = O.topk_select(O.composite_score(s, c, spans), kk)
    t_sel = time.perf_counter() - ts
    rows = idx[: max(1, min(len(idx), 8))]
    fr = synth.make_fresh_rows(w, len(rows), device="cpu")
    ts = time.perf_counter()
    n_ref_layers = min(len(layer_t), 2)
    for l in range(n_ref_layers):
        kp = O.kv_scatter(kl(l)[None], rows, fr["k_rows"][l:l + 1].double().numpy())
        vp = O.kv_scatter(vl(l)[None], rows, fr["v_rows"][l:l + 1].double().numpy())
        O.refresh_attention(fr["q_rows"][l:l + 1].double().numpy(), kp, vp, rows)
    t_ref = time.perf_counter() - ts
    n_sel_total = sum(O.budget(r, tok[i + 1] - tok[i]) for i, r in enumerate(inputs["ratios"]))
    per_layer = sum(layer_t) / len(layer_t)
    est = (per_layer * L * R + t_sel * R +
           t_ref / (n_ref_layers * len(rows)) * L * n_sel_total)
    desc = (f"request 0: scoring of {len(layer_t)}/{L} layers over all {t1 - t0} tokens, one "
            f"selection, refresh of {len(rows)} rows x {n_ref_layers} layers; extrapolated to "
            f"{R} request(s) x {L} layers x {n_sel_total} refreshed rows")
    return est, desc, time.perf_counter() - start


def _with_ratio(inputs: dict, ratio) -> dict:
    if ratio is not None:
        inputs["ratios"] = [float(ratio)] * (len(inputs["tok_off"]) - 1)
    return inputs


def cpu_baseline(cfg: str, seconds: float, ratio=None) -> dict:
    """The oracle, as it stands, on the host cores: repeated bounded samples for ~`seconds`."""
    from paper_2609_05821_gb300 import synth
    n_tok = _workload_tokens(cfg)
    inputs = _with_ratio(synth.make_inputs(synth.workload(cfg), device="cpu"), ratio)
    ests, spent, desc = [], 0.0, ""
    while spent < seconds:
        est, desc, dt = oracle_step_sample(cfg, seconds, inputs)
        ests.append(est)
        spent += dt
    est = statistics.median(ests)
    return {"value": round(n_tok / est, 2), "unit": UNIT, "cores": _CORES, "kind": "oracle",
            "sample": f"{len(ests)} repetition(s) of: {desc}", "sample_seconds": round(spent, 1),
            "cpu": _cpu_model(),
            "threads_note": f"numpy BLAS threads = {_CORES}; elementwise numpy is single-threaded"}


def _cpu_model() -> str:
    """The host CPU's model name (lscpu), else the machine type."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    import platform
    return platform.machine()


def _workload_tokens(cfg: str) -> int:
    from paper_2609_05821_gb300 import synth
    w = synth.workload(cfg)
    return w.num_requests * w.tokens_per_request


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from paper_2609_05821_gb300 import synth
    w = synth.workload(args.config)
    inputs = _with_ratio(synth.make_inputs(w, device="cpu"), args.ratio)
    n_tok = _workload_tokens(args.config)
    per_step = args.reference_step_seconds or max(2.0, min(20.0, 150.0 / max(1, args.steps + args.warmup)))
    for _ in range(args.warmup):
        oracle_step_sample(args.config, per_step, inputs)
    ests, spent, desc = [], [], ""
    for _ in range(args.steps):
        est, desc, dt = oracle_step_sample(args.config, per_step, inputs)
        ests.append(est)
        spent.append(dt)
    est = statistics.median(ests)
    sample_s = statistics.median(spent)
    # one oracle on the node's host cores does the whole job: N batches take N
    # times as long, so its throughput does not grow with the GPU count
    value = round(n_tok / est, 2)
    from oracle import conduit_oracle as O
    tok = inputs["tok_off"].tolist()
    budget_total = sum(O.budget(r, tok[i + 1] - tok[i]) for i, r in enumerate(inputs["ratios"]))
    out = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        # each timed step is one bounded sample of the workload (measured);
        # value is the whole step's token count over its extrapolated time
        "ms_per_step": round(sample_s * 1e3, 3),
        "step_kind": "bounded sample of the workload's step (measured); value extrapolated to the whole step",
        "extrapolated": True, "extrapolated_full_step_ms": round(est * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded; shapes and value laws of the paper's workloads)",
        "config": run_config(args, n_tok, budget_total, w.num_layers),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": _CORES, "kind": "oracle",
                         "sample": desc, "cpu": _cpu_model(),
                         "sample_seconds_per_step": round(sample_s, 3)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out), flush=True)


# ------------------------------------------- staleness diagnostic (App. D)
def run_staleness(args):
    """The cross-image diagnostic of App. D.3 on a synthetic workload: the
    isotropic Monte Carlo staleness E_iso(T) of the refresh sets of Conduit's
    global rule, the explicit per-image quotas, the global rule without image
    reweighting (lambda = 0) and a uniform random set of the same budgets,
    all under the same draws (M = 5); printed as E / E_uniform with the
    device time of one estimator call and its tensor roofline."""
    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_05821_gb300 import conduit as C
    from paper_2609_05821_gb300 import pipeline, synth
    w = synth.workload(args.config)
    inputs = synth.make_inputs(w, device=dev)
    _with_ratio(inputs, args.ratio)
    M, kappa = 5, 0.5
    L, Hkv, n_tot, d = inputs["k"].shape
    gen = torch.Generator().manual_seed(w.seed + 101)
    z = torch.randn((M, L, Hkv, n_tot, d), generator=gen).to(inputs["k"].dtype).to(dev)
    masks = {}
    for name, kw in (("conduit", {}), ("explicit_quota", {"selection": "quota"}),
                     ("global_no_reweight", {"lam": 0.0})):
        pipe = pipeline.from_inputs(inputs, **kw)
        pipe.score_select()
        masks[name] = pipe.mask.clone()
    tok = inputs["tok_off"].tolist()
    rng = torch.Generator().manual_seed(w.seed + 202)
    uni = torch.zeros(n_tot, dtype=torch.uint8)
    for r in range(len(tok) - 1):
        n_r = tok[r + 1] - tok[r]
        k_r = int(masks["conduit"][tok[r]:tok[r + 1]].sum().item())
        uni[tok[r] + torch.randperm(n_r, generator=rng)[:k_r]] = 1
    masks["uniform"] = uni.to(dev)
    ws = torch.empty(C.conduit_staleness_iso_workspace_size(pipe.kv, pipe.batch, M), dtype=torch.uint8,
                     device=dev)
    err = torch.empty(pipe.batch.num_requests, dtype=torch.float64, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    call = lambda m: C.conduit_staleness_iso(pipe.kv, pipe.batch, pipe.q, m, z, kappa, err=err,
                                             workspace=ws, status=status)
    results = {}
    for name, m in masks.items():
        call(m)
        results[name] = err.sum().item()
    flush_buf = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for _ in range(args.warmup):
        call(masks["conduit"])
    torch.cuda.synchronize()
    launches0 = C.conduit_launch_count()
    ms = time_steps(lambda: call(masks["conduit"]), args.steps, lambda: flush_buf.zero_())
    launches = (C.conduit_launch_count() - launches0) // max(args.steps, 1)
    mean_ms = sum(ms) / len(ms)
    qo = inputs["q_off"].tolist()
    flops = M * sum(4 * w.num_q_heads * d * (tok[r + 1] - tok[r]) * (qo[r + 1] - qo[r]) * L
                    for r in range(len(tok) - 1))
    hbm, tc, _, peak_src = _peaks()
    achieved = flops / (mean_ms / 1e3) / 1e12
    out = {
        "metric": "isotropic staleness evaluations/s (App. D, M = 5 draws)",
        "value": round(1e3 / mean_ms, 3), "unit": "evaluations/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(mean_ms, 4), "higher_is_better": True,
        "dtype": "bf16" if inputs["k"].dtype == torch.bfloat16 else "f32",
        "data": "synthetic (seeded; shapes and value laws of the paper's workloads; seeded draws)",
        "config": {"workload": DESCR[args.config], "name": args.config, "M": M, "kappa": kappa,
                   "l2": f"flushed between timed calls ({L2_FLUSH_BYTES >> 20} MB write)"},
        "E_over_E_uniform": {k: round(v / results["uniform"], 4) for k, v in results.items()},
        "E": {k: v for k, v in results.items()},
        "roofline": {"bound": "tensor", "achieved": round(achieved, 3), "peak": round(tc, 1),
                     "unit": "TFLOP/s", "frac": round(achieved / tc, 4), "traffic": None,
                     "kernel": "staleness (refresh attention over the draws)",
                     "peak_source": f"bf16 dense burst, {peak_src}"},
        "gpu_launches": launches * args.steps,
        "status": C.conduit_read_status(status),
    }
    print(json.dumps(out), flush=True)


def run_profile(args):
    """Eager steps with no timing, e2e or CPU leg: the program ncu captures.

    ``--requests N`` keeps the first N requests of a batched workload, so a
    capture of many passes holds a few GB on the device at most.
    """
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    from paper_2609_05821_gb300 import conduit as C
    pipe, _ = build_pipeline(args.config, dev, args.ratio, args.statistic, args.value_norm,
                             args.full_context, args.selection, args.requests)
    n0 = C.conduit_launch_count()
    for _ in range(args.warmup + args.steps):
        pipe.step()
    torch.cuda.synchronize()
    print(json.dumps({"profile": args.config, "requests": pipe.batch.num_requests,
                      "tokens": pipe.batch.n_tot, "steps": args.warmup + args.steps,
                      "launches": C.conduit_launch_count() - n0,
                      "status": C.conduit_read_status(pipe.status)}), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="conduit", choices=["conduit", "reference"])
    ap.add_argument("--config", default="batched", choices=sorted(DESCR))
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--reference-step-seconds", type=float, default=None,
                    help="oracle time budget per reference step (default: about 150 s over the run)")
    ap.add_argument("--value-norm", default="v", choices=["v", "side_cache", "none"],
                    help="value norms from V (default), the side cache (Sec. 4.3), or none")
    ap.add_argument("--statistic", default="mean", choices=["mean", "rms"],
                    help="attention statistic in s: mean (Eq. 6, default) or RMS (Eq. 4)")
    ap.add_argument("--selection", default="global", choices=["global", "quota"],
                    help="one global top-k (default) or explicit per-image quotas (App. D.3)")
    ap.add_argument("--full-context", action="store_true",
                    help="softmax denominators include outside keys (seeded log-sum-exps)")
    ap.add_argument("--ratio", type=float, default=None,
                    help="refresh ratio r for every request (default: the workload's own)")
    ap.add_argument("--diagnostic", default=None, choices=["staleness"],
                    help="run the App. D staleness diagnostic instead of the step")
    ap.add_argument("--profile", action="store_true",
                    help="eager steps only, for ncu captures (no timing, e2e or CPU leg)")
    ap.add_argument("--requests", type=int, default=None,
                    help="with --profile: the first N requests of the workload")
    args = ap.parse_args()
    if args.profile:
        run_profile(args)
    elif args.diagnostic == "staleness":
        run_staleness(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_conduit(args)


if __name__ == "__main__":
    main()
