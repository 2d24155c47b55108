#!/usr/bin/env python
"""Benchmark of the token-selection path (score -> top-k -> gather) on GB300.

One step = one pass of the whole path over one batch of synthetic input:
litevlm_select_score_topk and litevlm_select_compact through the C-ABI, inputs
resident in HBM. Prints ONE JSON line (rank 0). When a step's inputs are
larger than L2 (no flush between steps) the line's throughput comes from K
steps with consecutive batches overlapped (the gather of one step under the
scores of the next, as a server runs a stream of batches); the per-step
figures and the sequential throughput are reported beside it.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--ratio R]
  python bench.py --impl reference ...   # the CPU oracle, timed on the host cores

Workloads (paper_2506_07416_gb300/inputs.py): sweep (default; 128 requests x
(6 views x 576 = 3456 visual + 64 text tokens), 32 heads x 128, hidden 4096,
keep 30%; --ratio 0.1/0.2/0.3/0.5), single, highres, fp8_ragged. The default
run also measures the other three workloads and reports each one's full record
under "workloads" (--workloads none skips them).
Multi-GPU: one process per GPU (torchrun), each rank runs its own batch
(weak scaling, no collective on the data path); time = max over ranks.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "visual tokens scored+selected per sec (M/s), % of HBM/tensor roofline, p50 µs"
UNIT = "M visual tokens/s"
# (timed steps, warm-up steps) of the headline run; the sub-records of the other workloads take SUB_STEPS
DEFAULTS = {"single": (3000, 50), "highres": (2000, 30), "fp8_ragged": (200, 10), "sweep": (20, 5)}
SUB_STEPS = {"single": (500, 20), "highres": (300, 10), "fp8_ragged": (60, 5), "sweep": (10, 3)}
KERNEL_SOURCES = ["paper_2506_07416_gb300/csrc/score_tc.cu", "paper_2506_07416_gb300/csrc/score_res.cu",
                  "paper_2506_07416_gb300/csrc/pipe.cuh", "paper_2506_07416_gb300/csrc/ptx.cuh",
                  "paper_2506_07416_gb300/csrc/score.h"]
# the files each score kernel is compiled from: its own source and the shared headers
KERNEL_FILES = {"score_tc": [KERNEL_SOURCES[0]] + KERNEL_SOURCES[2:],
                "score_res": KERNEL_SOURCES[1:]}
WORKLOADS = ["sweep", "single", "highres", "fp8_ragged"]


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=None)
    ap.add_argument("--workload", default="sweep", choices=WORKLOADS)
    ap.add_argument("--ratio", type=float, default=None, help="keep ratio override (sweep: 0.1/0.2/0.3/0.5)")
    ap.add_argument("--batch", type=int, default=None, help="use only the first B requests (profiling)")
    ap.add_argument("--workloads", default="auto",
                    help="other workloads measured after the headline one, comma-separated, or 'none'; "
                         "auto: the three others when the headline is the default sweep on one GPU")
    ap.add_argument("--score-kernel", default="auto", choices=["auto", "reread", "resident", "resident_1buf",
                                                                     "resident_2buf", "resident_flat"])
    ap.add_argument("--query-split", default="whole", choices=["whole", "split"],
                    help="resident plans for T > 64: each head's text rows whole, or as two pseudo-heads")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-next", action="store_true", help="skip the next-row measurements (splice, ...)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="bounded CPU work for the oracle baseline")
    ap.add_argument("--e2e-steps", type=int, default=None)
    ap.add_argument("--measure-fp8-peak", action="store_true",
                    help="time a cuBLASLt e4m3 GEMM (torch._scaled_mm) and print its TFLOP/s, nothing else")
    return ap.parse_args(argv)


def sub_workloads(args, world: int):
    """The workloads measured after the headline one (full records under "workloads")."""
    if args.workloads == "none":
        return []
    if args.workloads == "auto":
        if world > 1 or args.workload != "sweep" or args.batch is not None:
            return []
        return [n for n in WORKLOADS if n != args.workload]
    names = [n.strip() for n in args.workloads.split(",") if n.strip()]
    for n in names:
        if n not in WORKLOADS:
            raise SystemExit(f"unknown workload {n!r}")
    return [n for n in names if n != args.workload]


# ----------------------------------------------------------------------------- work accounting

def workload_for(args, name=None):
    from paper_2506_07416_gb300 import inputs
    w = inputs.workload(name or args.workload)
    if name is None and args.ratio is not None:
        from dataclasses import replace
        w = replace(w, keep_ratio=args.ratio, keep_k=None)
    if name is None and args.batch is not None and args.batch < w.batch:
        w = inputs.sub_batch(w, list(range(args.batch)))
    return w


def algorithmic(w):
    """Bytes and FLOPs the method itself moves / computes per step (no re-reads).
    The kept counts come from the library's own keep-count call."""
    from paper_2506_07416_gb300 import select
    e = 2 if w.dtype == "bf16" else 1
    off = select.keep_offsets(w.seq_offsets(), w.keep_k, float(w.keep_ratio or 0.0))
    ks = [int(x) for x in np.diff(off)]
    rb = w.row_bytes()
    row_total = sum(rb[n] for n in w.gather)
    score_bytes = sum(n * w.hkv * w.head_dim * e + t * w.hq * w.head_dim * e + 4 * n for n, t in zip(w.n_vis, w.n_txt))
    score_flops = sum(2 * w.hq * t * n * w.head_dim for n, t in zip(w.n_vis, w.n_txt))
    topk_bytes = sum(4 * n + 4 * k for n, k in zip(w.n_vis, ks))
    compact_bytes = sum(2 * k * row_total + 4 * k for k in ks)
    return {"score_bytes": score_bytes, "score_flops": score_flops, "topk_bytes": topk_bytes,
            "compact_bytes": compact_bytes, "kept": ks, "row_total": row_total}


def stage_rooflines(alg, stage_us, step_us, pk, dtype):
    """Roofline of each stage and of the whole step.

    A stage's roofline time is the slower of its FLOPs at the tensor peak and
    its algorithmic bytes at the HBM peak. `frac` = roofline time / measured
    time. The step's roofline is the sum over the three stages, against the
    measured step time (events at step boundaries). The e4m3 tensor peak is
    the measured bf16 peak times the nominal 2:1 ratio of the two."""
    hbm = pk["hbm_gbs"] * 1e9
    tensor = pk["bf16_tflops"] * 1e12 * (1.0 if dtype == "bf16" else 2.0)
    work = {"score": (alg["score_flops"], alg["score_bytes"]), "topk": (0, alg["topk_bytes"]),
            "compact": (0, alg["compact_bytes"])}
    out = {}
    total = 0.0
    for name, (flops, nbytes) in work.items():
        t_flops, t_bytes = flops / tensor * 1e6, nbytes / hbm * 1e6
        roof_us = max(t_flops, t_bytes)
        total += roof_us
        measured = float(stage_us[name])
        out[name] = {"bound": "tensor" if t_flops > t_bytes else "hbm", "algorithmic_bytes": int(nbytes),
                     "flops": int(flops), "roofline_us": roof_us, "measured_us": measured,
                     "frac": roof_us / measured if measured > 0 else None}
    out["step"] = {"roofline_us": total, "measured_us": float(step_us),
                   "frac": total / step_us if step_us > 0 else None}
    out["peaks"] = {"hbm_gbs": pk["hbm_gbs"], "tensor_tflops": tensor / 1e12,
                    "source": pk["source"] + (" (bf16 burst)" if dtype == "bf16" else
                                              " (bf16 burst x 2, the nominal e4m3 ratio)")}
    return out


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def kernel_source_sha(kernel=None):
    """First 16 hex digits of the sha256 of the score kernels' sources: all of
    them (kernel=None), or the files one kernel is compiled from ("score_tc",
    "score_res")."""
    h = hashlib.sha256()
    for f in (KERNEL_FILES[kernel] if kernel else KERNEL_SOURCES):
        h.update(open(os.path.join(ROOT, f), "rb").read())
    return h.hexdigest()[:16]


def committed_traffic(workload):
    """DRAM bytes per score launch from the committed ncu summary, if it was
    taken on the current sources of the kernel that serves the workload; else
    None."""
    p = os.path.join(ROOT, "profiles", "score_traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p))
    ent = d.get(workload)
    if not ent:
        return None
    kernel = "score_res" if ent.get("kernel", "").startswith("score_res") else "score_tc"
    if ent.get("kernel_sha") != kernel_source_sha(kernel):
        return None
    return ent.get("dram_bytes_per_launch")


def config_of(w):
    """The workload as the JSON line names it (the same for both arms)."""
    return {"workload": f"{w.name}: {w.description}", "batch": w.batch, "visual_tokens": w.total_vis,
            "text_tokens": w.total_txt, "q_heads": w.hq, "kv_heads": w.hkv, "head_dim": w.head_dim,
            "keep": (f"ratio {w.keep_ratio}" if w.keep_k is None else "keep_k per request"),
            "gather": list(w.gather)}


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, ValueError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.12)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- CPU oracle

def host_cores() -> int:
    """Host cores this process may run on."""
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


def oracle_sample(w):
    """A bounded sample of the workload for the CPU oracle: whole requests."""
    from paper_2506_07416_gb300 import inputs
    if w.batch == 1:
        return w, [0]
    reqs = [0, w.batch // 2]
    return inputs.sub_batch(w, reqs), reqs


def _oracle_runs(ws, x, seconds: float, threads: int, max_runs: int = 1000):
    import oracle
    runs, t0 = 0, time.perf_counter()
    while True:
        oracle.select(x, ws.hq, ws.hkv, ws.head_dim, ws.dtype, keep_k=ws.keep_k, keep_ratio=ws.keep_ratio or 0.0,
                      gather=ws.gather, threads=threads)
        runs += 1
        el = time.perf_counter() - t0
        if el >= seconds or runs >= max_runs:
            return runs, el


def time_oracle(w, seconds: float):
    """Runs the oracle (score + top-k + gather) on a bounded sample, on all the
    host cores this process may use (the threaded score, bit-identical to the
    serial one) for about seconds / 2, and on one thread for about seconds / 2.
    Returns the cpu_baseline record (value = the all-cores rate)."""
    from paper_2506_07416_gb300 import inputs
    ws, reqs = oracle_sample(w)
    x = inputs.make_numpy(ws)
    cores = host_cores()
    runs_n, el_n = _oracle_runs(ws, x, seconds / 2, cores)
    runs_1, el_1 = _oracle_runs(ws, x, seconds / 2, 1)
    v_n = ws.total_vis * runs_n / el_n / 1e6
    v_1 = ws.total_vis * runs_1 / el_1 / 1e6
    desc = (f"the whole path (fp64 scores, full-sort top-k, row copies) on request(s) {reqs} of the workload "
            f"({ws.total_vis} visual tokens per run): {runs_n} run(s) in {el_n:.1f} s on {cores} threads "
            f"(scores threaded over (head, query) rows, then over tokens, in the serial summation order), "
            f"{runs_1} run(s) in {el_1:.1f} s on one thread")
    return {"value": v_n, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc,
            "single_thread": {"value": v_1, "unit": UNIT, "cores": 1, "runs": runs_1, "seconds": el_1},
            "all_cores": {"value": v_n, "unit": UNIT, "cores": cores, "runs": runs_n, "seconds": el_n}}


def whole_job(local_total_ms: float, tokens_per_rank: int, world: int, device):
    """The job's time is its slowest rank's: the max of the ranks' timed totals
    (an all-reduce when world > 1), and the whole-job rate is the tokens of all
    ranks over that time, in M/s. Returns (time_ms, rate)."""
    total_ms = local_total_ms
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([total_ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    return total_ms, tokens_per_rank * world / (total_ms / 1e3) / 1e6


def rank_seed(base_seed: int, rank: int) -> int:
    """Each rank draws its own batch (replicas: the same shapes, other values)."""
    return base_seed + 1000 * rank


def run_reference(args):
    """The reference arm: the CPU oracle as it stands, on the host cores, each
    step the whole path on a bounded sample of the workload (rank 0 only)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w = workload_for(args)
    steps = args.steps if args.steps is not None else 3
    warm = args.warmup if args.warmup is not None else 1
    import oracle
    from paper_2506_07416_gb300 import inputs
    ws, reqs = oracle_sample(w)
    x = inputs.make_numpy(ws)
    cores = host_cores()

    def one():
        oracle.select(x, ws.hq, ws.hkv, ws.head_dim, ws.dtype, keep_k=ws.keep_k, keep_ratio=ws.keep_ratio or 0.0,
                      gather=ws.gather, threads=cores)

    for _ in range(warm):
        one()
    times = []
    for _ in range(steps):
        t0 = time.perf_counter()
        one()
        times.append(time.perf_counter() - t0)
    tot = sum(times)
    value = ws.total_vis * steps / tot / 1e6
    desc = (f"each step: the whole path on request(s) {reqs} of the workload ({ws.total_vis} visual tokens), "
            f"scores threaded over {cores} host cores")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": steps, "warmup": warm, "ms_per_step": tot / steps * 1e3,
            "p50_us": statistics.median(times) * 1e6, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config_of(w),
            "sample_requests": reqs,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- our path

def run_ours(args):
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    w = workload_for(args)
    steps_d, warm_d = DEFAULTS[w.name]
    steps = args.steps if args.steps is not None else steps_d
    warm = args.warmup if args.warmup is not None else warm_d
    rec = measure(args, w, steps, warm, dev, rank, world, full=True)

    subs = {}
    for name in sub_workloads(args, world):
        ws = workload_for(args, name)
        s_steps, s_warm = SUB_STEPS[name]
        r = measure(args, ws, s_steps, max(3, s_warm), dev, rank, world, full=False)
        subs[name] = {k: r[k] for k in ("value", "unit", "steps", "warmup", "ms_per_step", "p50_us", "p10_us",
                                        "p90_us", "warm", "dtype", "config", "score_launch", "stages_p50_us",
                                        "stages_roofline", "roofline", "e2e", "gpu_launches", "clocks", "l2",
                                        "sequential")}
        if r.get("pipelined"):
            subs[name]["pipelined"] = r["pipelined"]

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = time_oracle(w, args.cpu_seconds)

    line = {"metric": METRIC, "value": rec["value"], "unit": UNIT, "n_gpus": world, "steps": steps, "warmup": warm,
            "ms_per_step": rec["ms_per_step"], "p50_us": rec["p50_us"], "p10_us": rec["p10_us"],
            "p90_us": rec["p90_us"], "warm": rec["warm"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": rec["dtype"],
            "data": "synthetic (seeded; shapes of the paper's multi-camera workloads)",
            "config": rec["config"], "l2": rec["l2"],
            "parallelism": f"replicas x{world}, one batch per GPU, no collective",
            "score_launch": rec["score_launch"], "stages_p50_us": rec["stages_p50_us"],
            "stages_roofline": rec["stages_roofline"], "roofline": rec["roofline"], "cpu_baseline": cpu,
            "e2e": rec["e2e"], "next": rec.get("next"), "workloads": subs or None,
            "gpu_launches": rec["gpu_launches"], "clocks": rec["clocks"], "wall_s": rec["wall_s"]}
    line["sequential"] = rec["sequential"]
    if rec.get("pipelined"):
        line["pipelined"] = rec["pipelined"]
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def run_pipelined(w, steps, stream, select_call, gather_call, kept, off_d, c_src, dev):
    """K steps with consecutive batches overlapped: the scores and top-k of step
    i + 1 run on the main stream while the gather of step i runs on a second
    one (kept indices and offsets double-buffered; a step's select waits for
    the gather that last read its buffers). Timed from the first launch to the
    end of the last gather, with CUDA events."""
    import torch
    side = torch.cuda.Stream(device=dev)
    kept2 = [kept, torch.empty_like(kept)]
    off2 = [off_d, torch.empty_like(off_d)]
    ev_sel = [torch.cuda.Event() for _ in range(steps)]
    ev_gat = [torch.cuda.Event() for _ in range(steps)]
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    t0.record(stream)
    for i in range(steps):
        if i >= 2:
            stream.wait_event(ev_gat[i - 2])
        select_call(*select_call.args_, stream.cuda_stream, kept2[i % 2], off2[i % 2])
        ev_sel[i].record(stream)
        side.wait_event(ev_sel[i])
        gather_call(kept2[i % 2], c_src, side.cuda_stream)
        ev_gat[i].record(side)
    stream.wait_event(ev_gat[steps - 1])
    t1.record(stream)
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    return {"ms_total": ms, "ms_per_step": ms / steps,
            "timing": "K steps, the gather of step i on a second stream overlapping the scores and top-k of step "
                      "i + 1 (kept indices and offsets double-buffered); CUDA events from the first launch to the "
                      "end of the last gather"}


def measure(args, w, steps, warm_steps, dev, rank, world, full):
    """Times `steps` steps of the path on workload w (after `warm_steps`
    untimed ones) and returns the record: the whole-job rate, step percentiles,
    stage times and rooflines, the clocks seen, and the end-to-end figure
    (full=True: also the e2e variants and the next-row measurements)."""
    import torch
    import torch.distributed as dist

    from paper_2506_07416_gb300 import inputs, select

    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    alg = algorithmic(w)

    xd = inputs.make_torch(w, dev, seed=rank_seed(w.seed, rank))
    so_h, to_h = w.seq_offsets(), w.text_offsets()
    kk_h = None if w.keep_k is None else np.asarray(w.keep_k, np.int32)
    kk_d = None if kk_h is None else torch.from_numpy(kk_h).to(dev)
    ratio = float(w.keep_ratio or 0.0)
    total_kept = int(sum(alg["kept"]))
    sel = select.Selector(w.batch, w.total_vis, w.total_txt, w.hq, w.hkv, w.head_dim, w.dtype,
                          score_kernel=args.score_kernel, query_split=args.query_split)
    h = sel.handle
    scores = torch.empty(w.total_vis, dtype=torch.float32, device=dev)
    kept = torch.empty(max(1, total_kept), dtype=torch.int32, device=dev)
    off_d = torch.empty(w.batch + 1, dtype=torch.int32, device=dev)
    off_h = np.zeros(w.batch + 1, np.int32)
    srcs = [xd[n] for n in w.gather]
    dsts = [torch.empty((max(1, total_kept),) + tuple(s.shape[1:]), dtype=s.dtype, device=dev) for s in srcs]
    rb = [s[0].numel() * s.element_size() for s in srcs]

    L = select.LIB
    c_so_h, c_to_h = so_h.ctypes.data, to_h.ctypes.data
    c_kk_h = None if kk_h is None else kk_h.ctypes.data
    c_kk_d = None if kk_d is None else kk_d.data_ptr()
    n_t = len(srcs)
    c_src = (ctypes.c_void_p * n_t)(*[s.data_ptr() for s in srcs])
    c_dst = (ctypes.c_void_p * n_t)(*[d.data_ptr() for d in dsts])
    c_rb = (ctypes.c_int64 * n_t)(*rb)

    def call(rc):
        if rc != 0:
            raise select.LitevlmError(rc, L.litevlm_select_last_error(h).decode())

    def select_call(q, k, so_d, to_d, s_ptr, kept_t, off_t):
        """Scores and top-k in one call (the top-k kernel adds the head-group
        partials); returns the kernels launched."""
        call(L.litevlm_select_score_topk(h, w.batch, q.data_ptr(), to_d.data_ptr(), c_to_h, k.data_ptr(),
                                         so_d.data_ptr(), c_so_h, xd["q_scale"], xd["k_scale"], scores.data_ptr(),
                                         c_kk_d, c_kk_h, ratio, kept_t.data_ptr(), off_t.data_ptr(),
                                         off_h.ctypes.data, s_ptr))
        return L.litevlm_select_last_launches(h)

    def gather_call(kept_t, srcs, s_ptr):
        call(L.litevlm_select_compact(h, total_kept, kept_t.data_ptr(), w.total_vis, n_t, srcs, c_dst, c_rb, s_ptr))
        return L.litevlm_select_last_launches(h)

    def step(q, k, so_d, to_d, hidden_srcs=None, s_ptr=None):
        """One step: scores and top-k, then the gather; returns the kernels launched."""
        st_ = sp if s_ptr is None else s_ptr
        n = select_call(q, k, so_d, to_d, st_, kept, off_d)
        return n + gather_call(kept, hidden_srcs if hidden_srcs is not None else c_src, st_)

    q, k, so_d, to_d = xd["q"], xd["k"], xd["seq_offsets"], xd["text_offsets"]
    select_call.args_ = (q, k, so_d, to_d)
    launches_per_step = 0
    for _ in range(warm_steps):
        launches_per_step = step(q, k, so_d, to_d)
    sel.check_device()

    # L2: flush between timed steps unless the step's inputs are larger than L2
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    step_bytes = alg["score_bytes"] + alg["compact_bytes"]
    flush = None
    if step_bytes < 2 * l2:
        flush = torch.empty(max(8 * l2, 1 << 30) // 4, dtype=torch.int32, device=dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
    ev_stage = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
    plan = sel.score_plan(to_h, so_h)

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clk = ClockSampler(dev.index or 0)
    clk.start()
    time.sleep(0.15)
    wall0 = time.perf_counter()
    for i in range(steps):
        if flush is not None:
            flush.fill_(i)
        e = ev[i]
        e[0].record(stream)
        step(q, k, so_d, to_d)
        e[3].record(stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - wall0
    # With inputs larger than L2 (no flush between steps) the line's throughput
    # comes from K steps with consecutive batches overlapped, as a server runs
    # them; the per-step figures (p50, stages) stay those of the sequential steps.
    pipelined = None
    if flush is None:
        pipelined = run_pipelined(w, steps, stream, select_call, gather_call, kept, off_d, c_src, dev)
    # Stage times for the roofline: the same calls with events between the
    # kernels (an event between two kernels keeps the second from launching
    # early, so these steps are not part of the step timing above)
    for i in range(steps):
        if flush is not None:
            flush.fill_(steps + i)
        e = ev_stage[i]
        e[0].record(stream)
        call(L.litevlm_select_score(h, w.batch, q.data_ptr(), to_d.data_ptr(), c_to_h, k.data_ptr(),
                                    so_d.data_ptr(), c_so_h, xd["q_scale"], xd["k_scale"], scores.data_ptr(), sp))
        e[1].record(stream)
        call(L.litevlm_select_topk(h, w.batch, scores.data_ptr(), so_d.data_ptr(), c_so_h, c_kk_d, c_kk_h, ratio,
                                   kept.data_ptr(), off_d.data_ptr(), off_h.ctypes.data, sp))
        e[2].record(stream)
        call(L.litevlm_select_compact(h, total_kept, kept.data_ptr(), w.total_vis, n_t, c_src, c_dst, c_rb, sp))
        e[3].record(stream)
    torch.cuda.synchronize()
    # Warm steps (inputs left in L2 by the previous step), reported beside the
    # cold ones when the timed steps flush L2. A GPU spin queued first lets the
    # host enqueue every step before the GPU reaches them, so the events
    # bracket GPU work only.
    warm_stats = None
    if flush is not None:
        n_warm = min(steps, 500)
        ev_warm = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(n_warm)]
        step(q, k, so_d, to_d)
        with torch.cuda.stream(stream):
            torch.cuda._sleep(100_000 * n_warm)
        for e0, e1 in ev_warm:
            e0.record(stream)
            step(q, k, so_d, to_d)
            e1.record(stream)
        torch.cuda.synchronize()
        wt = np.array([a.elapsed_time(b) for a, b in ev_warm]) * 1e3
        warm_stats = {"p10_us": float(np.percentile(wt, 10)), "p50_us": float(np.median(wt)),
                      "p90_us": float(np.percentile(wt, 90)), "steps": n_warm,
                      "timing": "the same step back to back without the L2 flush, events at step boundaries"}
    clocks = clk.stop()
    if world > 1:
        dist.barrier()
    sel.check_device()

    per_step_ms = np.array([e[0].elapsed_time(e[3]) for e in ev])
    st = np.array([[e[0].elapsed_time(e[1]), e[1].elapsed_time(e[2]), e[2].elapsed_time(e[3])] for e in ev_stage])
    seq_total_ms, seq_value = whole_job(float(per_step_ms.sum()), w.total_vis * steps, world, dev)
    if pipelined is not None:
        total_ms, value = whole_job(float(pipelined["ms_total"]), w.total_vis * steps, world, dev)
    else:
        total_ms, value = seq_total_ms, seq_value

    pk = peaks()
    score_us = float(st[:, 0].mean() * 1e3)
    ai = alg["score_flops"] / alg["score_bytes"]
    ridge = pk["bf16_tflops"] * 1e12 / (pk["hbm_gbs"] * 1e9)
    if ai < ridge or w.dtype != "bf16":
        achieved = alg["score_bytes"] / (score_us * 1e-6) / 1e9
        roof = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / pk["hbm_gbs"], "traffic": committed_traffic(w.name),
                "kernel": select.KERNELS.get(plan[0], "score"),
                "algorithmic_bytes_per_launch": alg["score_bytes"], "peak_source": pk["source"] + " (burst copy)",
                "duration_us": score_us, "duration_source": "mean CUDA-event time of the score call, stage pass"}
    else:
        achieved = alg["score_flops"] / (score_us * 1e-6) / 1e12
        roof = {"bound": "tensor", "achieved": achieved, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                "frac": achieved / pk["bf16_tflops"], "traffic": committed_traffic(w.name),
                "kernel": select.KERNELS.get(plan[0], "score"), "algorithmic_flops_per_launch": alg["score_flops"],
                "peak_source": pk["source"] + " (burst cuBLAS bf16)",
                "duration_us": score_us, "duration_source": "mean CUDA-event time of the score call, stage pass"}

    nxt = None
    if full and not args.no_next:
        # next-step rows, each timed on its own after the step: prefill splice
        # (32 system rows and the text rows of every request around its kept
        # visual rows), full-key scores, view gating, layer-0 projection
        nxt = {"splice": run_splice(w, xd, sel, kept, off_d, off_h, dev, stream, steps, flush, pk),
               "full_keys": run_full_keys(w, xd, sel, dev, stream, steps, flush, pk),
               "views": run_views(w, sel, dev, stream, steps),
               "project": run_project(w, xd, sel, dev, stream, steps, pk)}

    # end to end through the public API with host buffers
    calls = (select_call, gather_call)
    e2e = run_e2e(args, w, xd, calls, dev, stream, kept, off_d, total_kept, sel)
    if full:
        e2e["copy_all_inputs"] = run_e2e(args, w, xd, calls, dev, stream, kept, off_d, total_kept, sel,
                                         gather_from_host=False)
        e2e["eager"] = run_e2e(args, w, xd, calls, dev, stream, kept, off_d, total_kept, sel, graph=False)

    stage_us = {n: float(np.median(st[:, i]) * 1e3) for i, n in enumerate(("score", "topk", "compact"))}
    stage_us["timing"] = ("a second pass with CUDA events between the separate calls (score with its own "
                          "head-group fold, top-k, gather); the timed steps use the one-call score + top-k, "
                          "whose top-k kernel adds the head-group partials, with events at step boundaries only")
    rec = {"value": value, "unit": UNIT, "steps": steps, "warmup": warm_steps, "ms_per_step": total_ms / steps,
           "p50_us": float(np.median(per_step_ms) * 1e3), "p10_us": float(np.percentile(per_step_ms, 10) * 1e3),
           "p90_us": float(np.percentile(per_step_ms, 90) * 1e3), "warm": warm_stats,
           "dtype": "bf16" if w.dtype == "bf16" else "e4m3", "config": config_of(w),
           "kept_tokens": total_kept,
           "l2": ("flushed between timed steps (write of %d MB); steps run one after another" % (flush.numel() * 4 >> 20))
           if flush is not None else "inputs larger than L2, no flush; consecutive steps overlapped (pipelined)",
           "sequential": {"value": seq_value, "ms_per_step": seq_total_ms / steps,
                          "timing": "the same K steps one after another on one stream, events at step "
                                    "boundaries (p50_us, p10_us, p90_us and the step roofline come from these)"},
           "score_launch": {"kernel": select.KERNELS.get(plan[0]), "cluster": plan[1], "tiles_per_cta": plan[2],
                            "head_groups": plan[3]},
           "stages_p50_us": stage_us,
           "stages_roofline": stage_rooflines(alg, stage_us, float(np.median(per_step_ms) * 1e3), pk, w.dtype),
           "roofline": roof, "e2e": e2e, "next": nxt, "gpu_launches": launches_per_step * steps,
           "clocks": clocks, "wall_s": wall}
    if pipelined is not None:
        rec["pipelined"] = pipelined
    sel.close()
    del xd, dsts, scores, kept, flush
    torch.cuda.empty_cache()
    return rec


def run_splice(w, xd, sel, kept, off_d, off_h, dev, stream, steps, flush, pk):
    """litevlm_select_splice on the step's kept indices: [32 system rows; kept
    visual rows; text rows] per request, rows of `hidden` bf16, with position ids."""
    import torch
    from paper_2506_07416_gb300 import select
    n_sys = 32
    rb = w.hidden * 2
    g = torch.Generator(device=dev).manual_seed(7)
    sys_rows = torch.randn((n_sys * w.batch, w.hidden), generator=g, device=dev).to(torch.bfloat16)
    txt_rows = torch.randn((max(1, w.total_txt), w.hidden), generator=g, device=dev).to(torch.bfloat16)
    sys_h = np.arange(0, n_sys * (w.batch + 1), n_sys, dtype=np.int32)
    sys_d = torch.from_numpy(sys_h).to(dev)
    so_h, to_h = w.seq_offsets(), w.text_offsets()
    total = int(sys_h[-1] + off_h[-1] + to_h[-1])
    out = torch.empty((max(total, 1), w.hidden), dtype=torch.bfloat16, device=dev)
    pos = torch.empty(max(total, 1), dtype=torch.int32, device=dev)
    out_off = torch.empty(w.batch + 1, dtype=torch.int32, device=dev)
    L = select.LIB
    args = (sel.handle, w.batch, sys_rows.data_ptr(), sys_d.data_ptr(), sys_h.ctypes.data, xd["hidden"].data_ptr(),
            xd["seq_offsets"].data_ptr(), so_h.ctypes.data, kept.data_ptr(), off_d.data_ptr(), off_h.ctypes.data,
            txt_rows.data_ptr(), xd["text_offsets"].data_ptr(), to_h.ctypes.data, rb, out.data_ptr(),
            out_off.data_ptr(), None, pos.data_ptr(), stream.cuda_stream)
    n = max(3, min(steps, 200))
    for _ in range(3):
        assert L.litevlm_select_splice(*args) == 0
    ts = []
    for i in range(n):
        if flush is not None:
            flush.fill_(i)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        assert L.litevlm_select_splice(*args) == 0
        e1.record(stream)
        ts.append((e0, e1))
    torch.cuda.synchronize()
    sel.check_device()
    us = float(np.median([a.elapsed_time(b) for a, b in ts]) * 1e3)
    alg = 2 * total * rb + 4 * total
    gbs = alg / (us * 1e-6) / 1e9
    return {"us_p50": us, "rows": total, "row_bytes": rb, "algorithmic_bytes": alg, "achieved_gbs": gbs,
            "frac_of_hbm": gbs / pk["hbm_gbs"], "system_rows_per_request": n_sys}


def run_full_keys(w, xd, sel, dev, stream, steps, flush, pk):
    """litevlm_select_score_full_keys against litevlm_select_score on the same
    batch: the softmax over [32 system keys; visual keys; causal text keys] per
    request. Both calls timed alone (CUDA events, median); the difference is
    the cost of the context-key statistics kernel and the merge."""
    import torch
    from paper_2506_07416_gb300 import inputs, select
    n_sys = 32
    c = inputs.context_keys_torch(w, [n_sys] * w.batch, dev, k_scale=xd["k_scale"])
    sys_h = np.arange(0, n_sys * (w.batch + 1), n_sys, dtype=np.int32)
    so_h, to_h = w.seq_offsets(), w.text_offsets()
    scores = torch.empty(max(1, w.total_vis), dtype=torch.float32, device=dev)
    L = select.LIB
    base = (sel.handle, w.batch, xd["q"].data_ptr(), xd["text_offsets"].data_ptr(), to_h.ctypes.data,
            xd["k"].data_ptr(), xd["seq_offsets"].data_ptr(), so_h.ctypes.data)
    tail = (xd["q_scale"], xd["k_scale"], scores.data_ptr(), stream.cuda_stream)
    full = base + (c["k_sys"].data_ptr(), c["sys_offsets"].data_ptr(), sys_h.ctypes.data, c["k_txt"].data_ptr()) + tail
    calls = {"visual_keys": lambda: L.litevlm_select_score(*base, *tail),
             "full_keys": lambda: L.litevlm_select_score_full_keys(*full)}
    n = max(3, min(steps, 200))
    us = {}
    for name, fn in calls.items():
        for _ in range(3):
            assert fn() == 0
        ts = []
        for i in range(n):
            if flush is not None:
                flush.fill_(i)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            assert fn() == 0
            e1.record(stream)
            ts.append((e0, e1))
        torch.cuda.synchronize()
        us[name] = float(np.median([a.elapsed_time(b) for a, b in ts]) * 1e3)
    sel.check_device()
    rb = w.head_dim * (2 if w.dtype == "bf16" else 1)
    # context-key statistics: q rows and the system / text key rows once, e[t][h] out
    ctx_bytes = (w.total_txt * w.hq + (n_sys * w.batch + w.total_txt) * w.hkv) * rb + w.total_txt * w.hq * 4
    return {"us_p50": us["full_keys"], "visual_keys_us_p50": us["visual_keys"],
            "extra_us": us["full_keys"] - us["visual_keys"], "system_keys_per_request": n_sys,
            "context_algorithmic_bytes": ctx_bytes,
            "tokens_per_s_M": w.total_vis / (us["full_keys"] * 1e-6) / 1e6}


def run_project(w, xd, sel, dev, stream, steps, pk):
    """litevlm_select_project: the keys of the workload's visual rows from their
    hidden states (RMSNorm folded into a random W_k [Hkv*d, hidden], RoPE at
    positions 32 + j), at most 65536 rows, timed alone (CUDA events, median),
    with a plain cuBLAS bf16 GEMM of the same shape (no norm, no rotation) timed
    beside it for reference."""
    import torch
    from paper_2506_07416_gb300 import select
    rows = min(w.total_vis, 65536)
    H, O, d = w.hidden, w.hkv * w.head_dim, w.head_dim
    if O % 128 != 0 or H % 8 != 0:
        return None
    g = torch.Generator(device=dev).manual_seed(17)
    x = xd["hidden"][:rows]
    wk = (torch.randn((O, H), generator=g, device=dev) / H ** 0.5).to(torch.bfloat16)
    gamma = torch.rand(H, generator=g, device=dev) + 0.5
    wf = sel.fold_norm(wk, gamma)
    table = sel.rope_table(rows + 64, d, 1e6)
    pos = (torch.arange(rows, device=dev, dtype=torch.int32) + 32).contiguous()
    y = torch.empty((rows, O), dtype=torch.bfloat16, device=dev)
    L = select.LIB
    args = (sel.handle, rows, H, O, x.data_ptr(), wf.data_ptr(), None, 1e-6, d, pos.data_ptr(), table.data_ptr(),
            rows + 64, 0.0, y.data_ptr(), stream.cuda_stream)
    n = max(3, min(steps, 50))
    res = {}
    def ours():
        assert L.litevlm_select_project(*args) == 0

    def plain():
        torch.matmul(x, wk.t(), out=y)

    for name, fn in (("ours", ours), ("cublas_plain_gemm", plain)):
        for _ in range(3):
            fn()
        ts = []
        for _ in range(n):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            ts.append((e0, e1))
        torch.cuda.synchronize()
        res[name] = float(np.median([a.elapsed_time(b) for a, b in ts]) * 1e3)
    sel.check_device()
    flops = 2.0 * rows * H * O
    tf = flops / (res["ours"] * 1e-6) / 1e12
    return {"rows": rows, "hidden": H, "out_features": O, "head_dim": d, "us_p50": res["ours"],
            "tflops": tf, "frac_of_bf16_peak": tf / pk["bf16_tflops"],
            "cublas_plain_gemm_us_p50": res["cublas_plain_gemm"],
            "cublas_plain_gemm_tflops": flops / (res["cublas_plain_gemm"] * 1e-6) / 1e12}


def run_views(w, sel, dev, stream, steps):
    """litevlm_select_views (patch-selection gating) on the workload's batch x 6
    camera views (2 tiles x 256 tokens each), timed alone (CUDA events, median)."""
    import torch
    from paper_2506_07416_gb300 import inputs, select
    nv = 6
    lex, lg = inputs.view_gating_numpy(w.batch, nv, seed=w.seed)
    lex_d, lg_d = torch.from_numpy(lex).to(dev), torch.from_numpy(lg).to(dev)
    tpv = np.full(nv, 512, np.int32)
    mask = torch.empty((w.batch, nv), dtype=torch.uint8, device=dev)
    vo = torch.empty(w.batch + 1, dtype=torch.int32, device=dev)
    sv = torch.empty(w.batch * nv, dtype=torch.int32, device=dev)
    so = torch.empty(w.batch + 1, dtype=torch.int32, device=dev)
    L = select.LIB
    args = (sel.handle, w.batch, nv, lex_d.data_ptr(), lg_d.data_ptr(), tpv.ctypes.data, 2.0, 1.0, 1.0, 1,
            mask.data_ptr(), vo.data_ptr(), sv.data_ptr(), so.data_ptr(), None, stream.cuda_stream)
    for _ in range(3):
        assert L.litevlm_select_views(*args) == 0
    n = max(3, min(steps, 200))
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    # the kernel takes a few microseconds, less than the host needs per call: a
    # spin on the GPU (about 50 us per call) lets the host queue every call
    # first, so each event pair brackets GPU work only, not host gaps
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        torch.cuda._sleep(100_000 * n)
    ts = []
    for e0, e1 in evs:
        e0.record(stream)
        assert L.litevlm_select_views(*args) == 0
        e1.record(stream)
        ts.append((e0, e1))
    torch.cuda.synchronize()
    sel.check_device()
    sel_views = int(vo[-1].item())
    return {"us_p50": float(np.median([a.elapsed_time(b) for a, b in ts]) * 1e3), "requests": w.batch,
            "views_per_request": nv, "selected_views": sel_views,
            "mean_views_selected": sel_views / max(1, w.batch)}


def run_e2e(args, w, xd, calls, dev, stream, kept, off_d, total_kept, sel, gather_from_host=True, graph=True):
    """Host buffers in, selection out, through the C-ABI, all inside the timed
    region: every step copies q, K and the offsets (packed in one pinned host
    buffer) to the device, runs the three calls, and reads the kept indices and
    offsets back into pinned host memory. Inputs are double-buffered on the
    device and copied on a second stream, so the copy of step i + 1 overlaps the
    kernels of step i (the way a serving loop would run it); each step's kernels
    wait for its own copy. The gather of step i runs on a third stream, so it
    overlaps the scores and top-k of step i + 1; the kept indices and offsets
    are double-buffered for that, and a step's input buffer is reused only
    after both its select and its gather are done.

    The gathered tensors other than K (hidden states, V) stay in pinned host
    memory and the gather reads only their kept rows through the device view
    (litevlm_select_host_view), so only those rows cross the host link
    (gather_from_host=True). With gather_from_host=False they are copied whole
    with the other inputs every step. h2d_bytes_per_step counts what crosses
    the link either way.

    graph=True: the calls of 8 consecutive steps (copies, the C-ABI calls with
    their kernels, result copies, and the events between the two streams) are
    captured once into a CUDA graph, which the timed loop replays, so the host
    issues one launch per 8 steps instead of about fifteen API calls per step.
    The device work is the same as in the eager loop (graph=False), whose time
    is bound by the host's issue rate on small workloads."""
    import torch
    host_gather = [n for n in w.gather if n != "k"] if gather_from_host else []
    names = ["q", "k", "seq_offsets", "text_offsets"] + [n for n in w.gather if n != "k" and n not in host_gather]
    sizes = {n: xd[n].numel() * xd[n].element_size() for n in names + host_gather}
    offs, tot = {}, 0
    for n in names:
        offs[n] = tot
        tot += (sizes[n] + 255) // 256 * 256
    host = torch.empty(tot, dtype=torch.uint8).pin_memory()
    for n in names:
        host[offs[n]:offs[n] + sizes[n]].copy_(xd[n].contiguous().view(-1).view(torch.uint8).cpu())
    # the host-resident gather sources and their device views
    resident = {n: xd[n].cpu().pin_memory() for n in host_gather}
    resident_view = {n: sel.host_view(resident[n]) for n in host_gather}
    bufs = [torch.empty(tot, dtype=torch.uint8, device=dev) for _ in range(2)]

    def views(buf):
        return {n: buf[offs[n]:offs[n] + sizes[n]].view(xd[n].dtype).view(xd[n].shape) for n in names}

    dv = [views(b) for b in bufs]
    c_srcs = [(ctypes.c_void_p * len(w.gather))(*[resident_view[n] if n in resident_view else d[n].data_ptr()
                                                  for n in w.gather]) for d in dv]
    res_h = torch.empty(kept.numel() + off_d.numel(), dtype=torch.int32).pin_memory()
    nk = kept.numel()
    steps = args.e2e_steps if args.e2e_steps is not None else max(3, min(200, (args.steps or DEFAULTS[w.name][0])))
    select_call, gather_call = calls
    kept2 = [kept, torch.empty_like(kept)]
    off2 = [off_d, torch.empty_like(off_d)]
    copy_stream = torch.cuda.Stream(device=dev)
    gather_stream = torch.cuda.Stream(device=dev)
    copied = [torch.cuda.Event() for _ in range(2)]
    selected = [torch.cuda.Event() for _ in range(2)]
    gathered = [torch.cuda.Event() for _ in range(2)]
    h2d = tot + sum(total_kept * (sizes[n] // xd[n].shape[0]) for n in host_gather)
    d2h = res_h.numel() * 4

    def one(i, st, wait_used=True):
        sl = i & 1
        with torch.cuda.stream(copy_stream):
            if wait_used:  # the select and the gather of step i - 2 are done with this buffer
                copy_stream.wait_event(selected[sl])
                copy_stream.wait_event(gathered[sl])
            bufs[sl].copy_(host, non_blocking=True)
            copied[sl].record(copy_stream)
        st.wait_event(copied[sl])
        if wait_used:
            st.wait_event(gathered[sl])  # the gather of step i - 2 has read kept2[sl]
        d = dv[sl]
        select_call(d["q"], d["k"], d["seq_offsets"], d["text_offsets"], st.cuda_stream, kept2[sl], off2[sl])
        selected[sl].record(st)
        with torch.cuda.stream(st):
            res_h[:nk].copy_(kept2[sl], non_blocking=True)
            res_h[nk:].copy_(off2[sl], non_blocking=True)
        gather_stream.wait_event(selected[sl])
        gather_call(kept2[sl], c_srcs[sl], gather_stream.cuda_stream)
        gathered[sl].record(gather_stream)

    for i in range(4):
        one(i, stream)
    torch.cuda.synchronize()
    per_graph = 8
    g = None
    if graph:
        cap = torch.cuda.Stream(device=dev)
        cap.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap, capture_error_mode="relaxed"):
            fork = torch.cuda.Event()
            fork.record(cap)
            copy_stream.wait_event(fork)  # the copy and gather streams join the capture
            gather_stream.wait_event(fork)
            for i in range(per_graph):
                # steps 0 and 1 of a replay follow the previous replay in stream order
                one(i, cap, wait_used=i >= 2)
            cap.wait_stream(copy_stream)  # and leave it
            cap.wait_stream(gather_stream)
        torch.cuda.synchronize()
        steps = max(per_graph, (steps + per_graph - 1) // per_graph * per_graph)
        g.replay()
        torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    copy_stream.wait_event(e0)
    gather_stream.wait_event(e0)
    if g is not None:
        with torch.cuda.stream(stream):
            for _ in range(steps // per_graph):
                g.replay()
    else:
        for i in range(steps):
            one(i, stream)
    stream.wait_stream(copy_stream)
    stream.wait_stream(gather_stream)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    if host_gather:
        api = ("litevlm_select_score_topk + compact" + (" (8 steps captured into a CUDA graph, replayed)" if g else "")
               + "; the gather of step i overlaps the select of step i + 1 (own stream)"
               + "; each step copies q, K and the offsets from one pinned host "
               "buffer into one of two device buffers on a copy stream; the gather reads the kept rows of "
               + ", ".join(host_gather) + " straight from pinned host memory (litevlm_select_host_view); "
               "kept indices + offsets copied back")
    else:
        api = ("litevlm_select_score_topk + compact" + (" (8 steps captured into a CUDA graph, replayed)" if g else "")
               + "; each step's inputs (gathered tensors included) copied from "
               "one pinned host buffer into one of two device buffers on a copy stream, kept indices + offsets "
               "copied back")
    return {"value": w.total_vis * steps / (ms / 1e3) / 1e6, "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": steps, "ms_per_step": ms / steps, "api": api}


def measure_fp8_peak(n: int = 8192, reps: int = 50):
    """Dense e4m3 x e4m3 -> bf16 GEMM throughput of the library GEMM (cuBLASLt
    through torch._scaled_mm), n x n x n, the e4m3 counterpart of the measured
    bf16 peak. Inputs far larger than L2 are not needed for a compute-bound GEMM."""
    import torch
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(0)
    a = torch.randn((n, n), generator=g, device=dev).to(torch.float8_e4m3fn)
    b = torch.randn((n, n), generator=g, device=dev).to(torch.float8_e4m3fn).t()  # column-major operand
    one = torch.ones((), device=dev)
    for _ in range(5):
        torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        torch._scaled_mm(a, b, scale_a=one, scale_b=one, out_dtype=torch.bfloat16)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    tf = 2.0 * n ** 3 / (ms * 1e-3) / 1e12
    print(json.dumps({"fp8_e4m3_tflops": tf, "n": n, "ms_per_gemm": ms, "library": "cuBLASLt via torch._scaled_mm",
                      "bf16_tflops_measured": peaks()["bf16_tflops"]}), flush=True)
    return 0


def main():
    args = parse_args()
    if args.measure_fp8_peak:
        return measure_fp8_peak()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
