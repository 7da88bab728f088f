#!/usr/bin/env python3
"""Benchmark of the ProViP in-LLM pruning step on GB300.

One step = one pass of the whole hot path over one batch: head-aware scores
(both passes), top-k with the fused score reduction, and the compaction of
hidden states, K, V and position ids (provip_prune). The workload is the
LLaVA-NeXT-7B anyres batch of 8 (2880 -> 960 visual tokens before the LLM,
960 -> 320 at the pruning layer; 32 heads x 128, hidden 4096, 96 text tokens,
8 selected heads), seeded synthetic data.

Timing: W warm-up steps, then exactly K steps replayed from CUDA graphs
(chunks of up to 100 steps) between CUDA events on the launching stream, with a
barrier and a device synchronisation on both sides; inputs rotate over three
device copies (3 x 286 MB, larger than the 129 MB L2). value = samples pruned
per second over all ranks (max time over ranks).

Extra keys: roofline of the dominant kernel (the compaction; its algorithmic
bytes per launch over its event-timed duration), the whole path's achieved
bandwidth, e2e through the C ABI with pinned host buffers (copies inside the
timed region), the fp64 oracle timed on the host cores (cpu_baseline), SM
clocks sampled with nvidia-smi during the timed region.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                  [--impl reference]
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "pruned samples/s for head_scores+topk+compact; % of GB300 HBM roofline"
UNIT = "samples/s"
DEFAULT_WORKLOAD = "llava_next_7b_bf16_b8"
FALLBACK_HBM_GBS = 6800.0
GRAPH_CHUNK = 100
N_COPIES = 3
L2_BYTES = 129e6  # GB300's L2; the rotating inputs of a timed loop span at least 3x this
N_VIS = 6  # visual heads per pruning layer (the paper's setting, Sec. 5.1)

# DRAM traffic of one compaction launch on the default workload, from the ncu
# capture summarised in profiles/ (null when the kernel source has changed
# since: the sha1 of the kernel file is checked at run time).
COMPACT_TRAFFIC = {"sha1": "4d447a409e84a515a32c928dcba8278a535f9f57", "bytes": 115457280,
                   "profile": "profiles/prune_llava_next_b8_kernels.md"}


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--algo", default="auto", choices=["auto", "simt", "tcgen05", "stream", "cluster"],
                    help="head-score kernel form (auto: tcgen05 for bf16, and the streaming form when "
                         "several single-sample streams run concurrently)")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--copies", type=int, default=N_COPIES, help="rotating device copies of the inputs")
    ap.add_argument("--compact-only", action="store_true",
                    help="time the compaction alone (provip_compact, no programmatic dependency) on --workload "
                         "and print one JSON line (the command the compaction profiles use)")
    ap.add_argument("--prellm-only", action="store_true",
                    help="time only the pre-LLM pass (provip_similarity_reduce) and print its JSON")
    ap.add_argument("--prellm-reps", type=int, default=20)
    ap.add_argument("--streams", type=int, default=None,
                    help="streams of independent batches run concurrently (default: 25 for "
                         "single-sample batches, else 2)")
    ap.add_argument("--target-s", type=float, default=1.0,
                    help="seconds of the timed region: the K-step graph is replayed that long, the "
                         "median repeat reported")
    ap.add_argument("--no-workloads", action="store_true",
                    help="skip the video workload block")
    ap.add_argument("--quick", action="store_true",
                    help="the headline steps only (no other legs): for profiler captures")
    return ap.parse_args(argv)


# ---------------------------------------------------------------------------
# distributed bookkeeping (one process per GPU; no collective on the data path)
# ---------------------------------------------------------------------------
class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local_rank = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None

    def init(self, backend):
        if self.world > 1:
            import torch.distributed as dist
            os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
            dist.init_process_group(backend=backend, rank=self.rank, world_size=self.world)
            self.pg = dist

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64)
        if self.pg.get_backend() == "nccl":
            t = t.cuda()
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def sum(self, x: float) -> float:
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64)
        if self.pg.get_backend() == "nccl":
            t = t.cuda()
        self.pg.all_reduce(t, op=self.pg.ReduceOp.SUM)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


def aggregate(units_per_rank_total: float, max_seconds: float) -> float:
    """whole-job throughput: units all ranks processed / slowest rank's time"""
    return units_per_rank_total / max_seconds if max_seconds > 0 else float("nan")


# ---------------------------------------------------------------------------
# peaks, clocks
# ---------------------------------------------------------------------------
def hbm_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def bf16_peak(sustained=False):
    """burst figure for a kernel timed alone; the sustained one (a seconds-long
    loop under the power cap) for work timed as a whole multi-kernel pass"""
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["bf16_tflops_sustained" if sustained else "bf16_tflops"]), "measured"
    except Exception:
        return (1700.0 if sustained else 1900.0), "fallback"


def prellm_measure(w, dev, reps=20):
    """The pre-LLM pass (Sec. 4.2-4.3) on the same workload: the whole
    provip_similarity_reduce call, and the nearest-centroid assignment alone
    (provip_merge without the mean), whose pruned x kept Gram is the pass's
    dominant contraction T_RT = 2 d (N_v - N1) N1."""
    import torch
    from paper_2608_25332_gb300 import provip as P
    from paper_2608_25332_gb300 import synth
    g = {k: v.to(dev) for k, v in synth.pre_llm_inputs(w).items()}
    ws = P.workspace(P.lib().provip_similarity_reduce_workspace_size(w.B, w.N_v, w.D, w.n_t[1], w.keep_pre), dev)
    full = lambda: P.provip_similarity_reduce(g["emb_v"], g["emb_t"], g["text_len"], w.keep_pre, ws=ws)
    first = full()
    idx = first["idx"]
    n_T = first["mask"].sum(dim=1).double().cpu()  # |T| per sample
    assign_only = lambda: P.provip_merge(g["emb_v"], idx, want_merged=False)

    def t_eager(f):
        for _ in range(3):
            f()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            f()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps * 1e3

    def t(f):
        # device time: reps calls in one CUDA graph, replayed once untimed, then timed
        for _ in range(3):
            f()
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=torch.cuda.Stream(device=dev)):
            for _ in range(reps):
                f()
        graph.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(3):
            graph.replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / (3 * reps) * 1e3

    us_full, us_assign = t(full), t(assign_only)
    us_eager = t_eager(full)
    flops = 2.0 * w.D * (w.N_v - w.keep_pre) * w.keep_pre * w.B
    peak, src = bf16_peak()
    ach = flops / us_assign / 1e6
    # the paper's cost of the pass's contractions (appendix on the computational
    # cost, T_4): 2 d (|T| N_v + (N_v - N1) N1) per sample, over the whole pass
    k1_flops = float((2.0 * w.D * (n_T * w.N_v + (w.N_v - w.keep_pre) * w.keep_pre)).sum())
    k1_peak, k1_src = bf16_peak(sustained=True)
    k1_ach = k1_flops / us_full / 1e6
    return {"workload": w.name, "us_per_call": us_full, "samples_per_s": w.B / us_full * 1e6,
            "timing": "CUDA graphs of the calls (device time); us_per_call_eager: the same calls "
                      "launched one by one from Python",
            "us_per_call_eager": us_eager,
            "k1": {"flops": k1_flops, "achieved": k1_ach, "peak": k1_peak, "peak_source": k1_src,
                   "unit": "TFLOP/s", "frac": k1_ach / k1_peak,
                   "note": "the whole pass (text Gram, relevance, top-k, gather, merge Gram, "
                           "assignment, means) against the sustained tensor peak"},
            "assign_us": us_assign, "assign_gram_flops": flops,
            "tensor_roofline": {"bound": "tensor", "kernel": "merge_argmax_pair_tc (bf16 merge Gram on "
                                "pairs of SMs; timed with its gather, norm and assignment kernels)",
                                "achieved": ach, "peak": peak,
                                "peak_source": src, "unit": "TFLOP/s", "frac": ach / peak}}


def schedule_measure(w, dev, reps=10):
    """The progressive schedule (Sec. 4.1) on the workload's batch: pre-LLM
    N_v -> keep_pre, shallow layer keep_pre -> keep with each sample's N_VIS
    visual heads, middle layer keep -> keep / 2 over every head; one CUDA graph
    per call, timed back to back (one input set larger than L2)."""
    import torch
    from paper_2608_25332_gb300 import synth
    from paper_2608_25332_gb300.schedule import ProgressiveSchedule
    cpu = synth.schedule_inputs(w)
    g = {k: {kk: (vv.to(dev) if isinstance(vv, torch.Tensor) else vv) for kk, vv in v.items()}
         for k, v in cpu.items()}
    n3 = w.keep // 2
    sched = ProgressiveSchedule(w.B, w.N_v, w.D, w.n_t[1], w.L_max, w.H_q, w.H_kv, w.D, w.P, w.keep_pre,
                                w.keep, n3, min(N_VIS, w.H_q), dtype=w.torch_dtype, device=dev)
    sh = g["shallow"]
    call = lambda: sched(g["pre"]["emb_v"], g["pre"]["emb_t"], g["pre"]["text_len"], sh, g["middle"],
                         sh["vis_start"])
    for _ in range(3):
        call()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.graph(graph, stream=stream):
        call()
    graph.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        graph.replay()
    b.record()
    torch.cuda.synchronize()
    us = a.elapsed_time(b) / reps * 1e3
    return {"workload": w.name, "stages": f"{w.N_v} -> {w.keep_pre} -> {w.keep} -> {n3} visual tokens",
            "n_vis": min(N_VIS, w.H_q), "us_per_call": us, "samples_per_s": w.B / us * 1e6,
            "host_syncs": 0}


def ablation_measure(dev, reps=20):
    """The ablation of Sec. 5 on LLaVA-1.5-7B (batch of 16, bf16): no pruning
    before the LLM, 576 visual tokens -> the paper's shallow / middle budgets,
    visual heads at the shallow layer (critical rows still found). One CUDA
    graph per call."""
    import torch
    from paper_2608_25332_gb300 import synth
    from paper_2608_25332_gb300.schedule import ProgressiveSchedule
    out = {}
    for n2, n3 in synth.ABLATION_BUDGETS:
        w = synth.ablation_workload(n2)
        cpu = synth.schedule_inputs(w)
        g = {k: {kk: (vv.to(dev) if isinstance(vv, torch.Tensor) else vv) for kk, vv in v.items()}
             for k, v in cpu.items()}
        sched = ProgressiveSchedule(w.B, w.N_v, w.D, w.n_t[1], w.L_max, w.H_q, w.H_kv, w.D, w.P, w.N_v, n2,
                                    n3, min(N_VIS, w.H_q), dtype=w.torch_dtype, device=dev, pre_llm=False)
        sh = g["shallow"]
        call = lambda: sched(g["pre"]["emb_v"], g["pre"]["emb_t"], g["pre"]["text_len"], sh, g["middle"],
                             sh["vis_start"])
        for _ in range(3):
            call()
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        stream = torch.cuda.Stream(device=dev)
        with torch.cuda.graph(graph, stream=stream):
            call()
        graph.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            graph.replay()
        b.record()
        torch.cuda.synchronize()
        us = a.elapsed_time(b) / reps * 1e3
        out[f"{w.N_v}->{n2}->{n3}"] = {"us_per_call": us, "samples_per_s": w.B / us * 1e6}
    return {"workload": "llava15_7b_bf16_b16 without pre-LLM pruning, visual heads at the shallow layer",
            "budgets": out}


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                   "-lms", "50"]
            if self.dev is not None:
                cmd += ["-i", str(self.dev)]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self):
        return time.time()

    def stop(self, t0, t1):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons, n = [], None, set(), 0
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ts, line in self.lines:
            if ts < t0 - 0.06 or ts > t1 + 0.06:
                continue
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            n += 1
            for nm, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": n}


def visible_device_index(local_rank):
    v = os.environ.get("CUDA_VISIBLE_DEVICES")
    if v:
        ids = [x.strip() for x in v.split(",") if x.strip()]
        if local_rank < len(ids):
            return ids[local_rank]
    return local_rank


# ---------------------------------------------------------------------------
# algorithmic bytes (what the method must move), per launch
# ---------------------------------------------------------------------------
def workload_config(w, algo="auto", copies=N_COPIES, input_mb=None):
    """the config object both arms print for the workload"""
    return {"workload": w.name, "B": w.B, "N_v": w.keep_pre, "keep": w.keep, "L_max": w.L_max,
            "H_q": w.H_q, "H_kv": w.H_kv, "H_sel": w.H_sel, "D": w.D, "algo": algo,
            "l2": f"inputs larger than L2: {copies} rotating device copies of "
                  f"{input_mb if input_mb is not None else 286:.0f} MB",
            "timing": f"CUDA graphs of {GRAPH_CHUNK} steps per stream, events on the launching stream",
            "overlap": "independent batches: each step's head scores may start under the previous "
                       "step's compaction (PROVIP_PRUNE_OVERLAP_PREVIOUS)"}


def algorithmic_bytes(w, inp, all_heads=False):
    """bytes the step must move: keys of the key/value heads the scored heads use
    and the scored heads' text queries (read once), scores and indices, and the
    compaction's reads + writes of the surviving rows"""
    import numpy as np
    es = 4 if w.dtype == "f32" else 2
    dh = 128
    seq = inp["seq_len"].cpu().numpy().astype(np.int64)
    tl = inp["text_len"].cpu().numpy().astype(np.int64)
    heads = np.arange(w.H_q) if all_heads else inp["head_list"].cpu().numpy()
    group = w.H_q // w.H_kv
    n_kv_used = len(set(int(h) // group for h in heads))
    out_rows = seq - w.keep_pre + w.keep
    row = (w.D + 2 * w.H_kv * dh) * es
    compact = int((2 * out_rows * row).sum() + (2 * out_rows * w.P * 4).sum() + w.B * w.keep * 4)
    scores = int((seq * n_kv_used * dh * es).sum() + (tl * len(heads) * dh * es).sum()
                 + w.B * w.keep_pre * 4 + w.B * w.keep * 4)
    return {"compact": compact, "head_topk": scores, "path": compact + scores}


def kernel_sha1(*names):
    h = hashlib.sha1()
    for n in names:
        with open(os.path.join(ROOT, "paper_2608_25332_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


# ---------------------------------------------------------------------------
# CPU baseline: the fp64 oracle as it stands
# ---------------------------------------------------------------------------
def oracle_inputs(cpu):
    import numpy as np
    return dict(Q=cpu["Q"].float().numpy().astype(np.float64),
                K=cpu["K"].float().numpy().astype(np.float64),
                heads=cpu["head_list"].numpy(), ts=cpu["text_start"].numpy(),
                tl=cpu["text_len"].numpy(), sl=cpu["seq_len"].numpy(),
                hidden=cpu["hidden"].view(__import__("torch").int16).numpy(),
                Kraw=cpu["K"].view(__import__("torch").int16).numpy(),
                Vraw=cpu["V"].view(__import__("torch").int16).numpy(),
                pos=cpu["pos"].numpy())


def oracle_step(o, w, samples, vis_start, N_v, keep, threads):
    import oracle
    sel = slice(samples[0], samples[1])
    return oracle.prune_batch(o["Q"][sel], o["K"][sel], o["heads"], o["ts"][sel], o["tl"][sel], o["sl"][sel],
                              vis_start, N_v, keep, o["hidden"][sel], o["Kraw"][sel], o["Vraw"][sel],
                              o["pos"][:, sel], threads=threads)


def cpu_baseline(cpu, w, vis_start, N_v, keep, budget_s=12.0):
    """The oracle on the workload's samples, all host cores, repeated until ~budget_s wall."""
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    o = oracle_inputs(cpu)
    B = w.B
    done, t0 = 0, time.perf_counter()
    reps = 0
    while True:
        oracle_step(o, w, (0, B), vis_start, N_v, keep, threads)
        done += B
        reps += 1
        el = time.perf_counter() - t0
        if el >= budget_s or reps >= 400:
            break
    used = min(threads, B)
    # the same on one host thread, for about a third of the budget
    done1, reps1, t1 = 0, 0, time.perf_counter()
    while True:
        oracle_step(o, w, (0, B), vis_start, N_v, keep, 1)
        done1 += B
        reps1 += 1
        el1 = time.perf_counter() - t1
        if el1 >= budget_s / 3 or reps1 >= 400:
            break
    return {"value": done / el, "unit": UNIT, "cores": used, "kind": "oracle",
            "sample": f"{reps} x the {B}-sample batch of {w.name} (fp64 oracle: scores, top-k, "
                      f"compaction), OpenMP over samples, {el:.1f} s wall",
            "single_thread": {"value": done1 / el1, "unit": UNIT, "cores": 1,
                              "sample": f"{reps1} x the same batch on one thread, {el1:.1f} s wall"}}


# ---------------------------------------------------------------------------
# the reference arm: the oracle, K steps of a bounded slice of the workload
# ---------------------------------------------------------------------------
def run_reference(args, dist):
    import numpy as np
    import torch
    import oracle
    from paper_2608_25332_gb300 import synth
    if dist.rank != 0:
        return 0
    oracle.build()
    w = synth.BY_NAME[args.workload]
    cpu = synth.in_llm_inputs(w)
    o = oracle_inputs(cpu)
    threads = os.cpu_count() or 1
    vis, nv, keep = cpu["vis_start"], cpu["N_v"], cpu["keep"]
    rows_per_sample = int(cpu["text_len"][0])
    heads = o["heads"]
    # Unit of work: one text row of one sample scored over every selected head
    # (the oracle's inner loop); the sample's top-k and compaction run with its
    # last row. Rows per step are sized so that W + K steps fit ~120 s.
    t0 = time.perf_counter()
    oracle.head_scores(o["Q"][0, :o["sl"][0]], o["K"][0, :o["sl"][0]], heads, [int(o["ts"][0])], vis, nv)
    t_row = max(time.perf_counter() - t0, 1e-5)
    budget = 120.0 / max(1, args.steps + args.warmup)
    rows_per_step = max(1, min(rows_per_sample * w.B, int(budget / t_row)))
    state = {"b": 0, "r": 0, "acc": np.zeros(nv)}

    def step():
        left = rows_per_step
        while left > 0:
            b, r = state["b"], state["r"]
            n = min(left, int(o["tl"][b]) - r)
            rows = np.arange(int(o["ts"][b]) + r, int(o["ts"][b]) + r + n)
            sl = int(o["sl"][b])
            state["acc"] += oracle.head_scores(o["Q"][b, :sl], o["K"][b, :sl], heads, rows, vis, nv) * n
            state["r"] += n
            left -= n
            if state["r"] == int(o["tl"][b]):
                v = state["acc"] / int(o["tl"][b])
                idx = oracle.topk(v, keep)
                src = oracle.compact_map(sl, vis, nv, idx)
                for key in ("hidden", "Kraw", "Vraw"):
                    oracle.gather_rows(o[key][b], src)
                state.update(b=(b + 1) % w.B, r=0, acc=np.zeros(nv))
        return rows_per_step

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    rows = sum(step() for _ in range(args.steps))
    el = time.perf_counter() - t0
    samples = rows / rows_per_sample
    value = samples / el
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * el / max(1, args.steps),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": workload_config(w),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{rows_per_step} text row(s) per step of {w.name} scored over "
                                       f"{w.H_sel} heads, each sample's top-k + compaction with its last "
                                       f"row; {samples:.2f} samples in {el:.1f} s"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ---------------------------------------------------------------------------
# the GB300 arm
# ---------------------------------------------------------------------------
class Lanes:
    """S streams of independent batches of one workload (S = 1: a single
    stream). Lane s has its own inputs (n_copies device copies rotating, so
    that the data come from HBM), outputs and workspace; step i runs on lane
    i % S with copy (i // S) % n_copies. Consecutive steps of a lane overlap:
    each step's head scores may start under that lane's previous compaction
    (PROVIP_PRUNE_OVERLAP_PREVIOUS); with S > 1 the calls also declare
    PROVIP_PRUNE_CONCURRENT."""

    def __init__(self, P, synth, w, dev, S, algo, n_copies, seed):
        import math
        import torch
        self.P, self.torch, self.dev, self.S = P, torch, dev, S
        flags = P.PRUNE_OVERLAP_PREVIOUS | (P.PRUNE_CONCURRENT if S > 1 else 0)
        self.lanes = []
        for s_ in range(S):
            cpu = synth.in_llm_inputs(w, seed=seed + 7 * s_)
            if s_ == 0:
                # at least n_copies per lane, and enough that all lanes' inputs span 3x the L2
                self.copy_bytes = sum(v.numel() * v.element_size() for v in cpu.values()
                                      if isinstance(v, torch.Tensor))
                n_copies = max(1, n_copies, math.ceil(3 * L2_BYTES / (S * self.copy_bytes)))
                self.n_copies = n_copies
            cs = [{k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
                  for _ in range(max(1, n_copies))]
            st = P.PruneStep(cs[0]["Q"], cs[0]["K"], cs[0]["V"], cs[0]["hidden"], cs[0]["pos"], cpu["head_list"],
                             w.n_t[1], cpu["N_v"], cpu["keep"], algo=algo, want_scores=False, flags=flags)
            self.lanes.append((cs, st))
            if s_ == 0:
                self.cpu0 = cpu
        self.vis = self.cpu0["vis_start"]
        self.streams = [torch.cuda.Stream(device=dev) for _ in range(S)] if S > 1 else None

    def step(self, i):
        cs, st = self.lanes[i % self.S]
        c = cs[(i // self.S) % len(cs)]
        st(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"], c["seq_len"], self.vis,
           stream=self.streams[i % self.S] if self.S > 1 else None)

    def run(self, n):
        """n consecutive steps; with S > 1, forked onto the lane streams and joined"""
        torch = self.torch
        if self.S == 1:
            for i in range(n):
                self.step(i)
            return
        main = torch.cuda.current_stream(self.dev)
        ev = torch.cuda.Event()
        ev.record(main)
        for ls in self.streams:
            ls.wait_event(ev)
        for i in range(n):
            self.step(i)
        for ls in self.streams:
            e2 = torch.cuda.Event()
            e2.record(ls)
            main.wait_event(e2)

    def graphs(self, K, stream):
        """CUDA graphs covering exactly K steps (each at most GRAPH_CHUNK steps
        per lane), each replayed once untimed (a freshly captured graph's first
        launch runs slower)"""
        torch = self.torch
        chunk = GRAPH_CHUNK * self.S
        sizes, left = [], K
        while left > 0:
            sizes.append(min(chunk, left))
            left -= sizes[-1]
        made = {}
        for n in sorted(set(sizes)):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                self.run(n)
            made[n] = g
        torch.cuda.synchronize()
        for g in made.values():
            g.replay()
        torch.cuda.synchronize()
        return [made[n] for n in sizes]


def timed_repeats(torch, graphs, dist, target_s, sampler=None):
    """Replays the K-step graphs R times back to back between CUDA events (one
    event per repeat), R sized so that the timed region lasts about target_s;
    barrier and device synchronisation on both sides. Returns the per-repeat
    seconds (max over ranks, repeat by repeat) and the clock record."""
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for g in graphs:
        g.replay()
    b.record()
    torch.cuda.synchronize()
    t1 = max(a.elapsed_time(b) / 1e3, 1e-6)
    R = int(dist.max(float(max(3, min(20000, math.ceil(target_s / t1))))))
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(R + 1)]
    if sampler is not None:
        sampler.start()
    dist.barrier()
    torch.cuda.synchronize()
    w0 = time.time()
    ev[0].record()
    for r in range(R):
        for g in graphs:
            g.replay()
        ev[r + 1].record()
    torch.cuda.synchronize()
    w1 = time.time()
    dist.barrier()
    clocks = sampler.stop(w0, w1) if sampler is not None else None
    times = [dist.max(ev[r].elapsed_time(ev[r + 1]) / 1e3) for r in range(R)]
    return times, clocks


def summarize(times, units, K, path_bytes, peak):
    """samples/s from the median repeat, with the spread of the repeats"""
    med = statistics.median(times)
    gbs = path_bytes * K / med / 1e9
    return {"value": units / med, "ms_per_step": 1e3 * med / K, "frac": gbs / peak, "achieved_gbs": gbs,
            "repeats": {"n": len(times), "min_value": units / max(times), "max_value": units / min(times),
                        "spread": (max(times) - min(times)) / med}}


def run_gb300(args, dist):
    import numpy as np
    import torch
    import __graft_entry__
    from paper_2608_25332_gb300 import provip as P
    from paper_2608_25332_gb300 import synth

    torch.cuda.set_device(dist.local_rank)
    dev = torch.device("cuda", dist.local_rank)
    __graft_entry__.build()
    w = synth.BY_NAME[args.workload]
    S = args.streams if args.streams is not None else (25 if w.B == 1 else 2)
    # concurrent streams: the streaming head-score form takes less SM time per
    # sample than the cluster form (at a higher latency), which leaves more of
    # the GPU to the other streams' compactions
    algo_name = "stream" if (args.algo == "auto" and S > 1 and w.dtype == "bf16") else args.algo
    algo_of = {"auto": P.ALGO_AUTO, "simt": P.ALGO_SIMT, "tcgen05": P.ALGO_TCGEN05,
               "stream": P.ALGO_TCGEN05_STREAM, "cluster": P.ALGO_TCGEN05_CLUSTER}
    algo = algo_of[algo_name]
    n_copies = max(1, args.copies)
    K = args.steps
    if S < 1 or K % S:
        raise SystemExit(f"--streams {S} must divide --steps")
    peak, peak_src = hbm_peak()
    stream = torch.cuda.Stream(device=dev)
    seed = w.seed + 1000 * dist.rank  # each rank prunes its own shard of samples

    # ---- the headline: S concurrent streams of independent batches ----
    lanes = Lanes(P, synth, w, dev, S, algo, n_copies, seed)
    cpu = lanes.cpu0
    vis, nv, keep = cpu["vis_start"], cpu["N_v"], cpu["keep"]
    input_mb = sum(v.numel() * v.element_size() for v in cpu.values() if isinstance(v, torch.Tensor)) / 1e6
    lanes.run(max(args.warmup, 1) * S)
    torch.cuda.synchronize()
    rc, bits = P.provip_device_status(clear=True)
    if rc != 0:
        raise RuntimeError(f"device status {rc} {bits} after warm-up")
    ab = algorithmic_bytes(w, cpu)
    graphs = lanes.graphs(K, stream)
    sampler = ClockSampler(visible_device_index(dist.local_rank)) if dist.rank == 0 else None
    times, clocks = timed_repeats(torch, graphs, dist, args.target_s, sampler)
    units = dist.sum(float(w.B * K))
    head = summarize(times, units, K, ab["path"], peak)
    max_sec = statistics.median(times)
    value = head["value"]
    rc, bits = P.provip_device_status(clear=True)
    if rc != 0:
        raise RuntimeError(f"device status {rc} {bits} after the timed region")
    del graphs
    if args.quick:
        if dist.rank == 0:
            print(json.dumps({"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": K,
                              "warmup": args.warmup, "ms_per_step": 1e3 * max_sec / K, "quick": True,
                              "config": workload_config(w, algo_name, lanes.n_copies, input_mb),
                              "repeats": head["repeats"]}))
        return 0

    # ---- the same workload on one stream: the configuration as stated ----
    single_algo = P.ALGO_AUTO if args.algo == "auto" else algo
    if S > 1:
        one = Lanes(P, synth, w, dev, 1, single_algo, n_copies, seed)
        one.run(3)
        g1 = one.graphs(K, stream)
        t1s, _ = timed_repeats(torch, g1, dist, args.target_s / 2)
        single = dict(summarize(t1s, units, K, ab["path"], peak), streams=1,
                      algo="auto" if single_algo == P.ALGO_AUTO else algo_name,
                      l2=f"inputs larger than L2: {one.n_copies} rotating device copies of "
                         f"{one.copy_bytes / 1e6:.0f} MB")
        del g1
    else:
        single = dict(head, streams=1, algo=algo_name)

    # per-kernel durations of the headline's launch configuration (graphs of
    # GRAPH_CHUNK launches): the compaction (dominant), head scores + top-k, the
    # step with no cross-step overlap
    g0 = lanes.lanes[0][0][0]
    step0 = lanes.lanes[0][1]
    copies = lanes.lanes[0][0]
    out = step0(g0["Q"], g0["K"], g0["V"], g0["hidden"], g0["pos"], g0["text_start"], g0["text_len"], g0["seq_len"],
                vis)
    idx = out["idx"].clone()
    outs = (step0.hidden_out, step0.K_out, step0.V_out, step0.pos_out)
    ws_ht = P.workspace(step0.ws.numel(), dev)
    heads_host = cpu["head_list"].tolist()

    def time_graph(fn, reps):
        for i in range(3):
            fn(i)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(GRAPH_CHUNK):
                fn(i)
        torch.cuda.synchronize()
        g.replay()  # untimed first launch
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(reps):
            g.replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b) / 1e3 / (reps * GRAPH_CHUNK)

    def compact_i(i):
        c = copies[i % len(copies)]
        P.provip_compact(idx, c["hidden"], c["K"], c["V"], c["pos"], c["seq_len"], vis, nv, out=outs)

    def head_topk_i(i):
        c = copies[i % len(copies)]
        P.provip_head_topk(c["Q"], c["K"], heads_host, c["text_start"], c["text_len"], c["seq_len"], vis, nv,
                           keep, algo=algo, N_t_max=w.n_t[1], ws=ws_ht, want_scores=False)

    step_serial = P.PruneStep(g0["Q"], g0["K"], g0["V"], g0["hidden"], g0["pos"], cpu["head_list"], w.n_t[1], nv,
                              keep, algo=algo, want_scores=False, flags=0, ws=step0.ws)

    def serial_i(i):
        c = copies[i % len(copies)]
        step_serial(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"], c["seq_len"], vis)

    launches_per_step = kernels_per_step(w, algo_name)
    reps = 20
    t_compact = time_graph(compact_i, reps)
    t_head = time_graph(head_topk_i, reps)
    t_serial = time_graph(serial_i, reps)
    ach = ab["compact"] / t_compact / 1e9
    traffic = None
    if COMPACT_TRAFFIC["bytes"] and COMPACT_TRAFFIC["sha1"] == kernel_sha1("compact.cu") and \
            args.workload == DEFAULT_WORKLOAD:
        traffic = COMPACT_TRAFFIC["bytes"]

    # ---- the next rows on the same batches ----
    ab_all = algorithmic_bytes(w, cpu, all_heads=True)
    next_rows = {}
    for name, make in (
            ("visual_heads", lambda c, fl: P.VisualHeadsPruneStep(
                c["Q"], c["K"], c["V"], c["hidden"], c["pos"], w.n_t[1], nv, keep, min(N_VIS, w.H_q), algo=algo,
                want_scores=False, want_conf=False, flags=fl)),
            ("all_heads", lambda c, fl: P.PruneStep(
                c["Q"], c["K"], c["V"], c["hidden"], c["pos"], None, w.n_t[1], nv, keep, algo=algo,
                want_scores=False, flags=fl))):
        obj = make(g0, P.PRUNE_OVERLAP_PREVIOUS)

        def fn(i, obj=obj):
            c = copies[i % len(copies)]
            obj(c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"], c["seq_len"], vis)

        t = time_graph(fn, reps)
        gbs = ab_all["path"] / t / 1e9
        next_rows[name] = {"us_per_step": t * 1e6, "samples_per_s": w.B / t, "frac": gbs / peak}
    next_rows["heads_scored"] = w.H_q
    next_rows["algorithmic_bytes"] = ab_all["path"]
    rc, bits = P.provip_device_status(clear=True)
    if rc != 0:
        raise RuntimeError(f"device status {rc} {bits} after the per-kernel legs")

    # ---- e2e through the C ABI with host buffers ----
    e2e = e2e_measure(P, torch, dist, w, cpu, step0, algo, dev, max(1, args.e2e_steps))
    head_copies = lanes.n_copies
    del lanes

    # ---- the video GQA workload (one sample per batch): as stated, and as
    # concurrent single-sample batches (an effective batch of S_v) ----
    workloads = {}
    if not args.no_workloads and w.name != VIDEO_WORKLOAD:
        workloads[VIDEO_WORKLOAD] = video_measure(P, synth, torch, dist, dev, stream, args, peak)

    prellm = prellm_measure(w, dev) if dist.rank == 0 else None
    schedule = schedule_measure(w, dev) if dist.rank == 0 else None
    ablation = ablation_measure(dev) if dist.rank == 0 else None
    cpu_base = None
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline:
        cpu_base = cpu_baseline(cpu, w, vis, nv, keep)

    if dist.rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": dist.world, "steps": K,
            "warmup": args.warmup, "ms_per_step": 1e3 * max_sec / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
            "config": dict(workload_config(w, algo_name, head_copies, input_mb), streams=S,
                           **({"concurrency": f"{S} streams of independent batches run concurrently (each with its "
                                              f"own inputs, outputs and workspace); value counts the samples of all "
                                              f"streams; single_stream is one stream"} if S > 1 else {})),
            "single_stream": single,
            "repeats": head["repeats"],
            "roofline": {"bound": "hbm", "kernel": "compact_kernel", "achieved": ach, "peak": peak,
                         "peak_source": peak_src, "unit": "GB/s", "frac": ach / peak, "traffic": traffic,
                         "algorithmic_bytes": ab["compact"], "duration_us": t_compact * 1e6},
            "path": {"algorithmic_bytes": ab["path"], "achieved_gbs": head["achieved_gbs"], "frac": head["frac"],
                     "head_topk_us": t_head * 1e6, "compact_us": t_compact * 1e6,
                     "step_us_without_overlap": t_serial * 1e6},
            "workloads": workloads,
            "e2e": e2e,
            "cpu_baseline": cpu_base,
            "gpu_launches": launches_per_step * K * head["repeats"]["n"],
            "prellm": prellm,
            "next_rows": dict(next_rows, schedule=schedule, ablation=ablation),
            "clocks": clocks,
        }
        print(json.dumps(line))
    return 0


VIDEO_WORKLOAD = "video_gqa_bf16_b1"


def video_measure(P, synth, torch, dist, dev, stream, args, peak):
    """The video GQA workload (B = 1): one stream with the library's automatic
    head-score form (the configuration as stated), then S_v concurrent streams
    of independent single-sample batches with the streaming form (an effective
    batch of S_v), each timed as repeats of 100-step graphs per stream; the
    compaction alone on one stream for the roofline."""
    w = synth.BY_NAME[VIDEO_WORKLOAD]
    seed = w.seed + 1000 * dist.rank
    n_copies = max(1, args.copies)
    out = {}
    for label, S, algo_name in (("single_stream", 1, "auto"), ("streams", 25, "stream")):
        lanes = Lanes(P, synth, w, dev, S, P.ALGO_AUTO if algo_name == "auto" else P.ALGO_TCGEN05_STREAM,
                      n_copies, seed)
        lanes.run(3 * S)
        K = GRAPH_CHUNK * S
        graphs = lanes.graphs(K, stream)
        times, _ = timed_repeats(torch, graphs, dist, args.target_s / 2)
        ab = algorithmic_bytes(w, lanes.cpu0)
        r = summarize(times, dist.sum(float(w.B * K)), K, ab["path"], peak)
        r.update(streams=S, algo=algo_name, us_per_sample=1e6 / r["value"] * dist.world,
                 l2=f"inputs larger than L2: {S} x {lanes.n_copies} rotating device copies of "
                    f"{lanes.copy_bytes / 1e6:.0f} MB")
        if S > 1:
            r["effective_batch"] = S
        out[label] = r
        if S == 1:
            cs, st = lanes.lanes[0]
            c0 = cs[0]
            res = st(c0["Q"], c0["K"], c0["V"], c0["hidden"], c0["pos"], c0["text_start"], c0["text_len"],
                     c0["seq_len"], lanes.vis)
            idx = res["idx"].clone()
            outs = (st.hidden_out, st.K_out, st.V_out, st.pos_out)

            def compact_i(i):
                c = cs[i % len(cs)]
                P.provip_compact(idx, c["hidden"], c["K"], c["V"], c["pos"], c["seq_len"], lanes.vis,
                                 lanes.cpu0["N_v"], out=outs)

            for i in range(3):
                compact_i(i)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i in range(GRAPH_CHUNK):
                    compact_i(i)
            g.replay()
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for _ in range(20):
                g.replay()
            b.record()
            torch.cuda.synchronize()
            tc = a.elapsed_time(b) / 1e3 / (20 * GRAPH_CHUNK)
            ach = ab["compact"] / tc / 1e9
            out["roofline"] = {"bound": "hbm", "kernel": "compact_kernel", "achieved": ach, "peak": peak,
                               "unit": "GB/s", "frac": ach / peak, "algorithmic_bytes": ab["compact"],
                               "duration_us": tc * 1e6}
            out["path_bytes"] = ab["path"]
        del lanes
        torch.cuda.synchronize()
    rc, bits = P.provip_device_status(clear=True)
    if rc != 0:
        raise RuntimeError(f"device status {rc} {bits} after the video legs")
    return out


def kernels_per_step(w, algo_name):
    """Kernels one pruning step launches: the one-pass tensor-core head scores
    (L_max <= 8192; the streaming or the cluster form), the top-k and the
    compaction; the two-pass and CUDA-core forms launch two head kernels."""
    if w.dtype != "bf16" or w.L_max > 8192 or algo_name not in ("auto", "tcgen05", "stream", "cluster"):
        return 4
    return 3


def e2e_measure(P, torch, dist, w, cpu, step0, algo, dev, E):
    """e2e through the C ABI with the batch in pinned host memory. Every step
    copies to the device what the tensor-core head scores read through tensor
    maps: each sample's text rows of Q and, with one 2-D copy per key/value head
    the selected query heads use, that head's key columns of every row; and the
    lengths. provip_head_topk selects on the device, then provip_compact reads
    the kept rows of hidden, K, V and the position ids where they are, in host
    memory (the library detects it: only the surviving rows cross the host
    link), and writes the compacted rows into device buffers, the input of the
    layers after the pruning; the kept indices and output lengths are copied
    back. The bytes declared are the copies plus the rows the compaction reads
    from host memory (in) and the indices and lengths (out). Two buffer sets
    alternate so that one step's copies overlap the other's kernels (a stream
    per copy direction and one for the kernels, ordered by events). Three timed
    runs of E steps, the median reported with the three beside it (the host link
    is shared with other jobs)."""
    import ctypes
    import numpy as np
    cudart = ctypes.CDLL("libcudart.so.13")
    memcpy2d = cudart.cudaMemcpy2DAsync
    memcpy2d.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_size_t,
                         ctypes.c_size_t, ctypes.c_int, ctypes.c_void_p]
    memcpy2d.restype = ctypes.c_int
    H2D = 1  # cudaMemcpyHostToDevice
    L = P.lib()
    nv, keep, vis = cpu["N_v"], cpu["keep"], cpu["vis_start"]
    B, Lm, Hq, dh = cpu["Q"].shape
    Hkv, D, Pn = cpu["K"].shape[2], cpu["hidden"].shape[2], cpu["pos"].shape[0]
    heads, hs = P._heads_arg(cpu["head_list"], Hq)
    kv_used = sorted({int(h) // (Hq // Hkv) for h in cpu["head_list"].tolist()})
    pin = {k: v.pin_memory() for k, v in cpu.items() if isinstance(v, torch.Tensor)}
    ts, tl = cpu["text_start"].numpy(), cpu["text_len"].numpy()
    seq = cpu["seq_len"].numpy().astype(np.int64)
    L_out = Lm - nv + keep
    es = pin["Q"].element_size()
    dt = P._dtype_code(pin["Q"])
    ws_bytes = L.provip_head_scores_workspace_size(B, Lm, hs, w.n_t[1], nv, algo, dt)
    sets = []
    for j in range(2):
        db = {k: torch.zeros_like(pin[k], device=dev) for k in ("Q", "K", "text_start", "text_len", "seq_len")}
        outs = {"idx": torch.empty((B, keep), dtype=torch.int32, device=dev),
                "hidden": torch.empty((B, L_out, D), dtype=pin["hidden"].dtype, device=dev),
                "K": torch.empty((B, L_out, Hkv, dh), dtype=pin["K"].dtype, device=dev),
                "V": torch.empty((B, L_out, Hkv, dh), dtype=pin["V"].dtype, device=dev),
                "pos": torch.empty((Pn, B, L_out), dtype=torch.int32, device=dev),
                "seq_len": torch.empty(B, dtype=torch.int32, device=dev)}
        ws = P.workspace(ws_bytes, dev)
        ho = {"idx": torch.empty((B, keep), dtype=torch.int32, pin_memory=True),
              "seq_len": torch.empty(B, dtype=torch.int32, pin_memory=True)}
        ev = {n: torch.cuda.Event() for n in ("h2d", "comp", "d2h")}
        sets.append((db, outs, ws, ho, ev))
    q_rows = int(tl.sum()) * Hq * dh * es
    k_cols = len(kv_used) * B * Lm * dh * es
    small = sum(pin[k].numel() * 4 for k in ("text_start", "text_len", "seq_len"))
    out_rows = seq - nv + keep
    row_in = (D + 2 * Hkv * dh) * es + Pn * 4  # hidden, K and V rows and position ids read in place
    h2d = q_rows + k_cols + small + int((out_rows * row_in).sum())
    d2h = sets[0][3]["idx"].numel() * 4 + sets[0][3]["seq_len"].numel() * 4
    s_comp, s_d2h, s_h2d = (torch.cuda.Stream(device=dev) for _ in range(3))
    fresh = [True, True]
    kp, kpitch, kw = pin["K"].data_ptr(), Hkv * dh * es, dh * es

    def one(n):
        j = n % 2
        db, outs, ws, ho, ev = sets[j]
        with torch.cuda.stream(s_h2d):
            if not fresh[j]:
                s_h2d.wait_event(ev["comp"])  # the set's device inputs were consumed by step n - 2
            for b in range(B):
                db["Q"][b, ts[b]:ts[b] + tl[b]].copy_(pin["Q"][b, ts[b]:ts[b] + tl[b]], non_blocking=True)
            for g in kv_used:
                rc = memcpy2d(db["K"].data_ptr() + g * kw, kpitch, kp + g * kw, kpitch, kw, B * Lm, H2D,
                              s_h2d.cuda_stream)
                if rc != 0:
                    raise RuntimeError(f"cudaMemcpy2DAsync returned {rc}")
            for k in ("text_start", "text_len", "seq_len"):
                db[k].copy_(pin[k], non_blocking=True)
            ev["h2d"].record(s_h2d)
        with torch.cuda.stream(s_comp):
            s_comp.wait_event(ev["h2d"])
            if not fresh[j]:
                s_comp.wait_event(ev["d2h"])  # step n - 2's indices have left this set
            st = ctypes.c_void_p(s_comp.cuda_stream)
            rc = L.provip_head_topk(P._ptr(db["Q"]), P._ptr(db["K"]), B, Lm, Hq, Hkv, dh, heads, hs,
                                    P._i32(db["text_start"]), P._i32(db["text_len"]), None, w.n_t[1], vis, nv,
                                    P._i32(db["seq_len"]), keep, dt, algo, P._ptr(outs["idx"]), None,
                                    P._ptr(ws), ws.numel(), st)
            P._check(rc, "provip_head_topk")
            rc = L.provip_compact(P._ptr(outs["idx"]), B, nv, keep, P._ptr_host_ok(pin["hidden"]), D,
                                  P._ptr_host_ok(pin["K"]), P._ptr_host_ok(pin["V"]), Hkv, dh,
                                  P._i32_host_ok(pin["pos"]), Pn, P._i32(db["seq_len"]), Lm, vis, dt,
                                  P._ptr(outs["hidden"]), P._ptr(outs["K"]), P._ptr(outs["V"]),
                                  P._i32(outs["pos"]), P._i32(outs["seq_len"]), st)
            P._check(rc, "provip_compact")
            ev["comp"].record(s_comp)
        with torch.cuda.stream(s_d2h):
            s_d2h.wait_event(ev["comp"])
            ho["idx"].copy_(outs["idx"], non_blocking=True)
            ho["seq_len"].copy_(outs["seq_len"], non_blocking=True)
            ev["d2h"].record(s_d2h)
        fresh[j] = False

    def run(first, n_steps):
        main = torch.cuda.current_stream(dev)
        start = torch.cuda.Event()
        start.record(main)
        for st_ in (s_h2d, s_comp, s_d2h):
            st_.wait_event(start)
        for n in range(first, first + n_steps):
            one(n)
        for st_ in (s_h2d, s_comp, s_d2h):
            done = torch.cuda.Event()
            done.record(st_)
            main.wait_event(done)

    run(0, 4)
    torch.cuda.synchronize()
    # the e2e path's kept indices and rows are those of the device-resident step
    ref = step0(*(lambda c: (c["Q"], c["K"], c["V"], c["hidden"], c["pos"], c["text_start"], c["text_len"],
                             c["seq_len"], vis))({k: (v.to(dev) if isinstance(v, torch.Tensor) else v)
                                                  for k, v in cpu.items()}))
    torch.cuda.synchronize()
    slo = ref["seq_len"].cpu()
    same = torch.equal(sets[1][3]["idx"], ref["idx"].cpu()) and torch.equal(sets[1][3]["seq_len"], slo)
    for k in ("hidden", "K", "V"):
        for b_ in range(B):
            same = same and torch.equal(sets[1][1][k][b_, :int(slo[b_])], ref[k][b_, :int(slo[b_])])
    if not same:
        raise RuntimeError("e2e path disagrees with the device-resident step")
    runs, first = [], 4
    for _ in range(3):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        dist.barrier()
        a.record()
        run(first, E)
        b.record()
        torch.cuda.synchronize()
        first += E
        runs.append(aggregate(dist.sum(float(w.B * E)), dist.max(a.elapsed_time(b) / 1e3)))
    return {"value": sorted(runs)[1], "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "runs": runs, "note": f"median of 3 timed runs of {E} steps; the batch stays in pinned host memory: "
                                  f"Q text rows and the used key heads copied in, kept rows read in place by the "
                                  f"compaction, compacted rows left on the device, kept indices and lengths read "
                                  f"back"}


def run_prellm_only(args):
    import torch
    import __graft_entry__
    from paper_2608_25332_gb300 import synth
    __graft_entry__.build()
    dev = torch.device("cuda", 0)
    print(json.dumps({"prellm": prellm_measure(synth.BY_NAME[args.workload], dev, reps=args.prellm_reps)}))
    return 0


def run_compact_only(args):
    """The compaction on its own: one pruning step gives idx, then --steps calls
    of provip_compact on rotating input copies (a CUDA graph of them, replayed
    after one untimed launch), timed with events."""
    import torch
    import __graft_entry__
    from paper_2608_25332_gb300 import provip as P
    from paper_2608_25332_gb300 import synth
    __graft_entry__.build()
    dev = torch.device("cuda", 0)
    w = synth.BY_NAME[args.workload]
    cpu = synth.in_llm_inputs(w)
    copy_bytes = sum(v.numel() * v.element_size() for v in cpu.values() if isinstance(v, torch.Tensor))
    n_copies = max(1, args.copies, -(-int(3 * L2_BYTES) // copy_bytes))  # rotating inputs span 3x the L2
    copies = [{k: (v.to(dev) if isinstance(v, torch.Tensor) else v) for k, v in cpu.items()}
              for _ in range(n_copies)]
    c0 = copies[0]
    vis, nv, keep = cpu["vis_start"], cpu["N_v"], cpu["keep"]
    st = P.PruneStep(c0["Q"], c0["K"], c0["V"], c0["hidden"], c0["pos"], cpu["head_list"], w.n_t[1], nv, keep,
                     want_scores=False)
    idx = st(c0["Q"], c0["K"], c0["V"], c0["hidden"], c0["pos"], c0["text_start"], c0["text_len"],
             c0["seq_len"], vis)["idx"].clone()
    outs = (st.hidden_out, st.K_out, st.V_out, st.pos_out)
    n = max(1, min(args.steps, 500))

    def call(i):
        c = copies[i % len(copies)]
        P.provip_compact(idx, c["hidden"], c["K"], c["V"], c["pos"], c["seq_len"], vis, nv, out=outs)

    for i in range(max(args.warmup, 1)):
        call(i)
    stream = torch.cuda.Stream(device=dev)
    stream.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n):
            call(i)
    g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    g.replay()
    b.record()
    torch.cuda.synchronize()
    rc, bits = P.provip_device_status(clear=True)
    if rc != 0 or bits != 0:
        raise RuntimeError(f"device status {rc} {bits}")
    us = a.elapsed_time(b) * 1e3 / n
    ab = algorithmic_bytes(w, cpu)["compact"]
    peak, src = hbm_peak()
    print(json.dumps({"compact_only": {"workload": w.name, "calls": n, "us_per_call": us, "copies": n_copies,
                                       "algorithmic_bytes": ab, "achieved_gbs": ab / us / 1e3,
                                       "frac": ab / us / 1e3 / peak, "peak_source": src}}))
    return 0


def main(argv=None):
    args = parse_args(argv)
    if args.prellm_only:
        return run_prellm_only(args)
    if args.compact_only:
        return run_compact_only(args)
    dist = Dist()
    if args.impl == "reference":
        dist.init("gloo")
        try:
            return run_reference(args, dist)
        finally:
            dist.close()
    import torch
    dist.init("nccl" if torch.cuda.is_available() else "gloo")
    try:
        return run_gb300(args, dist)
    finally:
        dist.close()


if __name__ == "__main__":
    sys.exit(main())
