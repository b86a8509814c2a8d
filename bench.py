#!/usr/bin/env python
"""Throughput of the TReVS two-stage prune on GB300, one JSON line on stdout.

A step is one trevs_prune_varlen call over the LLaVA-1.5-shaped batch of 32 requests
(576 visual tokens each, d' = 4096, query lengths 16..64, stage-1 keep 64 at textual
ratio 0.5, stage 2 at layer 2 with 32 heads x 128, top 8 heads, final keep 32): Eq. 4-5
scores, the Sec. 3.1 split and gather, then attention statistics, Eq. 8-9 and compaction.

  value      visual tokens scored and pruned per second, inputs resident in HBM, the step
             replayed as a CUDA graph, 4 rotating input sets (0.93 GB > 129 MB L2);
  e2e        the same metric through the public call with pinned HOST inputs: every step
             copies its inputs host->device and reads the kept indices back;
  roofline   the dominant kernel (stage-1 scoring + selection): algorithmic bytes per
             launch / its CUDA-event duration, against the measured HBM copy bandwidth;
  cpu_baseline  the fp64 oracle on the host cores (one process per core, bounded sample);
  configs    the other single-GPU workloads (LLaVA-NeXT 8 x 2,880, video 2 x 16,384 with
             GQA, the ragged serving batch of 64), each timed the same way, with its own
             algorithmic bytes, roofline fraction, scoring-grid time and clocks.

--impl reference times the oracle itself as the reference arm. Under torchrun (N > 1)
every rank prunes its own copy of the batch (replicas, weak scaling, no collective on
the data path); rank 0 prints the max-over-ranks time.
"""
from __future__ import annotations

import argparse
import json
import os
import pathlib
import statistics
import subprocess
import sys
import threading
import time

for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, "1")          # one BLAS thread per oracle worker process

ROOT = pathlib.Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

import numpy as np  # noqa: E402

from workloads import synth  # noqa: E402

METRIC = "visual tokens scored+pruned/s (2-stage prune)"
UNIT = "visual tokens/s"
WORKLOAD = dict(k1=64, ratio=0.5, k2=32)
ROTATING_SETS = 4
DOMINANT = "pre_score_kernel"
METHOD_RHO = 0.25   # K_r:K_d = 3:1, the paper's setting for the diversity draws (Sec. 3.1)
CLS_HEADS, CLS_DH = 16, 64   # the [CLS] attention of CLIP ViT-L/14 (Eq. 2-3)


def workload():
    return synth.llava15_batch32(**WORKLOAD)


def config_of(w):
    return {"workload": f"llava15_576_b32_k1_{WORKLOAD['k1']}_r{WORKLOAD['ratio']}_k2_{WORKLOAD['k2']}",
            "requests": w.B, "visual_tokens_per_request": 576, "d": w.d,
            "query_tokens": f"{min(r.m for r in w.reqs)}..{max(r.m for r in w.reqs)}",
            "K1": WORKLOAD["k1"], "textual_ratio": WORKLOAD["ratio"], "K2": WORKLOAD["k2"],
            "heads": f"{w.hq}x{w.dh}, keep {w.n_keep_heads}", "select": "ratio",
            "l2": f"{ROTATING_SETS} rotating input sets (> L2)", "replay": "CUDA graph per step"}


def algorithmic_bytes(w):
    """Stage 1: read Z, T, s_v; write Z_out and the kept indices. Stage 2: read Q, K; read
    and write the kept rows of hidden, K and V; write the kept indices."""
    sn = sum(r.n for r in w.reqs)
    sm = sum(r.m for r in w.reqs)
    sk1 = sum(r.k1 for r in w.reqs)
    sl = sum(r.l for r in w.reqs)
    sk2 = sum(r.k2 for r in w.reqs)
    score = sn * w.d * 2 + sm * w.d * 2 + sn * 4 + sk1 * 4
    stage1 = score + sk1 * w.d * 2
    stage2 = (sl * w.hq * w.dh * 2 + sk1 * w.hkv * w.dh * 2
              + 2 * sk2 * (w.d + 2 * w.hkv * w.dh) * 2 + sk2 * 4)
    # the diversity draws need the distances of every row to the pivots, which exist only once
    # all of Z is scored: a second read of Z (and of the K_r pivot rows), the largest cosine per row
    skr = sum(r.k1 - int(np.floor(np.float32(METHOD_RHO) * r.k1 + 0.5)) for r in w.reqs)
    pivot_pass = sn * w.d * 2 + skr * w.d * 2 + sn * 4
    return {"score_kernel": score, "stage1": stage1, "stage2": stage2, "step": stage1 + stage2,
            "pivot_pass": pivot_pass, "method_step": stage1 + stage2 + pivot_pass}


def peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def committed_traffic():
    """dram bytes per launch of the dominant kernel from the committed ncu summary, if the
    kernel source is unchanged since the capture (else None)."""
    import hashlib
    f = ROOT / "profiles" / "traffic.txt"
    src = ROOT / "paper_2609_37581_gb300" / "csrc" / "pre_llm.cu"
    if not f.exists() or not src.exists():
        return None
    digest = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    for line in f.read_text().splitlines():
        parts = dict(kv.split("=", 1) for kv in line.split() if "=" in kv)
        if parts.get("kernel") == DOMINANT and parts.get("src_sha") == digest and "dram_bytes_per_launch" in parts:
            return int(parts["dram_bytes_per_launch"])
    return None


# ------------------------------------------------------------------ oracle timing (host)


def _oracle_job(args):
    import oracle.trevs_oracle as O
    b_list, reps = args
    w = _ORACLE_W
    t0 = time.perf_counter()
    for _ in range(reps):
        O.run_workload(w, requests=b_list)
    return time.perf_counter() - t0


_ORACLE_W = None


def time_oracle(w, budget_s=12.0, cores=None):
    """Oracle throughput on the host cores (fork pool created before any CUDA call)."""
    import multiprocessing as mp
    global _ORACLE_W
    _ORACLE_W = w
    cores = cores or os.cpu_count() or 1
    ctx = mp.get_context("fork")
    tokens_per_req = [r.n for r in w.reqs]
    with ctx.Pool(cores) as pool:
        # calibration: one pass over all requests
        t0 = time.perf_counter()
        pool.map(_oracle_job, [([b], 1) for b in range(w.B)], chunksize=1)
        per_pass = time.perf_counter() - t0
        passes = min(1000, max(1, int(budget_s / max(1e-3, per_pass))))
        jobs = [([b], passes) for b in range(w.B)]
        t0 = time.perf_counter()
        pool.map(_oracle_job, jobs, chunksize=1)
        wall = time.perf_counter() - t0
    tokens = sum(tokens_per_req) * passes
    return {"value": tokens / wall, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{passes} pass(es) over all {w.B} requests, both stages, fp64, one process per core",
            "seconds": round(wall, 3)}


# ------------------------------------------------------------------ clocks


class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.lines = []
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", self.gpu_id], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, ValueError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.monotonic(), line.strip()))

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0=None, t1=None):
        """Median SM clock, max clock and active throttle reasons of the samples taken in
        [t0, t1] (time.monotonic() seconds; all samples by default)."""
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ts, ln in list(self.lines):
            if (t0 is not None and ts < t0) or (t1 is not None and ts > t1):
                continue
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 7:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for nm, v in zip(names, f[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ GPU arm


def max_over_ranks(x: float, device) -> float:
    """The largest of every rank's x (the slowest rank sets the job's time)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(max_elapsed_ms: float, steps: int, tokens_per_rank_step: int, world: int):
    """(ms per step, whole-job tokens/s) for `world` replicas that each prune their own batch,
    timed by the slowest rank."""
    ms = max_elapsed_ms / steps
    return ms, tokens_per_rank_step * world / (ms * 1e-3)


OTHER_CONFIGS = {   # the other single-GPU workloads (2,880-token, 16,384-token and ragged batches), each timed like the headline one
    "llava_next_2880_b8": synth.llava_next_batch8,
    "long_16384_b2_gqa": synth.long_video_batch2,
    "ragged_varlen_b64": synth.ragged_serving_batch64,
}


def time_workload(T, w, stream, sampler, steps, peak, src, method=False):
    """us per trevs_prune_varlen call on workload `w`: CUDA-event timing around graph replays
    over ROTATING_SETS input sets (each set > L2), the scoring grid timed alone with the
    library's event hook, the clocks sampled meanwhile; with `method`, also the paper's
    Method settings (fused score, K_r:K_d = 3:1 diversity draws) the same way."""
    import torch
    from workloads.device import build_batches, dev_bf16, dev_f32
    params = T.default_params(T.SELECT_RATIO)
    with torch.cuda.stream(stream):
        base = {"Z": dev_bf16(w.Z), "T": dev_bf16(w.T), "s_v": dev_f32(w.s_v), "Q": dev_bf16(w.Q),
                "K": dev_bf16(w.K), "V": dev_bf16(w.V), "hidden": dev_bf16(w.hidden)}
        sets = [base] + [{k: v.clone() for k, v in base.items()} for _ in range(ROTATING_SETS - 1)]
        batches = [build_batches(w, T.SELECT_RATIO, dev=x) for x in sets]
        ws = T.workspace(max(T.trevs_prune_varlen_workspace_size(p, i) for p, i in batches))
        calls = [T.PreparedCall(p, i, ws, params) for p, i in batches]
        for c in calls:
            c(stream)
        launches = T.last_launch_count()
        graphs = []
        for c in calls:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                c(stream)
            graphs.append(g)
        score_only = []
        for p, _ in batches:
            q = T.PreBatch(reqs=p.reqs, Z=p.Z, T=p.T, s_v=p.s_v, kept_idx=p.kept_idx, Z_out=None, s_t=p.s_t)
            score_only.append((q, T.workspace(T.trevs_pre_llm_varlen_workspace_size(q))))
    torch.cuda.synchronize()
    t0 = time.monotonic()
    with torch.cuda.stream(stream):
        for i in range(10):
            graphs[i % ROTATING_SETS].replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(steps):
            graphs[i % ROTATING_SETS].replay()
        b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / steps
        nk = 64
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nk)]
        for x, y in evs:
            x.record(stream); y.record(stream)
        torch.cuda.synchronize()
        torch.cuda._sleep(int(2e9 * 3e-4 * nk))
        for i in range(nk):
            q, wsq = score_only[i % ROTATING_SETS]
            T.trevs_pre_llm_varlen_timed(q, wsq, evs[i][0], evs[i][1], params, stream)
        torch.cuda.synchronize()
        kernel_ms = statistics.median(x.elapsed_time(y) for x, y in evs[8:])
        method_out = None
        if method:
            mparams = T.default_params(T.SELECT_FUSED, diversity=METHOD_RHO)
            mcalls = [T.PreparedCall(p, i, ws, mparams) for p, i in batches]
            for c in mcalls:
                c(stream)
            mlaunches = T.last_launch_count()
            mgraphs = []
            for c in mcalls:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    c(stream)
                mgraphs.append(g)
            for i in range(4):
                mgraphs[i % ROTATING_SETS].replay()
            msteps = max(20, steps // 4)
            a.record(stream)
            for i in range(msteps):
                mgraphs[i % ROTATING_SETS].replay()
            b.record(stream)
            torch.cuda.synchronize()
            mms = a.elapsed_time(b) / msteps
            mb = algorithmic_bytes(w)["method_step"]
            kr = sorted({r.k1 - int(np.floor(np.float32(METHOD_RHO) * r.k1 + 0.5)) for r in w.reqs})
            method_out = {"select": "fused (Eq. 6-7)", "diversity": METHOD_RHO, "K_r": kr,
                          "us_per_prune": round(mms * 1e3, 2), "value": w.visual_tokens() / (mms * 1e-3),
                          "unit": UNIT, "steps": msteps, "launches_per_step": mlaunches, "algorithmic_bytes": mb,
                          "frac": round(mb / (mms * 1e-3) / 1e9 / peak, 4), "peak_source": src}
            del mgraphs, mcalls
    t1 = time.monotonic()
    nbytes = algorithmic_bytes(w)
    del graphs, calls, score_only, sets, batches, ws
    torch.cuda.empty_cache()
    return {
        "workload": w.name, "requests": w.B, "visual_tokens": w.visual_tokens(), "d": w.d,
        "query_tokens": f"{min(r.m for r in w.reqs)}..{max(r.m for r in w.reqs)}",
        "K1": sorted({r.k1 for r in w.reqs}), "K2": sorted({r.k2 for r in w.reqs}),
        "heads": f"{w.hq}/{w.hkv}x{w.dh}, keep {w.n_keep_heads}",
        "us_per_prune": round(ms * 1e3, 2), "value": w.visual_tokens() / (ms * 1e-3), "unit": UNIT,
        "steps": steps, "launches_per_step": launches,
        "algorithmic_bytes": nbytes["step"],
        "achieved_gbs": round(nbytes["step"] / (ms * 1e-3) / 1e9, 1),
        "frac": round(nbytes["step"] / (ms * 1e-3) / 1e9 / peak, 4), "peak": peak, "peak_source": src,
        "score_kernel": {"kernel_us": round(kernel_ms * 1e3, 2), "algorithmic_bytes": nbytes["score_kernel"],
                         "frac": round(nbytes["score_kernel"] / (kernel_ms * 1e-3) / 1e9 / peak, 4)},
        "clocks": sampler.summary(t0, t1),
        "timed": f"CUDA events around {steps} graph replays of trevs_prune_varlen, {ROTATING_SETS} rotating "
                 "input sets (> L2)",
        **({"method_path": method_out} if method_out else {})}


def gpu_arm(args, rank, world, w, cpu_baseline):
    import torch
    from paper_2609_37581_gb300 import trevs as T
    from workloads.device import build_batches, dev_bf16, dev_f32

    dev = torch.device("cuda", int(os.environ.get("LOCAL_RANK", 0)))
    torch.cuda.set_device(dev)
    T.load()
    stream = torch.cuda.Stream()
    params = T.default_params(T.SELECT_RATIO)
    with torch.cuda.stream(stream):
        base = {"Z": dev_bf16(w.Z), "T": dev_bf16(w.T), "s_v": dev_f32(w.s_v), "Q": dev_bf16(w.Q),
                "K": dev_bf16(w.K), "V": dev_bf16(w.V), "hidden": dev_bf16(w.hidden)}
        sets = [base] + [{k: v.clone() for k, v in base.items()} for _ in range(ROTATING_SETS - 1)]
        batches = [build_batches(w, T.SELECT_RATIO, dev=s) for s in sets]
        ws = T.workspace(max(T.trevs_prune_varlen_workspace_size(p, i) for p, i in batches))
        calls = [T.PreparedCall(p, i, ws, params) for p, i in batches]
        # stage 1 without the gather, for the dominant kernel's timing hook
        score_only = []
        for p, _ in batches:
            q = T.PreBatch(reqs=p.reqs, Z=p.Z, T=p.T, s_v=p.s_v, kept_idx=p.kept_idx, Z_out=None, s_t=p.s_t)
            score_only.append((q, T.workspace(T.trevs_pre_llm_varlen_workspace_size(q))))
        for c in calls:                       # eager warm-up (sets the kernels' smem limits)
            c(stream)
        launches_per_step = T.last_launch_count()
        T.trevs_pre_llm_varlen(score_only[0][0], score_only[0][1], params, stream)
        torch.cuda.synchronize()
        graphs = []
        for c in calls:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                c(stream)
            graphs.append(g)
        # the paper's Method settings on the same batch: Eq. 6-7 fused score for the K_r pivots
        # and K_d = K1 / 4 diversity draws by farthest point sampling (Sec. 3.1)
        mparams = T.default_params(T.SELECT_FUSED, diversity=METHOD_RHO)
        mcalls = [T.PreparedCall(p, i, ws, mparams) for p, i in batches]
        for c in mcalls:
            c(stream)
        method_launches = T.last_launch_count()
        mgraphs = []
        for c in mcalls:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                c(stream)
            mgraphs.append(g)
    torch.cuda.synchronize()

    import torch.distributed as dist
    distributed = world > 1

    def barrier():
        if distributed:
            dist.barrier()

    gpu_id = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")[dev.index] \
        if os.environ.get("CUDA_VISIBLE_DEVICES") else str(dev.index)
    sampler = ClockSampler(gpu_id)
    with sampler, torch.cuda.stream(stream):
        for i in range(args.warmup):
            graphs[i % ROTATING_SETS].replay()
        torch.cuda.synchronize()
        barrier()
        torch.cuda.synchronize()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        tw0 = time.monotonic()
        ev0.record(stream)
        for i in range(args.steps):
            graphs[i % ROTATING_SETS].replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        timed_window = (tw0, time.monotonic())
        barrier()
        elapsed_ms = ev0.elapsed_time(ev1)
        # dominant kernel: the library records two CUDA events on the stream right around the
        # scoring grid's launch (trevs_pre_llm_varlen_timed). A spin kernel holds the device
        # while the host enqueues every call, so no interval waits on the host.
        nk = max(20, min(args.steps, 400))
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(nk)]
        for a, b in evs:                      # create the event handles
            a.record(stream); b.record(stream)
        torch.cuda.synchronize()
        torch.cuda._sleep(int(2e9 * 2e-4 * nk))   # about 0.2 ms per call at 2 GHz
        for i in range(nk):
            q, wsq = score_only[i % ROTATING_SETS]
            T.trevs_pre_llm_varlen_timed(q, wsq, evs[i][0], evs[i][1], params, stream)
        torch.cuda.synchronize()
        kernel_ms = statistics.median(a.elapsed_time(b) for a, b in evs[8:])
        # the Method settings, same protocol (graph replay over the rotating input sets)
        msteps = max(10, min(args.steps, 4000))
        for i in range(max(3, args.warmup // 10)):
            mgraphs[i % ROTATING_SETS].replay()
        torch.cuda.synchronize()
        m0, m1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        m0.record(stream)
        for i in range(msteps):
            mgraphs[i % ROTATING_SETS].replay()
        m1.record(stream)
        torch.cuda.synchronize()
        method_ms = m0.elapsed_time(m1) / msteps
        # [CLS] saliency (Eq. 2-3) for the same requests: CLIP ViT-L/14 keys, 16 heads of 64,
        # 4 rotating input sets (151 MB > L2); the calls are queued behind a spin kernel so
        # that none waits on the host
        cn = [r.n for r in w.reqs]
        csets = []
        for k in range(ROTATING_SETS):
            qb, kb = synth.cls_inputs(cn, CLS_HEADS, CLS_DH, seed=500 + k)
            csets.append((dev_bf16(qb), dev_bf16(kb)))
        cs_v = torch.zeros(sum(cn), dtype=torch.float32, device=dev)
        cws = T.workspace(T.trevs_cls_saliency_workspace_size(cn, CLS_HEADS))
        for k in range(8):
            T.trevs_cls_saliency_varlen(*csets[k % ROTATING_SETS], cn, cs_v, ws=cws, stream=stream)
        torch.cuda.synchronize()
        csteps = 200
        torch.cuda._sleep(int(2e9 * 3e-5 * csteps))   # about 30 us of host time per queued call
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        c0.record(stream)
        for k in range(csteps):
            T.trevs_cls_saliency_varlen(*csets[k % ROTATING_SETS], cn, cs_v, ws=cws, stream=stream)
        c1.record(stream)
        torch.cuda.synchronize()
        cls_ms = c0.elapsed_time(c1) / csteps
        cls_bytes = sum(x.numel() * x.element_size() for x in csets[0]) + cs_v.numel() * 4
        # streaming probe: the scoring grid's copies of the same Z (4 rotating sets) on as many
        # CTAs as the timed scoring grid, released on landing, computing nothing
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        pws = T.workspace(256)
        zs = [x["Z"] for x in sets]
        for k in range(3):
            T.trevs_stream_probe(zs[k % ROTATING_SETS], sms, pws, stream)
        torch.cuda.synchronize()
        psteps = 40
        torch.cuda._sleep(int(2e9 * 3e-5 * psteps))
        p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        p0.record(stream)
        for k in range(psteps):
            T.trevs_stream_probe(zs[k % ROTATING_SETS], sms, pws, stream)
        p1.record(stream)
        torch.cuda.synchronize()
        T.workspace_status(pws, stream)
        probe_ms = p0.elapsed_time(p1) / psteps
        probe_bytes = zs[0].numel() * zs[0].element_size()
        # the other workloads, one after the other
        peak, src = peaks()
        others = {}
        if not args.no_configs:
            del csets, cs_v, cws
            for name, make in OTHER_CONFIGS.items():
                others[name] = time_workload(T, make(), stream, sampler, max(50, min(args.steps, 2000)), peak, src,
                                             method=name == "long_16384_b2_gqa")

    if distributed:
        elapsed_ms = max_over_ranks(elapsed_ms, dev)

    # end to end through the public call with host buffers. Each step copies its inputs from
    # pinned host memory (split across four copy streams, so several copy engines share the
    # transfer) into one of two device input sets, runs the call on the other stream's set
    # order, and reads back both kept lists; a set is overwritten only after the call that
    # last read it has completed.
    e2e = None
    if rank == 0:
        host = {k: v.cpu().pin_memory() for k, v in base.items()}
        kept_h = [torch.empty(batches[s][0].kept_idx.numel(), dtype=torch.int32).pin_memory() for s in range(2)]
        kept2_h = [torch.empty(batches[s][1].kept_local.numel(), dtype=torch.int32).pin_memory() for s in range(2)]
        h2d = sum(v.numel() * v.element_size() for v in host.values())
        d2h = (kept_h[0].numel() + kept2_h[0].numel()) * 4
        ne = max(5, min(args.steps, 100))
        copy_streams = [torch.cuda.Stream() for _ in range(4)]
        free = [torch.cuda.Event() for _ in range(2)]

        def step(i):
            s = i % 2
            for cs in copy_streams:
                cs.wait_event(free[s])
            done = []
            for j, cs in enumerate(copy_streams):
                with torch.cuda.stream(cs):
                    for k, v in host.items():
                        rows = v.shape[0]
                        lo, hi = rows * j // 4, rows * (j + 1) // 4
                        if hi > lo:
                            sets[s][k][lo:hi].copy_(v[lo:hi], non_blocking=True)
                    ev = torch.cuda.Event()
                    ev.record(cs)
                    done.append(ev)
            for ev in done:
                stream.wait_event(ev)
            calls[s](stream)
            free[s].record(stream)
            kept_h[s].copy_(batches[s][0].kept_idx, non_blocking=True)
            kept2_h[s].copy_(batches[s][1].kept_local, non_blocking=True)

        with torch.cuda.stream(stream):
            for ev in free:
                ev.record(stream)
            for i in range(4):
                step(i)
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for i in range(ne):
                step(i)
            for cs in copy_streams:
                stream.wait_stream(cs)
            b.record(stream)
            torch.cuda.synchronize()
        e2e_ms = a.elapsed_time(b) / ne
        e2e = {"value": w.visual_tokens() / (e2e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms, 4)}

    if rank != 0:
        return None
    ms, value = replica_throughput(elapsed_ms, args.steps, w.visual_tokens(), world)
    method_kd = int(np.floor(np.float32(METHOD_RHO) * WORKLOAD["k1"] + 0.5))
    nbytes = algorithmic_bytes(w)
    achieved = nbytes["score_kernel"] / (kernel_ms * 1e-3) / 1e9
    clk = sampler.summary(*timed_window)
    return {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 5),
        "us_per_prune": round(ms * 1e3, 2), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic (seeded, LLaVA-1.5-shaped; no dataset)",
        "config": config_of(w),
        "roofline": {"bound": "hbm", "kernel": DOMINANT, "achieved": round(achieved, 1), "peak": peak,
                     "peak_source": src, "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "traffic": committed_traffic(), "algorithmic_bytes": nbytes["score_kernel"],
                     "kernel_us": round(kernel_ms * 1e3, 2),
                     "timed": "median over trevs_pre_llm_varlen_timed calls (queued behind a spin "
                              "kernel) of the CUDA events the library records on the launching stream "
                              "just before and just after pre_score_kernel (4 rotating input sets > L2)"},
        "step_roofline": {"algorithmic_bytes": nbytes["step"],
                          "achieved_gbs": round(nbytes["step"] / (ms * 1e-3) / 1e9, 1),
                          "frac": round(nbytes["step"] / (ms * 1e-3) / 1e9 / peak, 4), "peak_source": src},
        "cpu_baseline": cpu_baseline, "e2e": e2e,
        "gpu_launches": launches_per_step * args.steps,
        "launches_per_step": launches_per_step,
        "clocks": clk,
        "method_path": {
            "select": "fused (Eq. 6-7)", "diversity": METHOD_RHO, "K_r": WORKLOAD["k1"] - method_kd,
            "K_d": method_kd, "us_per_prune": round(method_ms * 1e3, 2),
            "value": w.visual_tokens() / (method_ms * 1e-3), "unit": UNIT, "steps": msteps,
            "launches_per_step": method_launches, "algorithmic_bytes": nbytes["method_step"],
            "frac": round(nbytes["method_step"] / (method_ms * 1e-3) / 1e9 / peak, 4), "peak_source": src,
            "timed": "CUDA events around graph replays of trevs_prune_varlen, 4 rotating input sets"},
        "cls_saliency": {
            "config": f"{w.B} x 576 patches, {CLS_HEADS} heads x {CLS_DH} (CLIP ViT-L/14 penultimate layer)",
            "us_per_call": round(cls_ms * 1e3, 2), "algorithmic_bytes": cls_bytes,
            "achieved_gbs": round(cls_bytes / (cls_ms * 1e-3) / 1e9, 1),
            "frac": round(cls_bytes / (cls_ms * 1e-3) / 1e9 / peak, 4), "peak_source": src,
            "timed": "CUDA events around 200 trevs_cls_saliency_varlen calls queued behind a spin kernel, "
                     "4 rotating input sets"},
        "stream_probe": {
            "ctas": sms, "us_per_pass": round(probe_ms * 1e3, 2), "bytes": probe_bytes,
            "achieved_gbs": round(probe_bytes / (probe_ms * 1e-3) / 1e9, 1),
            "frac": round(probe_bytes / (probe_ms * 1e-3) / 1e9 / peak, 4), "peak_source": src,
            "what": "Z streamed with the scoring grid's TMA boxes and 2 x 64 KB ring, stages released on "
                    "landing, no compute (trevs_stream_probe); the rate the grid's copy pattern allows",
            "timed": f"CUDA events around {psteps} passes queued behind a spin kernel, 4 rotating input sets"},
        "configs": others,
    }


# ------------------------------------------------------------------ reference arm (oracle)


def reference_arm(args, w):
    import multiprocessing as mp
    global _ORACLE_W
    _ORACLE_W = w
    cores = os.cpu_count() or 1
    ctx = mp.get_context("fork")
    with ctx.Pool(cores) as pool:
        t0 = time.perf_counter()
        pool.map(_oracle_job, [([b % w.B], 1) for b in range(cores)])
        per_round = time.perf_counter() - t0           # one request per core
        # each step: a bounded sample of requests so that warmup + steps fit in ~2 minutes
        total = args.steps + args.warmup
        rounds = max(1, int(120.0 / max(1e-3, per_round) / max(1, total)))
        sample = [b % w.B for b in range(min(w.B, cores * rounds))]
        jobs = [([b], 1) for b in sample]
        for _ in range(args.warmup):
            pool.map(_oracle_job, jobs, chunksize=1)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            pool.map(_oracle_job, jobs, chunksize=1)
        wall = time.perf_counter() - t0
    tokens = sum(w.reqs[b].n for b in sample) * args.steps
    value = tokens / wall
    ms = wall / args.steps * 1e3
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded, LLaVA-1.5-shaped; no dataset)", "config": config_of(w),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{len(sample)} of {w.B} requests per step, both stages, fp64, "
                                   f"one process per core"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def profile_run(w, stage="stage1", launches=5):
    """Stage 1 (scoring + selection; "method": with the fused score and the diversity draws),
    stage 2, or both stages ("both") of workload `w`, launched eagerly."""
    import torch
    from paper_2609_37581_gb300 import trevs as T
    from workloads.device import build_batches
    T.load()
    pre, inb = build_batches(w, T.SELECT_RATIO)
    if stage == "both":
        ws = T.workspace(T.trevs_prune_varlen_workspace_size(pre, inb))
        for _ in range(launches):
            T.trevs_prune_varlen(pre, inb, ws, T.default_params(T.SELECT_RATIO))
    elif stage in ("stage1", "method"):
        q = T.PreBatch(reqs=pre.reqs, Z=pre.Z, T=pre.T, s_v=pre.s_v, kept_idx=pre.kept_idx, s_t=pre.s_t)
        ws = T.workspace(T.trevs_pre_llm_varlen_workspace_size(q))
        params = (T.default_params(T.SELECT_RATIO) if stage == "stage1"
                  else T.default_params(T.SELECT_FUSED, diversity=METHOD_RHO))
        for _ in range(launches):
            T.trevs_pre_llm_varlen(q, ws, params)
    else:
        ws = T.workspace(T.trevs_in_llm_varlen_workspace_size(inb))
        for _ in range(launches):
            T.trevs_in_llm_varlen(inb, ws)
    torch.cuda.synchronize()
    print(json.dumps({"profile": stage, "launches": launches}))


def reserve_sweep(names, values, steps=1000, repeats=3):
    """us per trevs_prune_varlen call for each overlap reserve (SMs the scoring grid leaves to
    stage 2; -1 = the library's estimate), CUDA events around graph replays over
    ROTATING_SETS input sets; one JSON line per (workload, reserve)."""
    import torch
    from paper_2609_37581_gb300 import trevs as T
    from workloads.device import build_batches, dev_bf16, dev_f32
    lib = T.load()
    params = T.default_params(T.SELECT_RATIO)
    stream = torch.cuda.Stream()
    for name in names:
        w = workload() if name == "llava15_576_b32" else synth.WORKLOADS[name]()
        with torch.cuda.stream(stream):
            base = {"Z": dev_bf16(w.Z), "T": dev_bf16(w.T), "s_v": dev_f32(w.s_v), "Q": dev_bf16(w.Q),
                    "K": dev_bf16(w.K), "V": dev_bf16(w.V), "hidden": dev_bf16(w.hidden)}
            sets = [base] + [{k: v.clone() for k, v in base.items()} for _ in range(ROTATING_SETS - 1)]
            batches = [build_batches(w, T.SELECT_RATIO, dev=x) for x in sets]
            ws = T.workspace(max(T.trevs_prune_varlen_workspace_size(p, i) for p, i in batches))
        for r in values:
            lib.trevs_set_overlap_reserve(r)
            try:
                with torch.cuda.stream(stream):
                    calls = [T.PreparedCall(p, i, ws, params) for p, i in batches]
                    for c in calls:
                        c(stream)
                    graphs = []
                    for c in calls:
                        g = torch.cuda.CUDAGraph()
                        with torch.cuda.graph(g, stream=stream):
                            c(stream)
                        graphs.append(g)
                    us = []
                    for _ in range(repeats):
                        for i in range(20):
                            graphs[i % ROTATING_SETS].replay()
                        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                        a.record(stream)
                        for i in range(steps):
                            graphs[i % ROTATING_SETS].replay()
                        b.record(stream)
                        torch.cuda.synchronize()
                        us.append(round(a.elapsed_time(b) / steps * 1e3, 2))
            finally:
                lib.trevs_set_overlap_reserve(-1)
            print(json.dumps({"workload": w.name, "reserve": r, "us_per_prune": us}), flush=True)
            del graphs, calls
        del sets, batches, ws
        torch.cuda.empty_cache()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20000)
    ap.add_argument("--warmup", type=int, default=200)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the timing of the other configurations (2,880, 16,384 tokens, ragged batch)")
    ap.add_argument("--profile", nargs="?", const="stage1", choices=["stage1", "stage2", "method", "both"],
                    help="only run stage 1 (stage 2, stage 1 with the Method's diversity draws, or the "
                         "two-stage call) of a workload a few times, for an ncu capture")
    ap.add_argument("--workload", default="llava15_576_b32", choices=sorted(synth.WORKLOADS),
                    help="workload of --profile (default: the bench batch)")
    ap.add_argument("--launches", type=int, default=5, help="calls made by --profile")
    ap.add_argument("--reserve-sweep", metavar="R,R,...",
                    help="time the two-stage call of every configuration with each overlap reserve "
                         "(-1 = the library's estimate) instead of the bench line")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    if world != args.gpus and "RANK" in os.environ:
        print(f"warning: WORLD_SIZE={world} but --gpus {args.gpus}", file=sys.stderr)

    if args.impl == "reference":
        if rank != 0:
            return
        w = workload()
        print(json.dumps(reference_arm(args, w)), flush=True)
        return

    if args.reserve_sweep:
        reserve_sweep(["llava15_576_b32", *OTHER_CONFIGS], [int(x) for x in args.reserve_sweep.split(",")])
        return
    if args.profile:
        pw = workload() if args.workload == "llava15_576_b32" else synth.WORKLOADS[args.workload]()
        profile_run(pw, args.profile, args.launches)
        return
    w = workload()
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = time_oracle(w)                     # before any CUDA call: the pool forks safely
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", 0)))
        dist.init_process_group("nccl")
    out = gpu_arm(args, rank, world, w, cpu)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
