#!/usr/bin/env python3
"""Benchmark of the per-step commit-set selection (Frechet profile decoding) on GB300.

One step = one full selection (vocab reduction + sort / scan / select / reveal) over one
batch of synthetic LLaDA-shaped logits (V = 126464).  Default workload: the large-batch
serving step, B = 64 rows of an active block of L = 32 positions, 50-100 % masked, bf16,
profile rule with f = 1 (delta = 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload NAME] [--no-graph]

Prints one JSON line (rank 0).  With N > 1 every rank runs its own batch on its own GPU
(weak scaling, no data exchange); the time is the max over ranks.  Started without
torchrun's environment, --gpus N > 1 launches the N ranks itself (torch.distributed.run on
127.0.0.1).  The main timed region covers at least --min-steps steps (1000).  The roofline
object times the vocabulary reduction by itself (fdllm_vocab_reduce) against the measured
copy bandwidth.  At N = 1 the line also carries, measured after the timed region:
`evolving` (the serving workload with masks evolving from step to step until every row has
finished), `per_config` (the single-block, mixed-mask, tie-group and full-sequence
workloads, each beside the oracle on a bounded sample, and the calibration-robust rule on
the serving workload), `lmhead` (the LM-head-fused step at B = 64, 32, 16 and 1) and `decode_loop`
(a 256-token generation of 8 sequences in blocks of 32 through the device-resident loop and
a host-driven one: NFE per block, tokens per step, tokens/s); --skip-evolving,
--skip-per-config, --skip-lmhead and --skip-decode-loop leave them out.
Other measurements, each one JSON line:
  --evolving      masks evolving from step to step until every row has finished
  --loop          the full-sequence workload (B = 16, L = 1024) selected until no mask remains
  --lmhead        the LM-head-fused step against cuBLAS logits + selection
                  (--lmhead-batch, --lmhead-vocab, --lmhead-variants)
  --decode-loop   the device-resident block loop against a host-driven loop

--impl reference times the fp64 CPU oracle (the reference arm of this benchmark) on the
host cores, each step a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import dataclasses
import datetime
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("decode-step selections/sec and logits HBM GB/s (fraction of GB300 peak) at "
          "V=126464")
UNIT = "selections/s"
FALLBACK_HBM_GBS = 6800.0
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "vocab_reduce_serving_b64_l32_bf16.md")
# the vocab reduction's sources: the kernel, the unit plan it shares with the interface and
# the inline-PTX copies and waits it is built from
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2606_02955_gb300", "csrc", f)
                  for f in ("vocab_reduce.cu", "fdllm_internal.cuh", "ptx.cuh")]


# ----------------------------------------------------------------------------- host logic
def aggregate(rows_per_rank: int, steps: int, times_s: list[float]) -> dict:
    """Whole-job throughput from per-rank timings: every rank decides rows_per_rank rows per
    step; the job takes as long as its slowest rank."""
    t = max(times_s)
    n = len(times_s)
    return {"value": rows_per_rank * steps * n / t, "seconds": t, "n_ranks": n}


def gather_times(dist, t_s: float, device) -> list[float]:
    """Every rank's timed seconds, in rank order (all_gather of one float64 per rank)."""
    import torch
    t = torch.tensor([t_s], dtype=torch.float64, device=device)
    out = [torch.zeros_like(t) for _ in range(dist.get_world_size())]
    dist.all_gather(out, t)
    return [float(x.item()) for x in out]


def rank_seed(base: int, rank: int) -> int:
    """Each rank draws its own batch (weak scaling: independent problems per GPU)."""
    return base + 7919 * rank


def peak_hbm_gbs():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            return float(json.load(fh)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def ncu_traffic(workload: str):
    """DRAM traffic per vocab-reduction launch from the committed ncu summary, only for the
    workload the summary was captured on and while the kernel's sources (hashed in order)
    are the ones the counters were taken on."""
    try:
        text = open(PROFILE_SUMMARY).read()
        h = hashlib.sha256()
        for f in KERNEL_SOURCES:
            h.update(open(f, "rb").read())
        sha = h.hexdigest()
    except OSError:
        return None
    m_sha = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    m_t = re.search(r"traffic_bytes_per_launch:\s*([0-9]+)", text)
    m_w = re.search(r"workload:\s*(\S+)", text)
    if not (m_sha and m_t and m_w) or m_sha.group(1) != sha or m_w.group(1) != workload:
        return None
    return int(m_t.group(1))


_REASON_BITS = {
    0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
    0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
    0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
    0x100: "display_clock_setting",
}


class ClockSampler:
    """SM clock and clock-event reasons sampled while work runs.  NVML is read through
    ctypes every `period_ms` milliseconds (read-only queries: nothing is set), so that even
    a timed region of some tens of milliseconds holds several samples; without NVML,
    nvidia-smi's own loop."""

    def __init__(self, gpu_index: int, period_ms: float = 4.0, pci_bus_id: str | None = None):
        self.gpu = gpu_index
        self.pci = pci_bus_id
        self.period = period_ms
        self.samples = []  # (t, sm_mhz, max_mhz, reasons_bitmask)
        self.source = None
        self.proc = None
        self.thread = None
        self._stop = threading.Event()

    def _nvml_handle(self):
        import ctypes
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
        except OSError:
            return None, None
        if lib.nvmlInit_v2() != 0:
            return None, None
        h = ctypes.c_void_p()
        ok = False
        if self.pci:
            ok = lib.nvmlDeviceGetHandleByPciBusId_v2(self.pci.encode(), ctypes.byref(h)) == 0
        if not ok:
            ok = lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(self.gpu), ctypes.byref(h)) == 0
        if not ok:
            lib.nvmlShutdown()
            return None, None
        return lib, h

    def start(self):
        lib, h = self._nvml_handle()
        if lib is not None:
            self.source = "nvml"
            self.thread = threading.Thread(target=self._poll_nvml, args=(lib, h), daemon=True)
            self.thread.start()
            return self
        cmd = ["nvidia-smi", "-i", str(self.gpu),
               "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active",
               "--format=csv,noheader,nounits", "-lms", str(max(20, int(self.period)))]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self.proc = None
            return self
        self.source = "nvidia-smi"
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        return self

    def _poll_nvml(self, lib, h):
        import ctypes
        sm, mx, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
        try:
            while not self._stop.is_set():
                if (lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(sm)) == 0
                        and lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0
                        and reasons_fn(h, ctypes.byref(rs)) == 0):
                    self.samples.append((time.time(), float(sm.value), float(mx.value),
                                         int(rs.value)))
                self._stop.wait(self.period / 1e3)
        finally:
            lib.nvmlShutdown()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 3:
                continue
            try:
                self.samples.append((time.time(), float(parts[0]), float(parts[1]),
                                     int(parts[2], 16)))
            except ValueError:
                continue

    def stop(self):
        self._stop.set()
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)

    def summary(self, t0: float, t1: float) -> dict:
        inside = [s for s in self.samples if t0 <= s[0] <= t1]
        used = inside if inside else self.samples
        if not used:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"],
                    "samples_in_timed_region": 0, "source": self.source}
        mask = 0
        for s in used:
            mask |= s[3]
        reasons = [name for bit, name in _REASON_BITS.items() if mask & bit and bit != 0x1]
        return {"sm_mhz": statistics.median(s[1] for s in used),
                "sm_max_mhz": max(s[2] for s in used), "reasons": reasons,
                "samples_in_timed_region": len(inside), "source": self.source,
                "period_ms": self.period}


def pci_bus_id(torch, dev) -> str | None:
    """The device's PCI address in NVML's form, so that the sampler watches the GPU this
    process runs on whatever CUDA_VISIBLE_DEVICES says."""
    p = torch.cuda.get_device_properties(dev)
    if not all(hasattr(p, k) for k in ("pci_domain_id", "pci_bus_id", "pci_device_id")):
        return None
    return "%08X:%02X:%02X.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)


# ----------------------------------------------------------------------------- ranks
def free_port() -> int:
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        return sk.getsockname()[1]


def launch_ranks(n: int, argv: list[str], script: str | None = None) -> int:
    """Run `script` (this file by default) as n ranks on this node through
    torch.distributed.run, rendezvous on 127.0.0.1; returns the launcher's exit code.  Each
    rank reads RANK / LOCAL_RANK / WORLD_SIZE from its environment."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
           "--nproc-per-node", str(n), "--master-addr", "127.0.0.1",
           "--master-port", str(free_port()), script or os.path.abspath(__file__), *argv]
    return subprocess.call(cmd)


def init_dist(world: int, device):
    """The process group of a multi-rank run (None for one rank): NCCL between GPUs, gloo for
    CPU ranks.  The only collectives are the timing gather and barriers."""
    if world <= 1:
        return None
    import torch.distributed as dist
    if getattr(device, "type", str(device)) == "cuda":
        dist.init_process_group("nccl", device_id=device)
    else:
        dist.init_process_group("gloo")
    return dist


# ----------------------------------------------------------------------------- our arm
def graph_runner(torch, stream, fn, per_replay: int, no_graph: bool = False):
    """A callable run(r) that issues `per_replay` consecutive calls fn(i) on `stream`: one
    CUDA graph replay (or eager launches with no_graph).  fn is called a few times first so
    that one-time set-up (kernel attributes, workspaces) stays out of the graph."""
    with torch.cuda.stream(stream):
        for i in range(max(3, per_replay)):
            fn(i)
    stream.synchronize()
    if no_graph:
        def run(r):
            with torch.cuda.stream(stream):
                for i in range(per_replay):
                    fn(r * per_replay + i)
        return run
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(per_replay):
            fn(i)

    def run(_r):
        g.replay()
    return run


def time_runner(torch, stream, run, n_rep: int, warm_rep: int, dist=None):
    """Seconds of n_rep runs on `stream` by CUDA events, after warm_rep untimed runs, with a
    synchronize (and a barrier across ranks) on both sides; also the wall-clock bounds."""
    for r in range(warm_rep):
        with torch.cuda.stream(stream):
            run(r)
    stream.synchronize()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    t_wall0 = time.time()
    e0.record(stream)
    with torch.cuda.stream(stream):
        for r in range(n_rep):
            run(r)
    e1.record(stream)
    e1.synchronize()
    t_wall1 = time.time()
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    return e0.elapsed_time(e1) / 1e3, t_wall0, t_wall1


class SelectionBench:
    """One workload's selection step over `n_buf` rotating logits buffers (each with its own
    copy of the initial mask, all restored by one copy per graph replay), so that a replay of
    n_buf steps reads more than the 129 MB L2 when n_buf * buffer size does."""

    def __init__(self, torch, fd, syn, w, seed: int, n_buf: int, dev, stream):
        self.torch, self.fd, self.w, self.dev, self.stream = torch, fd, w, dev, stream
        self.n_buf = max(1, n_buf)
        self.bufs = [syn.make_logits(w, seed=seed + i, device=dev) for i in range(self.n_buf)]
        self.mask0_np = syn.make_mask(w, seed=seed)
        self.mask0 = torch.from_numpy(self.mask0_np).to(dev)
        self.masked_rows = int(self.mask0_np.sum())
        self.alg_bytes = self.masked_rows * w.V * w.elem_bytes
        self.masks = self.mask0.unsqueeze(0).repeat(self.n_buf, 1, 1).contiguous()
        self.masks0 = self.masks.clone()
        self.tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device=dev)
        self.commit = torch.empty((w.B, w.L), dtype=torch.uint8, device=dev)
        self.n_out = torch.empty((w.B,), dtype=torch.int32, device=dev)

    @property
    def buffer_bytes(self) -> int:
        return self.bufs[0].numel() * self.bufs[0].element_size()

    def l2_policy(self) -> str:
        return ("inputs larger than L2: %d rotating logits buffers of %.1f MB (%.2f GB > "
                "129 MB L2)" % (self.n_buf, self.buffer_bytes / 1e6,
                                self.n_buf * self.buffer_bytes / 1e9))

    def step_fn(self, rule: str, param: float, eta: float = 0.0):
        fd, n_buf = self.fd, self.n_buf
        mode = fd.MODES["profile" if rule == "robust" else rule]

        def step(i):
            if i % n_buf == 0:  # steady state: the same masked rows every step
                self.masks.copy_(self.masks0, non_blocking=True)
            j = i % n_buf
            if rule == "robust":
                fd.fdllm_select_robust(self.bufs[j], self.masks[j], param, eta, None, self.tok,
                                       self.commit, self.n_out, stream=self.stream)
            else:
                fd.fdllm_select(self.bufs[j], self.masks[j], param, mode, self.tok,
                                self.commit, self.n_out, stream=self.stream)
        return step

    def time_steps(self, fn, steps: int, warmup: int, no_graph=False, dist=None):
        """(seconds, steps timed, wall bounds, runner) for at least `steps` calls of fn."""
        run = graph_runner(self.torch, self.stream, fn, self.n_buf, no_graph)
        replays = max(1, -(-steps // self.n_buf))
        warm = max(1, -(-warmup // self.n_buf))
        sec, t0, t1 = time_runner(self.torch, self.stream, run, replays, warm, dist)
        return sec, replays * self.n_buf, (t0, t1), run

    def step_distribution(self, run, replays: int) -> dict:
        """Per-step µs of `replays` graph replays timed one by one (median, min, max)."""
        import numpy as np
        torch, stream = self.torch, self.stream
        per = []
        for r in range(replays):
            a0 = torch.cuda.Event(enable_timing=True)
            a1 = torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            with torch.cuda.stream(stream):
                run(r)
            a1.record(stream)
            a1.synchronize()
            per.append(a0.elapsed_time(a1) * 1e3 / self.n_buf)
        return {"median": float(np.median(per)), "min": float(min(per)),
                "max": float(max(per)), "replays": len(per), "steps_per_replay": self.n_buf}


def run_ours(args, rank: int, world: int, local_rank: int) -> dict | None:
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = init_dist(world, dev)

    w = syn.WORKLOADS[args.workload]
    stream = torch.cuda.Stream(device=dev)
    sb = SelectionBench(torch, fd, syn, w, rank_seed(1234, rank), args.buffers, dev, stream)
    conf = torch.empty((w.B, w.L), dtype=torch.float32, device=dev)
    amax = torch.empty((w.B, w.L), dtype=torch.int32, device=dev)
    step = sb.step_fn(args.mode, args.param, args.eta)

    def k1_only(i):
        fd.fdllm_confidence(sb.bufs[i % sb.n_buf], sb.mask0, conf, amax, stream=stream)

    def k1_alone(i):  # the reduction kernel by itself
        fd.fdllm_vocab_reduce(sb.bufs[i % sb.n_buf], sb.mask0, stream=stream)

    # at least min_steps timed steps whatever --steps says (the serving workload is quoted
    # over 1000 steps), so that the region holds several clock samples and >= 100 replays
    want = max(args.steps, args.min_steps)
    sampler = None
    if rank == 0:
        sampler = ClockSampler(local_rank, pci_bus_id=pci_bus_id(torch, dev)).start()
    t_step, steps, (tw0, tw1), step_run = sb.time_steps(step, want, args.warmup, args.no_graph,
                                                        dist)
    t_k1, _, _, _ = sb.time_steps(k1_only, want, args.warmup, args.no_graph, dist)
    t_k1a, _, _, _ = sb.time_steps(k1_alone, want, args.warmup, args.no_graph, dist)
    # distribution of the step time: replays timed one by one (outside the timed region)
    dist_us = sb.step_distribution(step_run, 125)
    if sampler is not None:
        time.sleep(0.02)
        sampler.stop()

    times = gather_times(dist, t_step, dev) if dist is not None else [t_step]
    agg = aggregate(w.B, steps, times)
    ms_per_step = agg["seconds"] / steps * 1e3
    warm_steps = max(1, -(-args.warmup // sb.n_buf)) * sb.n_buf

    # end to end: the public call with pinned host buffers, copies inside the timed region
    e2e = None
    if not args.skip_e2e and rank == 0:  # the host link is the node's: rank 0 alone
        e2e = run_e2e(args, torch, fd, w, sb)

    result = None
    if rank == 0:
        peak, peak_kind = peak_hbm_gbs()
        k1_s = t_k1a / steps
        achieved = sb.alg_bytes / k1_s / 1e9
        traffic = ncu_traffic(w.name)
        clocks = sampler.summary(tw0, tw1) if sampler is not None else None
        result = {
            "metric": METRIC, "value": agg["value"], "unit": UNIT, "n_gpus": world,
            "steps": steps, "warmup": warm_steps,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
            "config": {
                "workload": w.name, "description": w.description, "B": w.B, "L": w.L,
                "V": w.V, "rule": args.mode, "param": args.param,
                "masked_rows_per_step": sb.masked_rows,
                "logits_bytes_per_step": sb.alg_bytes,
                "logits_gbs_per_step": sb.alg_bytes / (ms_per_step * 1e-3) / 1e9,
                "positions_per_s": sb.masked_rows * world / (ms_per_step * 1e-3),
                "steps_requested": args.steps,
                "step_us_distribution": dist_us,
                "l2_policy": sb.l2_policy(),
                "cuda_graph": not args.no_graph,
                "parallelism": "dp%d (independent batches, no collective)" % world,
            },
            "roofline": {
                "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic,
                "frac_of_nominal_7900_gbs": achieved / 7900.0,
                "kernel": "vocab_reduce (a1): CUDA-graph replays of fdllm_vocab_reduce, the "
                          "reduction kernel alone",
                "kernel_us": k1_s * 1e6, "peak_source": peak_kind,
                "kernel_us_with_finalize": t_k1 / steps * 1e6,
                "algorithmic_bytes_per_launch": sb.alg_bytes,
            },
            "clocks": clocks,
            "gpu_launches": 2 * steps,
            "e2e": e2e,
        }
    del sb
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return result


def run_e2e(args, torch, fd, w, sb) -> dict:
    """The public call with page-locked host buffers: the host copies of the step's inputs
    and results are inside the timed region (the masked rows are read by the GPU over the
    host link, the rest copied)."""
    h_logits = torch.empty(sb.bufs[0].shape, dtype=sb.bufs[0].dtype, pin_memory=True)
    h_logits.copy_(sb.bufs[0])
    h_mask = torch.from_numpy(sb.mask0_np.copy()).pin_memory()
    h_tok = torch.full((w.B, w.L), -1, dtype=torch.int32).pin_memory()
    h_commit = torch.empty((w.B, w.L), dtype=torch.uint8).pin_memory()
    h_n = torch.empty((w.B,), dtype=torch.int32).pin_memory()
    mode = fd.MODES["profile" if args.mode == "robust" else args.mode]
    for _ in range(2):
        h_mask.copy_(torch.from_numpy(sb.mask0_np))
        fd.fdllm_select(h_logits, h_mask, args.param, mode, h_tok, h_commit, h_n)
    e2e_steps = max(3, min(20, args.steps // 50))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        h_mask.copy_(torch.from_numpy(sb.mask0_np))
        fd.fdllm_select(h_logits, h_mask, args.param, mode, h_tok, h_commit, h_n)
    t_e2e = time.perf_counter() - t0
    out = {"value": w.B * e2e_steps / t_e2e, "unit": UNIT,
           # only the masked rows cross the host link (read by the GPU from pinned memory)
           "h2d_bytes_per_step": sb.masked_rows * w.V * w.elem_bytes
           + h_mask.numel() + h_tok.numel() * 4,
           "path": "fdllm_select_host (one C call): pinned host logits, the masked rows "
                   "read by the GPU over the host link, mask and tokens copied in, the step, "
                   "results and mask copied back",
           "d2h_bytes_per_step": h_tok.numel() * 4 + h_commit.numel() + h_n.numel() * 4
           + h_mask.numel(),
           "steps": e2e_steps}
    del h_logits
    return out


# Rules timed on each small config: the ones its recipe names.
CONFIG_RULES = {
    "single_block_b1_l32_bf16": [("profile", 1.0)],
    "mixed_mask_b8_l32_bf16": [("profile", 0.5), ("profile", 1.0), ("profile", 2.0),
                               ("factor", 0.5), ("factor", 1.0), ("factor", 2.0),
                               ("threshold", 0.9)],
    "tie_groups_b16_l64_fp32": [("profile", 1.0), ("factor", 1.0)],
}
CONFIG_BUFFERS = {"single_block_b1_l32_bf16": 32, "mixed_mask_b8_l32_bf16": 8,
                  "tie_groups_b16_l64_fp32": 4}


def run_per_config(args, torch, fd, syn, dev, peak_gbs: float) -> dict:
    """The other workloads of the metric at N = 1, each as CUDA-graph replays over rotating
    buffers larger than L2: per rule the time per step, selections/s (batch rows decided per
    second) and the algorithmic logits GB/s (masked rows x V x element size per step) with
    its fraction of the measured copy peak; the tie-group workload also reports whether the
    profile and factor rules took identical decisions (they must, Cor. factor-reduction);
    the full-sequence workload its step count and per-step latency for both rules; beside
    each, the CPU oracle on a bounded sample of the same recipe."""
    stream = torch.cuda.Stream(device=dev)
    out = {}
    for name, rules in CONFIG_RULES.items():
        w = syn.WORKLOADS[name]
        sb = SelectionBench(torch, fd, syn, w, 1234, CONFIG_BUFFERS[name], dev, stream)
        per_rule = {}
        decisions = {}
        for rule, param in rules:
            sec, steps, _, run = sb.time_steps(sb.step_fn(rule, param), args.config_steps, 32)
            us = sec / steps * 1e6
            per_rule["%s f=%g" % (rule, param) if rule != "threshold" else
                     "threshold tau=%g" % param] = {
                "us_per_step": us, "selections_per_s": w.B / (us * 1e-6),
                "logits_gbs": sb.alg_bytes / (us * 1e-6) / 1e9,
                "frac_of_measured_hbm": sb.alg_bytes / (us * 1e-6) / 1e9 / peak_gbs,
                "steps": steps,
                "step_us_distribution": sb.step_distribution(run, max(8, min(100, steps // sb.n_buf)))}
            m = sb.mask0.clone()
            with torch.cuda.stream(stream):
                fd.fdllm_select(sb.bufs[0], m, param, fd.MODES[rule], sb.tok, sb.commit,
                                sb.n_out, stream=stream)
            stream.synchronize()
            decisions[(rule, param)] = (sb.n_out.cpu().clone(), sb.commit.cpu().clone())
        entry = {"description": w.description, "B": w.B, "L": w.L, "V": w.V,
                 "dtype": w.dtype, "masked_rows_per_step": sb.masked_rows,
                 "logits_bytes_per_step": sb.alg_bytes, "l2_policy": sb.l2_policy(),
                 "rules": per_rule}
        if name == "tie_groups_b16_l64_fp32":
            (n_p, c_p), (n_f, c_f) = decisions[("profile", 1.0)], decisions[("factor", 1.0)]
            entry["identical_decisions_profile_factor"] = bool(torch.equal(n_p, n_f) and
                                                               torch.equal(c_p, c_f))
        if not args.skip_cpu_baseline:
            rule, param = rules[0]
            entry["cpu_baseline"] = oracle_bounded(name, rule, param, args.config_cpu_s,
                                                   rows=min(w.B, 2))
        out[name] = entry
        del sb
        torch.cuda.empty_cache()
    # the calibration-robust rule (App. C) on the serving workload, uniform allowance
    w = syn.WORKLOADS["serving_b64_l32_bf16"]
    sb = SelectionBench(torch, fd, syn, w, 1234, 8, dev, stream)
    timed_rules = {}
    for rule in ("profile", "robust"):
        sec, steps, _, _ = sb.time_steps(sb.step_fn(rule, 1.0, args.eta), 1000, 32)
        timed_rules[rule] = sec / steps * 1e6
    out["serving_b64_l32_bf16_robust"] = {
        "description": "the serving workload under the calibration-robust profile rule "
                       "(lower confidences max(0, c - eta), eta = %g) beside the plain rule, "
                       "same buffers, 1000 steps each" % args.eta,
        "robust_us_per_step": timed_rules["robust"],
        "profile_us_per_step": timed_rules["profile"],
        "robust_selections_per_s": w.B / (timed_rules["robust"] * 1e-6)}
    del sb
    torch.cuda.empty_cache()
    out["full_seq_b16_l1024_fp32"] = run_full_sequence(args, torch, fd, syn, dev, stream)
    if not args.skip_cpu_baseline:
        out["full_seq_b16_l1024_fp32"]["cpu_baseline"] = oracle_bounded(
            "full_seq_b16_l1024_fp32", "profile", 1.0, args.config_cpu_s, rows=1)
    return out


def run_full_sequence(args, torch, fd, syn, dev, stream,
                      name: str = "full_seq_b16_l1024_fp32", param: float = 1.0) -> dict:
    """A workload's selection + commit repeated until no mask remains (by default the
    full-sequence workload, B = 16, L = 1024, fp32), profile against factor at f = param,
    logits regenerated from (seed, step) before every step outside the timing; each step
    timed with events on its stream."""
    import numpy as np
    w = syn.WORKLOADS[name]
    res = {"description": w.description, "B": w.B, "L": w.L, "V": w.V, "dtype": w.dtype}
    logits = syn.make_logits(w, seed=4321, device=dev, step=0)
    for mode in (fd.PROFILE, fd.FACTOR):  # one untimed call per rule: one-time set-up
        m0 = torch.from_numpy(syn.make_mask(w, seed=4321)).to(dev)
        fd.fdllm_select(logits, m0, param, mode, stream=stream)
    stream.synchronize()
    del logits
    for rule in ("profile", "factor"):
        mask = torch.from_numpy(syn.make_mask(w, seed=4321)).to(dev)
        tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device=dev)
        commit = torch.empty((w.B, w.L), dtype=torch.uint8, device=dev)
        n = torch.empty((w.B,), dtype=torch.int32, device=dev)
        times, masked = [], []
        remaining = int(mask.sum().item())
        while remaining and len(times) < min(w.L + 1, args.full_seq_max_steps):
            logits = syn.make_logits(w, seed=4321, device=dev, step=len(times))
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fd.fdllm_select(logits, mask, param, fd.MODES[rule], tok, commit, n, stream=stream)
            e1.record(stream)
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
            masked.append(remaining)
            del logits
            remaining = int(mask.sum().item())
        t = np.array(times)
        res["%s f=%g" % (rule, param)] = {
            "steps": len(times), "finished": remaining == 0,
            "tokens_per_step": float((w.B * w.L - remaining) / max(len(times), 1)),
            "per_step_ms_median": float(np.median(t)), "per_step_ms_mean": float(t.mean()),
            "first_step_ms": float(t[0]),
            "first_step_logits_gbs": masked[0] * w.V * w.elem_bytes / (t[0] * 1e-3) / 1e9,
            "selections_per_s_median_step": w.B / (float(np.median(t)) * 1e-3)}
    return res


def oracle_bounded(name: str, rule: str, param: float, budget_s: float, rows: int,
                   step: int = 0) -> dict:
    """The CPU oracle on `rows` batch rows of a workload's recipe, on all host cores, for
    about budget_s seconds (at least one step)."""
    import fdllm_synth as syn
    import oracle
    w = syn.WORKLOADS[name]
    ws = dataclasses.replace(w, B=rows)
    host = syn.host_bits(syn.make_logits(ws, seed=1234, device="cpu", step=step))
    mask = syn.make_mask(ws, seed=1234)
    threads = os.cpu_count() or 1
    orc = oracle.default()
    mode = {"profile": oracle.PROFILE, "factor": oracle.FACTOR,
            "threshold": oracle.THRESHOLD}[rule]
    t0 = time.perf_counter()
    done = 0
    while done == 0 or time.perf_counter() - t0 < budget_s:
        orc.select(host, mask, mode, param, nthreads=threads)
        done += 1
    t = time.perf_counter() - t0
    return {"value": rows * done / t, "unit": UNIT, "cores": threads, "kind": "oracle",
            "ms_per_step_of_sample": t / done * 1e3,
            "sample": "%d batch row(s) of %s (%d masked positions of V=%d), %d steps"
                      % (rows, name, int(mask.sum()), w.V, done)}


def run_lmhead_key(args, torch) -> dict:
    """The LM-head-fused step at B = 64, 32, 16 and 1 for the default line: fused ms per step,
    the a1 path's PFLOP/s (2 R H V over the fdllm_lmhead_confidence time) against the
    measured bf16 burst peak (and the sustained one), and cuBLAS's GEMM on the same masked
    rows alone."""
    out = {}
    for b in (64, 32, 16, 1):
        a = argparse.Namespace(**vars(args))
        a.lmhead_batch, a.lmhead_vocab = b, 126464
        a.lmhead_variants = "fused,gemm,cublas_masked"
        a.lmhead_steps = 20
        r = run_lmhead(a)
        sustained = None
        try:
            with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
                sustained = float(json.load(fh)["bf16_tflops_sustained"])
        except (OSError, KeyError, ValueError):
            pass
        ach = r["roofline"]["achieved"]
        out["B=%d" % b] = {
            "masked_rows": r["masked_rows"], "fused_ms": r["ms_per_step"]["fused"],
            "a1_path_ms": r["ms_per_step"]["fused_confidence_only"],
            "a1_path_pflops": ach / 1e3 if ach else None,
            # timed alone after a rest (tens of ms of work): the burst figure is the peak;
            # the sustained one is beside it
            "frac_of_burst_bf16": r["roofline"]["frac"],
            "peak_source": r["roofline"]["peak_source"],
            "frac_of_sustained_bf16": ach / sustained if ach and sustained else None,
            "cublas_gemm_masked_rows_ms": r["ms_per_step"]["cublas_gemm_masked_rows_only"],
            "selections_per_s_fused": r["selections_per_s_fused"],
            "clocks": r["clocks"]}
        torch.cuda.empty_cache()
    return out


# ----------------------------------------------------------------------------- loop mode
def run_loop(args) -> dict:
    """--loop: a workload's selection + commit until no mask remains, profile against factor
    (f = args.param), as the default line's full-sequence figures (run_full_sequence)."""
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(device=dev)
    args.full_seq_max_steps = max(args.full_seq_max_steps, syn.WORKLOADS[args.workload].L + 1)
    res = run_full_sequence(args, torch, fd, syn, dev, stream, args.workload, args.param)
    return {"metric": "full-sequence loop: steps until no mask remains and per-step "
                      "selection latency", "workload": args.workload, "data": "synthetic",
            "param": args.param, "results": res}


def run_decode_loop(args) -> dict:
    """A whole generation (gen_len tokens per row in blocks of block_len) on the
    counter-based synthetic forward pass, two ways: the device-resident loop
    (fdllm_decode_loop: one call, one CUDA graph with a conditional WHILE node) and a
    host-driven loop (per step: forward launch, fdllm_select, reveal, and a host read of
    "any masked left").  Both take the same decisions, so the difference in wall time is the
    cost of the host round trips.  Wall time per generation, median of --repeats."""
    import time

    import numpy as np
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    B, gen, Lb, V = args.loop_batch, args.gen_len, args.block_len, syn.LLADA_VOCAB
    H = syn.LLADA_HIDDEN
    seed, peak = 2024, args.peak
    mode = fd.MODES[args.mode]
    lm = args.loop_lmhead
    stream = torch.cuda.current_stream()
    if lm:
        # the forward pass writes hidden states; the LM head (tcgen05) runs in the loop body
        _, w_vocab, _ = syn.make_lmhead_inputs(1, 1, H, V, seed=7, device=dev)
        logits = torch.empty((B, Lb, H), dtype=torch.bfloat16, device=dev)

        def forward(state, mask, out, strm):
            syn.synth_block_hidden_gpu(out, mask, B, Lb, H, V, w_vocab.data_ptr(), seed,
                                       step_ptr=state, beta_max=peak, stream_ptr=strm)

        def forward_step(step):
            syn.synth_block_hidden_gpu(logits.data_ptr(), mask.data_ptr(), B, Lb, H, V,
                                       w_vocab.data_ptr(), seed, step=step, beta_max=peak,
                                       stream_ptr=stream.cuda_stream)

        def select_step():
            fd.fdllm_lmhead_select(logits, w_vocab, mask, args.param, mode, tok, commit, n)

        def device_loop():
            return fd.fdllm_decode_loop_lmhead(forward, logits, w_vocab, gen, args.param, mode)
    else:
        logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device=dev)

        def forward(state, mask, out, strm):
            syn.synth_block_logits_gpu(out, mask, B, Lb, V, seed, step_ptr=state,
                                       peak_max=peak, stream_ptr=strm)

        def forward_step(step):
            syn.synth_block_logits_gpu(logits.data_ptr(), mask.data_ptr(), B, Lb, V, seed,
                                       step=step, peak_max=peak, stream_ptr=stream.cuda_stream)

        def select_step():
            fd.fdllm_select(logits, mask, args.param, mode, tok, commit, n)

        def device_loop():
            return fd.fdllm_decode_loop(forward, logits, gen, args.param, mode)

    seq_h = torch.empty((B, gen), dtype=torch.int32, device=dev)
    mask = torch.empty((B, Lb), dtype=torch.uint8, device=dev)
    tok = torch.empty((B, Lb), dtype=torch.int32, device=dev)
    commit = torch.empty((B, Lb), dtype=torch.uint8, device=dev)
    n = torch.empty((B,), dtype=torch.int32, device=dev)

    def host_loop():
        seq_h.fill_(-1)
        step, nfe = 0, []
        for blk in range(gen // Lb):
            mask.fill_(1)
            k = 0
            while bool(mask.any().item()):
                forward_step(step)
                select_step()
                view = seq_h[:, blk * Lb:(blk + 1) * Lb]
                view.copy_(torch.where(commit.bool(), tok, view))
                step += 1
                k += 1
            nfe.append(k)
        return seq_h, nfe, step

    def timed(fn):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        r = fn()
        torch.cuda.synchronize()
        return time.perf_counter() - t0, r

    for _ in range(max(1, args.warmup_loops)):
        timed(device_loop)
        timed(host_loop)
    dts, hts = [], []
    for _ in range(args.repeats):
        dt, (seq_d, nfe_d, steps_d) = timed(device_loop)
        ht, (seq_hh, nfe_hh, steps_hh) = timed(host_loop)
        dts.append(dt)
        hts.append(ht)
    dms, hms = 1e3 * float(np.median(dts)), 1e3 * float(np.median(hts))
    identical = bool(torch.equal(seq_d, seq_hh)) and list(nfe_d.cpu().numpy()) == nfe_hh
    tokens = B * gen
    return {
        "metric": "decode loop: generated tokens/s on a synthetic forward pass",
        "workload": "decode_loop%s_b%d_gen%d_block%d_bf16" % ("_lmhead_h%d" % H if lm else "",
                                                              B, gen, Lb),
        "B": B, "gen_len": gen, "block_len": Lb, "V": V, "dtype": "bf16",
        "forward": ("hidden states [B, 32, 4096] + the LM head fused with the selection"
                    if lm else "logits [B, 32, V]"),
        "mode": args.mode, "param": args.param, "peak": peak, "data": "synthetic",
        "steps": int(steps_d), "nfe_per_block": [int(x) for x in nfe_d.cpu().numpy()],
        "tokens_per_step": gen / max(int(steps_d), 1),
        "device_loop": {"ms_per_generation": dms, "tokens_per_s": tokens / (dms * 1e-3),
                        "ms_per_step": dms / max(steps_d, 1)},
        "host_loop": {"ms_per_generation": hms, "tokens_per_s": tokens / (hms * 1e-3),
                      "ms_per_step": hms / max(steps_hh, 1)},
        "host_round_trip_us_per_step": 1e3 * (hms - dms) / max(steps_d, 1),
        "identical_decisions": identical, "repeats": args.repeats,
    }


def run_lmhead(args) -> dict:
    """Step a1 fused into the LM head (fdllm_lmhead_select: a tcgen05 GEMM whose epilogue
    reduces the logits) against two unfused paths on the same inputs: our GEMM storing fp32
    logits then fdllm_select, and cuBLAS (torch.matmul, bf16 logits for all B*L rows) then
    fdllm_select.  LLaDA-8B head shape (H = 4096, V = 126464), the serving batch's masks.
    Each variant runs as CUDA-graph replays timed with events; the mask is restored from a
    saved copy before each step.  W (1.04 GB) exceeds L2, so every step reads it from HBM."""
    import numpy as np
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    wl = syn.WORKLOADS["serving_b64_l32_bf16"]
    if args.lmhead_batch != wl.B:
        wl = dataclasses.replace(wl, B=args.lmhead_batch)
    B, L, H, V = wl.B, wl.L, syn.LLADA_HIDDEN, args.lmhead_vocab
    variants = set(args.lmhead_variants.split(","))
    hidden, w, _ = syn.make_lmhead_inputs(B, L, H, V, seed=1234, device=dev)
    mask0_np = syn.make_mask(wl, seed=1234)
    R = int(mask0_np.sum())
    mask0 = torch.from_numpy(mask0_np).to(dev)
    mask = mask0.clone()
    mode = fd.MODES[args.mode]
    tok = torch.full((B, L), -1, dtype=torch.int32, device=dev)
    commit = torch.empty((B, L), dtype=torch.uint8, device=dev)
    n_out = torch.empty((B,), dtype=torch.int32, device=dev)
    logits32 = (torch.empty((B, L, V), dtype=torch.float32, device=dev)
                if "ours" in variants else None)
    rows_idx = torch.from_numpy(np.nonzero(mask0_np.reshape(-1))[0]).to(dev)
    stream = torch.cuda.Stream(device=dev)

    def fused():
        mask.copy_(mask0, non_blocking=True)
        fd.fdllm_lmhead_select(hidden, w, mask, args.param, mode, tok, commit, n_out,
                               stream=stream)

    def ours_unfused():
        mask.copy_(mask0, non_blocking=True)
        fd.fdllm_lmhead_logits(hidden, w, mask, logits32, stream=stream)
        fd.fdllm_select(logits32, mask, args.param, mode, tok, commit, n_out, stream=stream)

    def cublas_unfused():
        mask.copy_(mask0, non_blocking=True)
        x = torch.matmul(hidden.view(B * L, H), w.t()).view(B, L, V)
        fd.fdllm_select(x, mask, args.param, mode, tok, commit, n_out, stream=stream)

    def cublas_masked_gemm():
        # the same GEMM work as the fused path (masked rows only), logits in bf16, no selection
        torch.matmul(hidden.view(B * L, H).index_select(0, rows_idx), w.t())

    def gemm_only():
        fd.fdllm_lmhead_confidence(hidden, w, mask0, stream=stream)

    reps = max(3, args.lmhead_steps)

    def time_variant(fn):
        # each variant starts from a rested GPU: a ~1 ms, 1.4 kW step drives the board into
        # its power cap within tens of steps, which would penalise whichever runs later
        torch.cuda.synchronize()
        time.sleep(1.0)
        with torch.cuda.stream(stream):
            for _ in range(3):
                fn()
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        for _ in range(max(3, args.warmup // 4)):
            g.replay()
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        with torch.cuda.stream(stream):
            for _ in range(reps):
                g.replay()
        e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1) / reps

    sampler = ClockSampler(0).start()
    tw0 = time.time()
    t = {}
    for name, fn in (("fused", fused), ("fused_confidence_only", gemm_only),
                     ("ours_gemm_store_then_select", ours_unfused),
                     ("cublas_bf16_logits_then_select", cublas_unfused),
                     ("cublas_gemm_masked_rows_only", cublas_masked_gemm)):
        key = {"fused": "fused", "fused_confidence_only": "gemm",
               "ours_gemm_store_then_select": "ours",
               "cublas_bf16_logits_then_select": "cublas",
               "cublas_gemm_masked_rows_only": "cublas_masked"}[name]
        if key in variants:
            t[name] = time_variant(fn)
    tw1 = time.time()
    time.sleep(0.12)
    sampler.stop()

    # the fused path and the unfused ones take the same decisions on these inputs
    same = None
    if "ours" in variants:
        res = {}
        for name, fn in (("fused", fused), ("ours_unfused", ours_unfused)):
            with torch.cuda.stream(stream):
                fn()
            stream.synchronize()
            res[name] = (n_out.clone(), commit.clone())
        same = bool(torch.equal(res["fused"][0], res["ours_unfused"][0]) and
                    torch.equal(res["fused"][1], res["ours_unfused"][1]))

    flops = 2.0 * R * H * V
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    peak = float(peaks.get("bf16_tflops", 1900.0))
    t_gemm = t.get("fused_confidence_only", t.get("fused"))
    achieved = flops / (t_gemm * 1e-3) / 1e12 if t_gemm else None
    return {
        "metric": "LM head + commit-set selection: ms per step and GEMM TFLOP/s",
        "workload": "lmhead_b%d_l%d_h%d_v%d_bf16" % (B, L, H, V),
        "B": B, "L": L, "H": H, "V": V, "masked_rows": R, "mode": args.mode,
        "gemm_variant_env": {k: os.environ[k] for k in ("FDLLM_LMHEAD_GEMM", "FDLLM_LMHEAD_BN")
                             if k in os.environ},
        "param": args.param, "data": "synthetic",
        "ms_per_step": t,
        "selections_per_s_fused": B / (t["fused"] * 1e-3) if "fused" in t else None,
        "speedup_vs_cublas_unfused": (t["cublas_bf16_logits_then_select"] / t["fused"]
                                      if "fused" in t and "cublas_bf16_logits_then_select" in t
                                      else None),
        "cublas_masked_rows_tflops": (flops / (t["cublas_gemm_masked_rows_only"] * 1e-3) / 1e12
                                      if "cublas_gemm_masked_rows_only" in t else None),
        "identical_decisions_fused_vs_unfused": same,
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak if achieved else None,
                     "kernel": "fdllm_lmhead_confidence (compaction, "
                     "gather, GEMM with reducing epilogue, combine)",
                     "algorithmic_flops_per_launch": flops,
                     "peak_source": "measured" if "bf16_tflops" in peaks else "fallback"},
        "clocks": sampler.summary(tw0, tw1),
        "steps": reps,
    }


def run_evolving(args) -> dict:
    """The serving workload with evolving masks: each step commits on the mask the previous
    step left (no restore), on the same logits, until every row has finished (`period`
    steps), then the trajectory restarts from the initial mask.  Reports selections/s (batch
    rows decided per step, finished rows included) and the logits GB/s actually read, the
    masked rows of every step being counted once, after the timed region, on a replay of the
    same deterministic trajectory."""
    import numpy as np
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = syn.WORKLOADS[args.workload]
    logits = syn.make_logits(w, seed=1234, device=dev)
    mask0 = torch.from_numpy(syn.make_mask(w, seed=1234)).to(dev)
    mask = mask0.clone()
    mode = fd.MODES[args.mode if args.mode != "robust" else "profile"]
    tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device=dev)
    commit = torch.empty((w.B, w.L), dtype=torch.uint8, device=dev)
    n = torch.empty((w.B,), dtype=torch.int32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    # the trajectory's masked rows per step until every row has finished (outside any timing)
    masked = []
    with torch.cuda.stream(stream):
        mask.copy_(mask0)
        for _ in range(w.L):
            left = int(mask.sum().item())
            if left == 0:
                break
            masked.append(left)
            fd.fdllm_select(logits, mask, args.param, mode, tok, commit, n, stream=stream)
    stream.synchronize()
    assert int(mask.sum().item()) == 0, "a row did not finish within L steps"
    period = len(masked)

    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        mask.copy_(mask0)
        fd.fdllm_select(logits, mask, args.param, mode, tok, commit, n, stream=stream)
    stream.synchronize()
    with torch.cuda.graph(g, stream=stream):
        mask.copy_(mask0, non_blocking=True)
        for _ in range(period):
            fd.fdllm_select(logits, mask, args.param, mode, tok, commit, n, stream=stream)
    reps = max(3, args.steps // period)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(reps):
            g.replay()
    e1.record(stream)
    e1.synchronize()
    sec = e0.elapsed_time(e1) / 1e3
    steps = reps * period
    bytes_total = reps * sum(masked) * w.V * w.elem_bytes
    return {
        "metric": "evolving masks: selections/s and logits GB/s read",
        "workload": w.name, "B": w.B, "L": w.L, "V": w.V, "dtype": w.dtype,
        "mode": args.mode, "param": args.param, "data": "synthetic",
        "steps": steps, "period_steps": period,
        "selections_per_s": w.B * steps / sec, "us_per_step": sec / steps * 1e6,
        "logits_gbs": bytes_total / sec / 1e9,
        "masked_rows_per_step": masked,
        "note": "the same logits every step (the trajectory's later steps read few rows, "
                "which L2 may hold); the step time is bounded below by the fixed cost; "
                "restoring the mask is one 2 KB copy per trajectory",
    }


# ----------------------------------------------------------------------------- oracle arm
def oracle_sample_rows(args) -> int:
    return max(1, min(args.sample_rows, 64))


def run_oracle_timed(args, steps: int, warmup: int, budget_s: float | None):
    """The CPU oracle on a bounded sample of the workload: `sample_rows` batch rows drawn by
    the same seeded recipe, on all host cores.  Runs `steps` steps, or for `budget_s`
    seconds (at least one step) when a budget is given."""
    import dataclasses

    import fdllm_synth as syn
    import oracle

    w = syn.WORKLOADS[args.workload]
    rows = oracle_sample_rows(args)
    ws = dataclasses.replace(w, B=rows)
    host = syn.host_bits(syn.make_logits(ws, seed=1234, device="cpu"))
    mask = syn.make_mask(ws, seed=1234)
    threads = os.cpu_count() or 1
    orc = oracle.default()
    if args.mode == "robust":
        def one():
            orc.select_robust(host, mask, args.param, args.eta, None, nthreads=threads)
    else:
        mode = {"profile": oracle.PROFILE, "factor": oracle.FACTOR,
                "threshold": oracle.THRESHOLD}[args.mode]

        def one():
            orc.select(host, mask, mode, args.param, nthreads=threads)
    for _ in range(warmup):
        one()
    t0 = time.perf_counter()
    done = 0
    while True:
        one()
        done += 1
        elapsed = time.perf_counter() - t0
        if budget_s is not None and elapsed >= budget_s:
            break
        if budget_s is None and done >= steps:
            break
    t = time.perf_counter() - t0
    # the same oracle on one thread, one step
    t1 = time.perf_counter()
    if args.mode == "robust":
        orc.select_robust(host, mask, args.param, args.eta, None, nthreads=1)
    else:
        orc.select(host, mask, mode, args.param, nthreads=1)
    t_single = time.perf_counter() - t1
    cpu = "unknown"
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu model")):
                cpu = line.split(":", 1)[1].strip()
                break
    except OSError:
        pass
    if cpu == "unknown":
        try:
            out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
            for line in out.splitlines():
                if line.strip().lower().startswith(("model name", "vendor id")):
                    cpu = line.split(":", 1)[1].strip()
                    if line.strip().lower().startswith("model name"):
                        break
        except (OSError, subprocess.SubprocessError):
            pass
    return {
        "value": rows * done / t, "unit": UNIT, "cores": threads, "kind": "oracle",
        "sample": "%d batch rows of %s drawn by its recipe (%d masked positions of V=%d) "
                  "per step, %d steps, fp64 C oracle with OpenMP over positions"
                  % (rows, w.name, int(mask.sum()), w.V, done),
        "seconds": t, "steps": done, "cpu": cpu,
        "single_thread_value": rows / t_single,
    }


def run_reference(args, rank: int, world: int) -> dict | None:
    if rank != 0:
        return None
    base = run_oracle_timed(args, args.steps, args.warmup, None)
    import fdllm_synth as syn
    w = syn.WORKLOADS[args.workload]
    return {
        "impl": "reference", "metric": METRIC, "value": base["value"], "unit": UNIT,
        "n_gpus": world, "steps": base["steps"], "warmup": args.warmup,
        "ms_per_step": base["seconds"] / base["steps"] * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "L": w.L, "V": w.V, "rule": args.mode,
                   "param": args.param, "sample_rows": oracle_sample_rows(args)},
        "cpu_baseline": base,
        "e2e": {"value": base["value"], "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


# ----------------------------------------------------------------------------- main
def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--gpus", type=int, default=1,
                    help="ranks, one GPU each; without torchrun's environment, N > 1 starts "
                         "them through torch.distributed.run")
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--min-steps", type=int, default=1000,
                    help="the main timed region covers at least this many steps")
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="serving_b64_l32_bf16")
    ap.add_argument("--mode", choices=["profile", "factor", "threshold", "robust"],
                    default="profile")
    ap.add_argument("--eta", type=float, default=0.02,
                    help="calibration allowance of the robust rule (App. C)")
    ap.add_argument("--param", type=float, default=1.0)
    ap.add_argument("--buffers", type=int, default=16,
                    help="rotating logits buffers of the main workload (16: 8.3 GB); their "
                         "masks are restored by one copy per graph replay of as many steps")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--skip-cpu-baseline", action="store_true")
    ap.add_argument("--skip-evolving", action="store_true",
                    help="leave out the evolving-mask run that follows the timed region")
    ap.add_argument("--sample-rows", type=int, default=4,
                    help="batch rows per oracle step (reference arm / CPU baseline)")
    ap.add_argument("--cpu-budget-s", type=float, default=10.0)
    ap.add_argument("--loop", action="store_true",
                    help="run the selection until no mask remains (profile vs factor) and "
                         "report steps and per-step latency instead of the throughput line")
    ap.add_argument("--decode-loop", action="store_true",
                    help="time a whole generation through the device-resident decode loop "
                         "and through a host-driven loop, instead of the throughput line")
    ap.add_argument("--loop-batch", type=int, default=8)
    ap.add_argument("--gen-len", type=int, nargs="+", default=[256, 512, 1024])
    ap.add_argument("--block-len", type=int, default=32)
    ap.add_argument("--peak", type=float, default=20.0,
                    help="decode loop: largest planted logit height of the synthetic forward")
    ap.add_argument("--repeats", type=int, default=5)
    ap.add_argument("--loop-lmhead", action="store_true",
                    help="decode loop: the forward pass writes hidden states and the LM head "
                         "(H = 4096) runs fused with the selection inside the loop")
    ap.add_argument("--warmup-loops", type=int, default=2)
    ap.add_argument("--evolving", action="store_true",
                    help="the serving workload with masks evolving step to step (no restore)")
    ap.add_argument("--lmhead", action="store_true",
                    help="time the LM-head-fused selection against unfused paths, instead of "
                         "the throughput line")
    ap.add_argument("--lmhead-steps", type=int, default=50)
    ap.add_argument("--lmhead-batch", type=int, default=64)
    ap.add_argument("--lmhead-vocab", type=int, default=126464,
                    help="vocabulary size of the LM head (LLaDA-8B: 126464)")
    ap.add_argument("--lmhead-variants", default="fused,gemm,ours,cublas,cublas_masked",
                    help="comma list of: fused, gemm, ours, cublas, cublas_masked")
    ap.add_argument("--skip-per-config", action="store_true",
                    help="leave out the other workloads' figures (`per_config`)")
    ap.add_argument("--skip-lmhead", action="store_true",
                    help="leave out the LM-head-fused figures (`lmhead`)")
    ap.add_argument("--skip-decode-loop", action="store_true",
                    help="leave out the device-resident decode loop's figures (`decode_loop`)")
    ap.add_argument("--config-steps", type=int, default=512,
                    help="timed steps per rule of each small workload in `per_config`")
    ap.add_argument("--config-cpu-s", type=float, default=2.0,
                    help="seconds of oracle time per workload in `per_config`")
    ap.add_argument("--full-seq-max-steps", type=int, default=1025,
                    help="bound on the full-sequence loop's steps per rule in `per_config`")
    argv = sys.argv[1:] if argv is None else list(argv)
    args = ap.parse_args(argv)
    if args.evolving:
        print(json.dumps(run_evolving(args)), flush=True)
        return
    if args.lmhead:
        print(json.dumps(run_lmhead(args)), flush=True)
        return
    if args.decode_loop:
        lengths = list(args.gen_len)
        runs = []
        for g in lengths:
            args.gen_len = g
            runs.append(run_decode_loop(args))
        out = runs[0] if len(runs) == 1 else {
            "metric": runs[0]["metric"], "data": "synthetic",
            "workloads": runs}
        print(json.dumps(out), flush=True)
        return
    if args.loop:
        if args.workload == "serving_b64_l32_bf16":
            args.workload = "full_seq_b16_l1024_fp32"
        print(json.dumps(run_loop(args)), flush=True)
        return

    if "WORLD_SIZE" not in os.environ and args.gpus > 1:
        # one rank per GPU: start them here, each re-entering this file under torchrun
        sys.exit(launch_ranks(args.gpus, argv))
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world != args.gpus:
        ap.error("--gpus %d but the launcher started %d ranks" % (args.gpus, world))

    if args.impl == "reference":
        out = run_reference(args, rank, world)
    else:
        out = run_ours(args, rank, world, local_rank)
        if (out is not None and world == 1 and not args.skip_evolving
                and args.workload == "serving_b64_l32_bf16"):
            # the serving workload's second form: masks evolving from step to step until
            # every row has finished (after the timed region, not part of `value`)
            ev = run_evolving(args)
            out["evolving"] = {k: ev[k] for k in ("us_per_step", "selections_per_s",
                                                  "logits_gbs", "period_steps",
                                                  "masked_rows_per_step")}
        if (out is not None and world == 1 and not args.skip_per_config
                and args.workload == "serving_b64_l32_bf16"):
            import torch

            import fdllm_synth as syn
            import paper_2606_02955_gb300 as fd
            out["per_config"] = run_per_config(args, torch, fd, syn, torch.device("cuda", 0),
                                               peak_hbm_gbs()[0])
        if (out is not None and world == 1 and not args.skip_lmhead
                and args.workload == "serving_b64_l32_bf16"):
            import torch
            out["lmhead"] = run_lmhead_key(args, torch)
        if (out is not None and world == 1 and not args.skip_decode_loop
                and args.workload == "serving_b64_l32_bf16"):
            a = argparse.Namespace(**vars(args))
            a.gen_len, a.loop_lmhead, a.repeats, a.warmup_loops = 256, False, 3, 1
            a.mode, a.param = "profile", 1.0
            dl = run_decode_loop(a)
            out["decode_loop"] = {k: dl[k] for k in (
                "workload", "steps", "nfe_per_block", "tokens_per_step", "device_loop",
                "host_loop", "host_round_trip_us_per_step", "identical_decisions")}
        if out is not None and world == 1 and not args.skip_cpu_baseline:
            out["cpu_baseline"] = run_oracle_timed(args, 1, 1, args.cpu_budget_s)
    if out is not None:
        out["timestamp"] = datetime.datetime.now(datetime.timezone.utc).isoformat()
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
