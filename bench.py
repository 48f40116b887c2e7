#!/usr/bin/env python3
"""Benchmark of the per-step commit-set selection (Frechet profile decoding) on GB300.

One step = one full selection (vocab reduction + sort / scan / select / reveal) over one
batch of synthetic LLaDA-shaped logits (V = 126464).  Default workload: the large-batch
serving step, B = 64 rows of an active block of L = 32 positions, 50-100 % masked, bf16,
profile rule with f = 1 (delta = 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload NAME] [--no-graph]

Prints one JSON line (rank 0).  Under torchrun (N > 1) every rank runs its own batch on its
own GPU (weak scaling, no data exchange); the time is the max over ranks.  The roofline
object times the vocabulary reduction by itself (fdllm_vocab_reduce) against the measured
copy bandwidth.  At N = 1 the line also carries `evolving`: the serving workload with masks
evolving from step to step until every row has finished, measured after the timed region
(--skip-evolving leaves it out).  Other measurements, each one JSON line:
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
# the vocab reduction's sources: the kernel and the unit plan it shares with the interface
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2606_02955_gb300", "csrc", f)
                  for f in ("vocab_reduce.cu", "fdllm_internal.cuh")]


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


def ncu_traffic():
    """DRAM traffic per vocab-reduction launch from the committed ncu summary, only while
    the kernel's sources (hashed in order) are the ones the counters were taken on."""
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
    if not (m_sha and m_t) or m_sha.group(1) != sha:
        return None
    return int(m_t.group(1))


_REASON_BITS = {
    0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
    0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
    0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
    0x100: "display_clock_setting",
}


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while work runs."""

    def __init__(self, gpu_index: int, period_ms: int = 50):
        self.gpu = gpu_index
        self.period = period_ms
        self.samples = []  # (t, sm_mhz, max_mhz, reasons_bitmask)
        self.proc = None
        self.thread = None

    def start(self):
        cmd = ["nvidia-smi", "-i", str(self.gpu),
               "--query-gpu=clocks.sm,clocks.max.sm,clocks_event_reasons.active",
               "--format=csv,noheader,nounits", "-lms", str(self.period)]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self.proc = None
            return self
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        return self

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
                    "samples_in_timed_region": 0}
        mask = 0
        for s in used:
            mask |= s[3]
        reasons = [name for bit, name in _REASON_BITS.items() if mask & bit and bit != 0x1]
        return {"sm_mhz": statistics.median(s[1] for s in used),
                "sm_max_mhz": max(s[2] for s in used), "reasons": reasons,
                "samples_in_timed_region": len(inside)}


# ----------------------------------------------------------------------------- our arm
def run_ours(args, rank: int, world: int, local_rank: int) -> dict | None:
    import numpy as np
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    w = syn.WORKLOADS[args.workload]
    seed = rank_seed(1234, rank)
    n_buf = max(1, args.buffers)
    bufs = [syn.make_logits(w, seed=seed + i, device=dev) for i in range(n_buf)]
    mask0_np = syn.make_mask(w, seed=seed)
    mask0 = torch.from_numpy(mask0_np).to(dev)
    masked_rows = int(mask0_np.sum())
    alg_bytes = masked_rows * w.V * w.elem_bytes
    mode = {"profile": fd.PROFILE, "factor": fd.FACTOR, "threshold": fd.THRESHOLD,
            "robust": fd.PROFILE}[args.mode]

    # one mask buffer per logits buffer, all restored by a single copy per replay
    masks = mask0.unsqueeze(0).repeat(n_buf, 1, 1).contiguous()
    masks0 = masks.clone()
    tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device=dev)
    commit = torch.empty((w.B, w.L), dtype=torch.uint8, device=dev)
    n_out = torch.empty((w.B,), dtype=torch.int32, device=dev)
    conf = torch.empty((w.B, w.L), dtype=torch.float32, device=dev)
    amax = torch.empty((w.B, w.L), dtype=torch.int32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step(i):
        if i % n_buf == 0:  # steady state: the same masked rows every step
            masks.copy_(masks0, non_blocking=True)
        if args.mode == "robust":
            fd.fdllm_select_robust(bufs[i % n_buf], masks[i % n_buf], args.param, args.eta,
                                   None, tok, commit, n_out, stream=stream)
        else:
            fd.fdllm_select(bufs[i % n_buf], masks[i % n_buf], args.param, mode, tok, commit,
                            n_out, stream=stream)

    def k1_only(i):
        fd.fdllm_confidence(bufs[i % n_buf], mask0, conf, amax, stream=stream)

    def k1_alone(i):  # the reduction kernel by itself
        fd.fdllm_vocab_reduce(bufs[i % n_buf], mask0, stream=stream)

    def make_runner(fn, per_replay):
        """A callable running `per_replay` consecutive steps (one CUDA graph replay)."""
        with torch.cuda.stream(stream):
            for i in range(max(3, per_replay)):  # warm: allocations, attributes
                fn(i)
        stream.synchronize()
        if args.no_graph:
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

    per_replay = n_buf
    replays = max(1, -(-args.steps // per_replay))
    steps = replays * per_replay
    warm_replays = max(1, -(-args.warmup // per_replay))

    def timed(run, n_rep):
        for r in range(warm_replays):
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

    sampler = ClockSampler(local_rank).start() if rank == 0 else None
    step_run = make_runner(step, per_replay)
    t_step, tw0, tw1 = timed(step_run, replays)
    k1_run = make_runner(k1_only, per_replay)
    t_k1, _, _ = timed(k1_run, replays)
    k1a_run = make_runner(k1_alone, per_replay)
    t_k1a, _, _ = timed(k1a_run, replays)
    # distribution of the step time: replays timed one by one (outside the timed region)
    per_step_us = []
    for r in range(min(200, replays)):
        a0 = torch.cuda.Event(enable_timing=True)
        a1 = torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        with torch.cuda.stream(stream):
            step_run(r)
        a1.record(stream)
        a1.synchronize()
        per_step_us.append(a0.elapsed_time(a1) * 1e3 / per_replay)
    if sampler is not None:
        time.sleep(0.12)
        sampler.stop()

    times = gather_times(dist, t_step, dev) if dist is not None else [t_step]
    agg = aggregate(w.B, steps, times)
    ms_per_step = agg["seconds"] / steps * 1e3

    # end to end: the public call with pinned host buffers, copies inside the timed region
    e2e = None
    if not args.skip_e2e:
        h_logits = torch.empty(bufs[0].shape, dtype=bufs[0].dtype, pin_memory=True)
        h_logits.copy_(bufs[0])
        h_mask = torch.from_numpy(mask0_np.copy()).pin_memory()
        h_tok = torch.full((w.B, w.L), -1, dtype=torch.int32).pin_memory()
        h_commit = torch.empty((w.B, w.L), dtype=torch.uint8).pin_memory()
        h_n = torch.empty((w.B,), dtype=torch.int32).pin_memory()
        for _ in range(2):
            h_mask.copy_(torch.from_numpy(mask0_np))
            fd.fdllm_select(h_logits, h_mask, args.param, mode, h_tok, h_commit, h_n)
        e2e_steps = max(3, min(20, args.steps // 50))
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            h_mask.copy_(torch.from_numpy(mask0_np))
            fd.fdllm_select(h_logits, h_mask, args.param, mode, h_tok, h_commit, h_n)
        t_e2e = time.perf_counter() - t0
        e2e = {"value": w.B * e2e_steps / t_e2e, "unit": UNIT,
               # only the masked rows cross the host link (read by the GPU from pinned memory)
               "h2d_bytes_per_step": masked_rows * w.V * w.elem_bytes
               + h_mask.numel() + h_tok.numel() * 4,
               "path": "pinned host logits; masked rows read over the host link by "
                       "fdllm_gather_masked_rows, then fdllm_select; results copied back",
               "d2h_bytes_per_step": h_tok.numel() * 4 + h_commit.numel() + h_n.numel() * 4
               + h_mask.numel(),
               "steps": e2e_steps}
        del h_logits

    result = None
    if rank == 0:
        peak, peak_kind = peak_hbm_gbs()
        k1_s = t_k1a / steps
        achieved = alg_bytes / k1_s / 1e9
        traffic = ncu_traffic()
        clocks = sampler.summary(tw0, tw1) if sampler is not None else None
        result = {
            "metric": METRIC, "value": agg["value"], "unit": UNIT, "n_gpus": world,
            "steps": steps, "warmup": warm_replays * per_replay,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
            "config": {
                "workload": w.name, "description": w.description, "B": w.B, "L": w.L,
                "V": w.V, "rule": args.mode, "param": args.param,
                "masked_rows_per_step": masked_rows,
                "logits_bytes_per_step": alg_bytes,
                "logits_gbs_per_step": alg_bytes / (ms_per_step * 1e-3) / 1e9,
                "positions_per_s": masked_rows * world / (ms_per_step * 1e-3),
                "step_us_distribution": {
                    "median": float(np.median(per_step_us)), "min": float(min(per_step_us)),
                    "max": float(max(per_step_us)), "replays": len(per_step_us),
                    "steps_per_replay": per_replay},
                "l2_policy": "inputs larger than L2: %d rotating logits buffers of %.0f MB "
                             "(%.2f GB > 129 MB L2)" % (n_buf, bufs[0].numel() *
                                                        bufs[0].element_size() / 1e6,
                                                        n_buf * bufs[0].numel() *
                                                        bufs[0].element_size() / 1e9),
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
                "algorithmic_bytes_per_launch": alg_bytes,
            },
            "clocks": clocks,
            "gpu_launches": 2 * steps,
            "e2e": e2e,
        }
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return result


# ----------------------------------------------------------------------------- loop mode
def run_loop(args) -> dict:
    """Selection + commit repeated until no mask remains, for the profile and the factor
    rule (f = args.param): steps taken and per-step selection latency.  Logits are
    regenerated from (seed, step) before each step, outside the timed region; each step's
    selection is timed with CUDA events on its stream."""
    import numpy as np
    import torch

    import fdllm_synth as syn
    import paper_2606_02955_gb300 as fd

    w = syn.WORKLOADS[args.workload]
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.Stream(device=dev)
    out = {}
    # One untimed call per rule first, so that the library's one-time set-up (kernel
    # attributes, occupancy queries, its workspace) stays out of the first timed step.
    logits = syn.make_logits(w, seed=4321, device=dev, step=0)
    for mode in (fd.PROFILE, fd.FACTOR):
        m0 = torch.from_numpy(syn.make_mask(w, seed=4321)).to(dev)
        fd.fdllm_select(logits, m0, args.param, mode, stream=stream)
    torch.cuda.synchronize()
    del logits
    for mode_name, mode in (("profile", fd.PROFILE), ("factor", fd.FACTOR)):
        mask = torch.from_numpy(syn.make_mask(w, seed=4321)).to(dev)
        tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device=dev)
        commit = torch.empty((w.B, w.L), dtype=torch.uint8, device=dev)
        n = torch.empty((w.B,), dtype=torch.int32, device=dev)
        times, masked, step = [], [], 0
        while True:
            remaining = int(mask.sum().item())
            if remaining == 0 or step >= w.L + 1:
                break
            logits = syn.make_logits(w, seed=4321, device=dev, step=step)
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fd.fdllm_select(logits, mask, args.param, mode, tok, commit, n, stream=stream)
            e1.record(stream)
            e1.synchronize()
            times.append(e0.elapsed_time(e1))
            masked.append(remaining)
            del logits
            step += 1
        t = np.array(times)
        first_bytes = masked[0] * w.V * w.elem_bytes
        out[mode_name] = {
            "steps": step, "finished": remaining == 0,
            "per_step_ms_median": float(np.median(t)), "per_step_ms_mean": float(t.mean()),
            "first_step_ms": float(t[0]), "total_selection_ms": float(t.sum()),
            "first_step_logits_gbs": first_bytes / (t[0] * 1e-3) / 1e9,
            "tokens_per_step": float(w.B * w.L / max(step, 1)),
        }
    return {"metric": "full-sequence loop: steps until no mask remains and per-step "
                      "selection latency", "workload": w.name, "B": w.B, "L": w.L, "V": w.V,
            "dtype": w.dtype, "param": args.param, "data": "synthetic", "results": out}


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
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="serving_b64_l32_bf16")
    ap.add_argument("--mode", choices=["profile", "factor", "threshold", "robust"],
                    default="profile")
    ap.add_argument("--eta", type=float, default=0.02,
                    help="calibration allowance of the robust rule (App. C)")
    ap.add_argument("--param", type=float, default=1.0)
    ap.add_argument("--buffers", type=int, default=8)
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

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

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
        if out is not None and world == 1 and not args.skip_cpu_baseline:
            out["cpu_baseline"] = run_oracle_timed(args, 1, 1, args.cpu_budget_s)
    if out is not None:
        out["timestamp"] = datetime.datetime.now(datetime.timezone.utc).isoformat()
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
