"""Seeded synthetic inputs for the commit-set selection step.

Both the CUDA path and the CPU oracle consume what this module produces; it holds none
of the selection method's arithmetic (no softmax, no sort, no rule).  It only draws
random numbers, rounds fp32 to bf16 (round to nearest even, done by torch) and states
the recipe of each workload.

The paper's workloads are the logits of LLaDA-8B-Instruct on benchmark prompts (PrefixCache,
block size 32, generation lengths 256-1024).  Those models and datasets are not available,
so these seeded logits stand in for them: vocabulary V = 126464 (LLaDA), i.i.d. Gaussian
noise plus one planted peak per position, and masks shaped like an active decode block.

"Plus a planted peak of height h" means h is ADDED to the noise value at a seeded index.
With V = 126464 and N(0, 1) noise the background mass is about V * e^{1/2}, so the literal
recipes give confidences of at most ~0.44 (h = 12) or ~0.94 (h = 15).  The "target" recipes
set the peak to log(V - 1) + sigma^2 / 2 + logit(u) instead, which places the confidence
near a chosen u in (0, 1) (the background's expected mass, not its exact sum), so that
multi-token commits, ties and profile-vs-factor differences are exercised.
"""
from __future__ import annotations

import ctypes
import dataclasses
import math
import os
import shutil
import subprocess

import numpy as np
import torch

LLADA_VOCAB = 126464


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    L: int
    V: int
    dtype: str                 # "bf16" | "fp16" | "fp32"
    sigma: float = 1.0         # noise standard deviation
    peak: str = "uniform"      # "uniform" | "zipf" | "levels" | "target" | "none"
    peak_lo: float = 0.0       # uniform: h ~ U[lo, hi]; target: u = 1 - 10^-a, a ~ U[lo, hi]
    peak_hi: float = 12.0
    levels: tuple = ()         # "levels": per tie group, h (or u for target_levels)
    zipf_s: float = 1.1
    zipf_cap: float = 15.0
    masked: str = "all"        # "all" | "frac_u01" | "frac_half_to_one"
    tie_group: int = 1         # >1: groups of this many positions share identical logits
    level_is_target: bool = False
    description: str = ""

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "fp32" else 2

    @property
    def torch_dtype(self):
        return {"bf16": torch.bfloat16, "fp16": torch.float16, "fp32": torch.float32}[self.dtype]


WORKLOADS = {
    # One block of 32 positions, all masked, bf16.
    "single_block_b1_l32_bf16": Workload(
        "single_block_b1_l32_bf16", 1, 32, LLADA_VOCAB, "bf16", 1.0, "uniform", 0.0, 12.0,
        description="B=1, L=32 all masked, N(0,1) + planted peak h~U[0,12], profile f=1"),
    # Active block of a length-256 generation, partially masked, bf16.
    "mixed_mask_b8_l32_bf16": Workload(
        "mixed_mask_b8_l32_bf16", 8, 32, LLADA_VOCAB, "bf16", 1.5, "uniform", 2.0, 14.0,
        masked="frac_u01",
        description="B=8, L=32, masked fraction U[0,1] per row, N(0,1.5^2) + h~U[2,14]"),
    # Equal-confidence groups (identical logits within groups of 8), fp32.
    "tie_groups_b16_l64_fp32": Workload(
        "tie_groups_b16_l64_fp32", 16, 64, LLADA_VOCAB, "fp32", 1.0, "levels",
        levels=(4.0, 6.0, 8.0, 10.0), tie_group=8,
        description="B=16, L=64 all masked, groups of 8 identical rows, h in {4,6,8,10}"),
    # Large-batch serving step, bf16 (the throughput workload).
    "serving_b64_l32_bf16": Workload(
        "serving_b64_l32_bf16", 64, 32, LLADA_VOCAB, "bf16", 1.0, "zipf",
        masked="frac_half_to_one",
        description="B=64, L=32, masked fraction U[0.5,1], N(0,1) + h=min(Zipf(1.1),15)"),
    # Whole-sequence multi-step loop, fp32, regenerated every step.
    "full_seq_b16_l1024_fp32": Workload(
        "full_seq_b16_l1024_fp32", 16, 1024, LLADA_VOCAB, "fp32", 1.0, "uniform", 0.0, 12.0,
        description="B=16, L=1024 all masked initially, N(0,1) + h~U[0,12], regenerated "
                    "from (seed, step) every step until no mask remains"),
    # Supplementary: planted target confidences (multi-commit decisions).
    "target_b8_l32_bf16": Workload(
        "target_b8_l32_bf16", 8, 32, LLADA_VOCAB, "bf16", 1.0, "target", 0.3, 4.0,
        masked="frac_u01",
        description="B=8, L=32, confidence near u = 1 - 10^-a, a~U[0.3,4]"),
    # Supplementary: fp16 logits (models that emit half precision).
    "target_b8_l32_fp16": Workload(
        "target_b8_l32_fp16", 8, 32, LLADA_VOCAB, "fp16", 1.0, "target", 0.3, 4.0,
        masked="frac_u01",
        description="B=8, L=32, fp16, confidence near u = 1 - 10^-a, a~U[0.3,4]"),
    "target_ties_b16_l64_fp32": Workload(
        "target_ties_b16_l64_fp32", 16, 64, LLADA_VOCAB, "fp32", 1.0, "levels",
        levels=(0.9, 0.99, 0.999, 0.9999), tie_group=8, level_is_target=True,
        description="B=16, L=64, groups of 8 identical rows at u in {.9,.99,.999,.9999}"),
}


def _rng(seed: int, salt: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([int(seed), int(salt)]))


def make_mask(w: Workload, seed: int) -> np.ndarray:
    """uint8 [B, L], 1 = masked."""
    rng = _rng(seed, 1)
    B, L = w.B, w.L
    if w.masked == "all":
        return np.ones((B, L), np.uint8)
    mask = np.zeros((B, L), np.uint8)
    for b in range(B):
        if w.masked == "frac_u01":
            frac = rng.uniform(0.0, 1.0)
        elif w.masked == "frac_half_to_one":
            frac = rng.uniform(0.5, 1.0)
        else:
            raise ValueError(w.masked)
        k = int(round(frac * L))
        mask[b, rng.choice(L, size=k, replace=False)] = 1
    return mask


def _target_peak(V: int, sigma: float, u: np.ndarray) -> np.ndarray:
    # Background expected mass (V-1) e^{sigma^2/2}; peak value placing softmax mass ~u on it.
    return math.log(V - 1) + 0.5 * sigma * sigma + np.log(u) - np.log1p(-u)


def make_peaks(w: Workload, seed: int, step: int = 0):
    """Planted peak (index int64 [B,L], value float64 [B,L], additive bool)."""
    rng = _rng(seed, 2 + 1000003 * step)
    B, L, V = w.B, w.L, w.V
    idx = rng.integers(0, V, size=(B, L), dtype=np.int64)
    if w.peak == "none":
        return idx, np.zeros((B, L)), True
    if w.peak == "uniform":
        return idx, rng.uniform(w.peak_lo, w.peak_hi, size=(B, L)), True
    if w.peak == "zipf":
        h = np.minimum(rng.zipf(w.zipf_s, size=(B, L)).astype(np.float64), w.zipf_cap)
        return idx, h, True
    if w.peak == "target":
        a = rng.uniform(w.peak_lo, w.peak_hi, size=(B, L))
        return idx, _target_peak(V, w.sigma, 1.0 - 10.0 ** (-a)), False
    if w.peak == "levels":
        g = w.tie_group
        lv = np.asarray(w.levels, np.float64)
        choice = lv[rng.integers(0, len(lv), size=(B, (L + g - 1) // g))]
        val = np.repeat(choice, g, axis=1)[:, :L]
        gidx = np.repeat(idx[:, ::g], g, axis=1)[:, :L]
        if w.level_is_target:
            return gidx, _target_peak(V, w.sigma, val), False
        return gidx, val, True
    raise ValueError(w.peak)


def make_logits(w: Workload, seed: int, device="cpu", step: int = 0,
                V: int | None = None) -> torch.Tensor:
    """[B, L, V] logits in the workload's dtype on ``device`` (seeded, deterministic for a
    given seed, step and device type).  ``V`` overrides the vocabulary size (small tests)."""
    if V is not None:
        w = dataclasses.replace(w, V=V)
    B, L, V = w.B, w.L, w.V
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(int(seed) * 1000003 + int(step))
    if w.tie_group > 1:
        G = (L + w.tie_group - 1) // w.tie_group
        base = torch.randn((B, G, V), generator=g, device=dev, dtype=torch.float32)
        x = base.repeat_interleave(w.tie_group, dim=1)[:, :L].contiguous()
    else:
        x = torch.randn((B, L, V), generator=g, device=dev, dtype=torch.float32)
    if w.sigma != 1.0:
        x.mul_(w.sigma)
    idx, val, additive = make_peaks(w, seed, step)
    flat = x.view(B * L, V)
    rows = torch.arange(B * L, device=dev)
    cols = torch.from_numpy(idx.reshape(-1)).to(dev)
    vals = torch.from_numpy(val.reshape(-1).astype(np.float32)).to(dev)
    if additive:
        flat[rows, cols] += vals
    else:
        flat[rows, cols] = vals
    return x if w.dtype == "fp32" else x.to(w.torch_dtype)


def host_bits(logits: torch.Tensor) -> np.ndarray:
    """Exact host copy of device/host logits for the oracle: bf16 -> uint16 bits, fp16 and
    fp32 as they are."""
    t = logits.detach().to("cpu").contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    if t.dtype in (torch.float32, torch.float16):
        return t.numpy()
    raise TypeError(t.dtype)


# ----------------------------------------------------------------------------- LM head
LLADA_HIDDEN = 4096


def make_lmhead_inputs(B: int, L: int, H: int, V: int, seed: int, beta_lo: float = 0.0,
                       beta_hi: float = 20.0, device="cpu"):
    """Seeded LM-head inputs (bf16): W [V, H] with N(0, 1/H) entries (rows of norm ~1), and
    per position a target token t ~ U{0..V-1}, a height beta ~ U[beta_lo, beta_hi] and
    hidden h = z + beta w_t / |w_t|^2 with z ~ N(0, I_H).  Then w_t . h ~ beta + N(0, 1) and
    w_v . h ~ N(0, 1 + beta^2 / H) for v != t (N(0, ~1) at H = 4096): a planted peak of height
    beta in logit space, as in the logits recipes.  Returns (hidden [B, L, H], w [V, H], targets [B, L])."""
    dev = torch.device(device)
    g = torch.Generator(device=dev)
    g.manual_seed(int(seed) * 7919 + 17)
    w = torch.empty((V, H), device=dev, dtype=torch.bfloat16)
    chunk = 16384  # rows drawn in fp32 at a time (bounded temporary memory)
    for v0 in range(0, V, chunk):
        part = torch.randn((min(chunk, V - v0), H), generator=g, device=dev,
                           dtype=torch.float32)
        w[v0:v0 + part.shape[0]] = (part * (1.0 / math.sqrt(H))).to(torch.bfloat16)
    t = torch.randint(0, V, (B, L), generator=g, device=dev)
    beta = torch.rand((B, L), generator=g, device=dev, dtype=torch.float32)
    beta = beta * (beta_hi - beta_lo) + beta_lo
    h = torch.randn((B, L, H), generator=g, device=dev, dtype=torch.float32)
    wt = w[t].float()
    h += beta[..., None] * wt / (wt * wt).sum(-1, keepdim=True)
    return h.to(torch.bfloat16), w, t


# ----------------------------------------------------------------------------- GPU stand-in
# Counter-based synthetic logits on the GPU (fdllm_synth_cuda.cu): the forward pass of the
# decode-loop tests and benchmarks.  The CPU oracle implements the same generator itself.
_HERE = os.path.dirname(os.path.abspath(__file__))
_SYNTH_SRC = os.path.join(_HERE, "fdllm_synth_cuda.cu")
_SYNTH_LIB = os.path.join(_HERE, "_build", "libfdllm_synth.so")
_synth = None


def build_synth_cuda(force: bool = False) -> str:
    if (not force and os.path.exists(_SYNTH_LIB)
            and os.path.getmtime(_SYNTH_LIB) >= os.path.getmtime(_SYNTH_SRC)):
        return _SYNTH_LIB
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    os.makedirs(os.path.dirname(_SYNTH_LIB), exist_ok=True)
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
                    "-lineinfo", "-Xcompiler", "-fPIC", "-shared", _SYNTH_SRC, "-o",
                    _SYNTH_LIB + ".tmp"],
                   check=True, capture_output=True, text=True)
    os.replace(_SYNTH_LIB + ".tmp", _SYNTH_LIB)
    return _SYNTH_LIB


def _synth_lib():
    global _synth
    if _synth is None:
        lib = ctypes.CDLL(build_synth_cuda())
        p, i = ctypes.c_void_p, ctypes.c_int
        lib.fdllm_synth_block_logits.argtypes = [p, p, i, i, i, ctypes.c_ulonglong, p,
                                                 ctypes.c_longlong, ctypes.c_double, p]
        lib.fdllm_synth_block_logits.restype = i
        lib.fdllm_synth_block_hidden.argtypes = [p, p, i, i, i, i, p, ctypes.c_ulonglong, p,
                                                 ctypes.c_longlong, ctypes.c_double, p]
        lib.fdllm_synth_block_hidden.restype = i
        _synth = lib
    return _synth


def synth_block_logits_gpu(out_ptr, mask_ptr, B, L, V, seed, step_ptr=None, step=0,
                           peak_max=16.0, stream_ptr=None):
    """Enqueue counter-based bf16 logits [B, L, V] (raw device pointers; rows whose mask
    byte is 0 are skipped; the step is read from step_ptr on the device when given)."""
    err = _synth_lib().fdllm_synth_block_logits(out_ptr, mask_ptr, B, L, V, int(seed), step_ptr,
                                                int(step), float(peak_max), stream_ptr)
    if err != 0:
        raise RuntimeError("synthetic logits launch failed: %d" % err)


def synth_block_hidden_gpu(out_ptr, mask_ptr, B, L, H, V, w_ptr, seed, step_ptr=None, step=0,
                           beta_max=16.0, stream_ptr=None):
    """Enqueue counter-based bf16 hidden states [B, L, H] against the bf16 head w [V, H]
    (raw device pointers; rows whose mask byte is 0 are skipped; the step is read from
    step_ptr on the device when given)."""
    err = _synth_lib().fdllm_synth_block_hidden(out_ptr, mask_ptr, B, L, H, V, w_ptr, int(seed),
                                                step_ptr, int(step), float(beta_max), stream_ptr)
    if err != 0:
        raise RuntimeError("synthetic hidden-state launch failed: %d" % err)
