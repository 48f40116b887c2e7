"""Plain fp64 CPU oracle for Frechet profile commit-set selection.

TEST INFRASTRUCTURE ONLY.  The oracle checks the CUDA library; only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference arm may import
it.  The product package never imports it, and it imports nothing from the product.

The arithmetic lives in ``fdllm_oracle.c`` (plain C, double precision, the steps of the
paper's Algorithm 1 in order).  This module only compiles that file with gcc and
marshals numpy arrays through ctypes.

Parameter conventions (same meaning as the library's public interface):
  mode  0 = profile (Frechet, Sec. 3), 1 = factor, 2 = threshold.
  param profile: f with margin delta = 1 - f (Cor. factor-reduction); factor: f;
        threshold: tau.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

PROFILE, FACTOR, THRESHOLD = 0, 1, 2
BF16, FP32, F64, F16 = 0, 1, 2, 3

HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(HERE, "fdllm_oracle.c")
HEADER = os.path.join(HERE, "fdllm_oracle.h")
_OUT_DIR = os.path.join(HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_default = None


def compile_oracle(src: str, out: str) -> str:
    """gcc the C oracle at ``src`` into the shared library ``out`` (OpenMP when present)."""
    os.makedirs(os.path.dirname(out), exist_ok=True)
    base = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
            "-I", HERE, src, "-o", out + ".tmp", "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True, text=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True, text=True)
    os.replace(out + ".tmp", out)
    return out


def build_oracle(force: bool = False) -> str:
    """Compile the committed oracle if its library is missing or stale; return its path."""
    fresh = (os.path.exists(_LIB_PATH)
             and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(SOURCE)
             and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(HEADER))
    if fresh and not force:
        return _LIB_PATH
    return compile_oracle(SOURCE, _LIB_PATH)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _logits_view(logits: np.ndarray):
    """Accept fp16, fp32 or fp64 arrays, or bf16 given as raw uint16 bits; return (array,
    code)."""
    a = np.ascontiguousarray(logits)
    if a.dtype == np.uint16:
        return a, BF16
    if a.dtype == np.float32:
        return a, FP32
    if a.dtype == np.float64:
        return a, F64
    if a.dtype == np.float16:
        return a, F16
    raise TypeError("oracle logits must be float16, float32, float64 or uint16 (bf16 bits), "
                    "got %s" % a.dtype)


class Oracle:
    """ctypes front end of one compiled oracle library."""

    def __init__(self, lib_path: str):
        lib = ctypes.CDLL(lib_path)
        p, i64, i32, d = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double
        lib.oracle_confidence.argtypes = [p, i32, i64, i64, i64, p, p, p, i32]
        lib.oracle_confidence.restype = i64
        lib.oracle_frechet_scan.argtypes = [p, i64, p, p, p]
        lib.oracle_frechet_scan.restype = None
        lib.oracle_select_from_conf.argtypes = [p, p, i64, i64, p, i32, d, p, p, p, p]
        lib.oracle_select_from_conf.restype = i64
        lib.oracle_select_robust_from_conf.argtypes = [p, p, i64, i64, p, d, d, p, p, p, p, p]
        lib.oracle_select_robust_from_conf.restype = i64
        lib.oracle_bonus_terms.argtypes = [p, i64, p, p]
        lib.oracle_bonus_terms.restype = None
        lib.oracle_profile_terms.argtypes = [p, p, i64, i64, p, p, p, p]
        lib.oracle_profile_terms.restype = None
        u64 = ctypes.c_uint64
        lib.oracle_synth_block_logits.argtypes = [p, p, i64, i64, i64, u64, u64, d]
        lib.oracle_synth_block_logits.restype = None
        lib.oracle_decode_loop.argtypes = [i64, i64, i64, i64, i32, d, u64, d, i64, p, p, p, i32]
        lib.oracle_decode_loop.restype = i64
        lib.oracle_synth_block_hidden.argtypes = [p, p, i64, i64, i64, i64, p, u64, u64, d]
        lib.oracle_synth_block_hidden.restype = None
        lib.oracle_half_to_double.argtypes = [p, i64, p]
        lib.oracle_half_to_double.restype = None
        lib.oracle_lmhead_logits.argtypes = [p, p, i64, i64, i64, p, p, p, i32]
        lib.oracle_lmhead_logits.restype = None
        self.lib = lib
        self.path = lib_path

    def confidence(self, logits: np.ndarray, mask: np.ndarray, nthreads: int = 1):
        """Per masked position: (conf float64 [B,L], tok int32 [B,L], invalid row count).

        Unmasked positions hold conf = 0 and tok = -1 (the oracle does not write them)."""
        a, code = _logits_view(logits)
        B, L, V = a.shape
        m = np.ascontiguousarray(mask, dtype=np.uint8).reshape(B, L)
        conf = np.zeros((B, L), np.float64)
        tok = np.full((B, L), -1, np.int32)
        bad = self.lib.oracle_confidence(_ptr(a), code, B, L, V, _ptr(m), _ptr(conf),
                                         _ptr(tok), int(nthreads))
        return conf, tok, int(bad)

    def frechet_scan(self, c_sorted):
        """(L_n, U_n, G_n) for n = 1..m of a descending profile (Eq. frechet_Ln_Un)."""
        c = np.ascontiguousarray(c_sorted, dtype=np.float64)
        m = c.shape[0]
        Ln, Un, Gn = (np.zeros(m, np.float64) for _ in range(3))
        self.lib.oracle_frechet_scan(_ptr(c), m, _ptr(Ln), _ptr(Un), _ptr(Gn))
        return Ln, Un, Gn

    def bonus_terms(self, c_sorted):
        """(F_n, B_n) for n = 1..m of a descending profile (Eq. heterogeneity_decomp)."""
        c = np.ascontiguousarray(c_sorted, dtype=np.float64)
        m = c.shape[0]
        F, Bn = np.zeros(m), np.zeros(m)
        self.lib.oracle_bonus_terms(_ptr(c), m, _ptr(F), _ptr(Bn))
        return F, Bn

    def profile_terms(self, conf: np.ndarray, mask: np.ndarray):
        """Per batch row at each rank of the sorted masked profile: dict(G, F, B, order)."""
        c = np.ascontiguousarray(conf, dtype=np.float64)
        B, L = c.shape
        m = np.ascontiguousarray(mask, dtype=np.uint8).reshape(B, L)
        G, F, Bn = (np.zeros((B, L)) for _ in range(3))
        order = np.zeros((B, L), np.int32)
        self.lib.oracle_profile_terms(_ptr(c), _ptr(m), B, L, _ptr(G), _ptr(F), _ptr(Bn),
                                      _ptr(order))
        return dict(G=G, F=F, B=Bn, order=order)

    def half_to_double(self, bits: np.ndarray) -> np.ndarray:
        """The oracle's fp16 widening of raw half bit patterns (uint16) to float64."""
        b = np.ascontiguousarray(bits, np.uint16).reshape(-1)
        out = np.zeros(b.shape, np.float64)
        self.lib.oracle_half_to_double(_ptr(b), b.size, _ptr(out))
        return out

    def lmhead_logits(self, hidden_bits: np.ndarray, w_bits: np.ndarray, mask=None,
                      with_abs: bool = False, nthreads: int = 1):
        """Exact (fp64) logits of the LM head at masked rows: hidden [B, L, H] and w [V, H]
        as bf16 bits (uint16).  Returns logits [B, L, V] (zero at unmasked rows) and, with
        with_abs, the magnitudes sum_k |h_k w_vk| of the same shape."""
        h = np.ascontiguousarray(hidden_bits, np.uint16)
        w = np.ascontiguousarray(w_bits, np.uint16)
        B, L, H = h.shape
        V = w.shape[0]
        assert w.shape == (V, H)
        m = None if mask is None else np.ascontiguousarray(mask, np.uint8).reshape(B, L)
        out = np.zeros((B, L, V), np.float64)
        mag = np.zeros((B, L, V), np.float64) if with_abs else None
        self.lib.oracle_lmhead_logits(_ptr(h), _ptr(w), B * L, H, V,
                                      None if m is None else _ptr(m), _ptr(out),
                                      None if mag is None else _ptr(mag), int(nthreads))
        return (out, mag) if with_abs else out

    def synth_block_hidden(self, w_bits, B, L, seed, step, beta_max, mask=None):
        """Counter-based synthetic bf16 hidden states (uint16 bits [B, L, H]) against the
        bf16 head w (uint16 bits [V, H]); unmasked rows zero."""
        w = np.ascontiguousarray(w_bits, np.uint16)
        V, H = w.shape
        out = np.zeros((B, L, H), np.uint16)
        m = None if mask is None else np.ascontiguousarray(mask, np.uint8).reshape(B, L)
        self.lib.oracle_synth_block_hidden(_ptr(out), None if m is None else _ptr(m), B, L, H,
                                           V, _ptr(w), int(seed), int(step), float(beta_max))
        return out

    def synth_block_logits(self, B, L, V, seed, step, peak_max, mask=None):
        """Counter-based synthetic bf16 logits (uint16 bits [B, L, V]); unmasked rows zero."""
        out = np.zeros((B, L, V), np.uint16)
        m = None if mask is None else np.ascontiguousarray(mask, np.uint8).reshape(B, L)
        self.lib.oracle_synth_block_logits(_ptr(out), None if m is None else _ptr(m), B, L, V,
                                           int(seed), int(step), float(peak_max))
        return out

    def decode_loop(self, B, gen_len, block_len, V, mode, param, seed, peak_max, max_steps,
                    nthreads: int = 1):
        """Algorithm 1's outer loop on the synthetic forward: dict(seq, nfe, margin, steps)."""
        seq = np.zeros((B, gen_len), np.int32)
        nfe = np.zeros(gen_len // block_len, np.int32)
        margin = np.zeros(B, np.float64)
        steps = self.lib.oracle_decode_loop(B, gen_len, block_len, V, int(mode), float(param),
                                            int(seed), float(peak_max), int(max_steps),
                                            _ptr(seq), _ptr(nfe), _ptr(margin), int(nthreads))
        return dict(seq=seq, nfe=nfe, margin=margin, steps=int(steps))

    def select_from_conf(self, conf: np.ndarray, tok: np.ndarray, mask: np.ndarray, mode: int,
                         param: float, out_tokens: np.ndarray | None = None):
        """Sort / scan / select / reveal on given confidences.

        Returns dict(tokens, commit, n, margin, mask, invalid_rows); ``mask`` is the updated
        copy (the input array is left untouched)."""
        c = np.ascontiguousarray(conf, dtype=np.float64)
        B, L = c.shape
        t = np.ascontiguousarray(tok, dtype=np.int32).reshape(B, L)
        m = np.array(mask, dtype=np.uint8, copy=True).reshape(B, L)
        toks = (np.full((B, L), -1, np.int32) if out_tokens is None
                else np.array(out_tokens, dtype=np.int32, copy=True).reshape(B, L))
        commit = np.zeros((B, L), np.uint8)
        n = np.zeros(B, np.int32)
        margin = np.zeros(B, np.float64)
        bad = self.lib.oracle_select_from_conf(_ptr(c), _ptr(t), B, L, _ptr(m), int(mode),
                                               float(param), _ptr(toks), _ptr(commit), _ptr(n),
                                               _ptr(margin))
        return dict(tokens=toks, commit=commit, n=n, margin=margin, mask=m,
                    invalid_rows=int(bad))

    def select_robust_from_conf(self, conf: np.ndarray, tok: np.ndarray, mask: np.ndarray,
                                param: float, eta: float, eta_pos: np.ndarray | None = None,
                                out_tokens: np.ndarray | None = None):
        """Calibration-robust profile selection (App. C) on given confidences; eta_pos
        (per position, [B, L]) replaces the uniform eta when given.  Same result dict as
        select_from_conf."""
        c = np.ascontiguousarray(conf, dtype=np.float64)
        B, L = c.shape
        t = np.ascontiguousarray(tok, dtype=np.int32).reshape(B, L)
        m = np.array(mask, dtype=np.uint8, copy=True).reshape(B, L)
        e = None if eta_pos is None else np.ascontiguousarray(eta_pos, np.float64).reshape(B, L)
        toks = (np.full((B, L), -1, np.int32) if out_tokens is None
                else np.array(out_tokens, dtype=np.int32, copy=True).reshape(B, L))
        commit = np.zeros((B, L), np.uint8)
        n = np.zeros(B, np.int32)
        margin = np.zeros(B, np.float64)
        bad = self.lib.oracle_select_robust_from_conf(
            _ptr(c), _ptr(t), B, L, _ptr(m), float(param), float(eta),
            None if e is None else _ptr(e), _ptr(toks), _ptr(commit), _ptr(n), _ptr(margin))
        return dict(tokens=toks, commit=commit, n=n, margin=margin, mask=m,
                    invalid_rows=int(bad))

    def select_robust(self, logits: np.ndarray, mask: np.ndarray, param: float, eta: float,
                      eta_pos: np.ndarray | None = None, nthreads: int = 1):
        """Whole calibration-robust step on host logits."""
        conf, tok, _ = self.confidence(logits, mask, nthreads)
        res = self.select_robust_from_conf(conf, tok, mask, param, eta, eta_pos)
        res["conf"] = conf
        res["tok"] = tok
        return res

    def select(self, logits: np.ndarray, mask: np.ndarray, mode: int, param: float,
               out_tokens: np.ndarray | None = None, nthreads: int = 1):
        """Whole selection step (Alg. 1 from confidences to reveal) on host logits."""
        conf, tok, _ = self.confidence(logits, mask, nthreads)
        res = self.select_from_conf(conf, tok, mask, mode, param, out_tokens)
        res["conf"] = conf
        res["tok"] = tok
        return res


def default() -> Oracle:
    global _default
    with _lock:
        if _default is None:
            _default = Oracle(build_oracle())
        return _default


def confidence(logits, mask, nthreads: int = 1):
    return default().confidence(logits, mask, nthreads)


def frechet_scan(c_sorted):
    return default().frechet_scan(c_sorted)


def select_from_conf(conf, tok, mask, mode, param, out_tokens=None):
    return default().select_from_conf(conf, tok, mask, mode, param, out_tokens)


def select(logits, mask, mode, param, out_tokens=None, nthreads: int = 1):
    return default().select(logits, mask, mode, param, out_tokens, nthreads)
