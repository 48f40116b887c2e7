"""A seeded random sweep of the selection against the oracle, through the C interface.

Each case draws its own shape (B, L, V with ragged chunks and units), dtype, noise scale,
kind of planted peak (none, uniform height, Zipf height, or a target confidence), mask
density (empty rows included) and rule with its parameter, so that combinations that no
hand-written case names are exercised too.  The bars are the parity tests': tokens
bit-exact, confidences within 1e-5 relative, decisions bit-exact on rows with decision
margin >= 1e-5 and, on every row, equal to the rule applied to the GPU's own confidences.
"""
import numpy as np
import pytest

import fdllm_synth as syn
from gpu_util import CONF_RTOL, check_confidence, check_select

PROFILE, FACTOR, THRESHOLD = 0, 1, 2


def draw_case(seed):
    rng = np.random.default_rng(20_000 + seed)
    dtype = ("bf16", "fp16", "fp32")[rng.integers(3)]
    q = 4 if dtype == "fp32" else 8  # V * sizeof(dtype) a multiple of 16
    # from one vector per row to LLaDA's vocabulary: ragged chunks, units and tails
    V = int(rng.choice([8, 24, 1000, 1032, 8200, 32776, 40000, 126464]))
    V = (V + q - 1) // q * q
    B = int(rng.integers(1, 7))
    L = int(rng.integers(1, 71))
    sigma = float(rng.choice([0.5, 1.0, 2.0, 4.0]))
    peak = ("none", "uniform", "zipf", "target")[rng.integers(4)]
    if peak == "target":
        lo, hi = 0.3, 4.0  # confidence u = 1 - 10^-a, a ~ U[lo, hi]
    else:
        lo, hi = 0.0, float(rng.uniform(2.0, 20.0))
    w = syn.Workload("fuzz_%d" % seed, B, L, V, dtype, sigma, peak, lo, hi)
    mrng = np.random.default_rng(seed)
    frac = mrng.uniform(0.0, 1.0, size=(B, 1))
    frac[mrng.random((B, 1)) < 0.15] = 0.0  # some rows with nothing masked
    mask = (mrng.random((B, L)) < frac).astype(np.uint8)
    mode = int(rng.integers(3))
    if mode == THRESHOLD:
        param = float(rng.choice([0.3, 0.5, 0.9]))
    else:
        param = float(rng.choice([0.5, 0.75, 1.0, 2.0]))
    return w, mask, mode, param


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(128))
def test_random_case_matches_oracle(fd, orc, seed):
    w, mask, mode, param = draw_case(seed)
    logits = syn.make_logits(w, seed=seed, device="cuda")
    check_confidence(fd, orc, logits, mask)
    check_select(fd, orc, logits, mask, mode, param)


def test_draws_cover_the_space():
    """The 32 drawn cases span every dtype, peak kind and rule, and include empty rows."""
    cases = [draw_case(s) for s in range(32)]
    assert {c[0].dtype for c in cases} == {"bf16", "fp16", "fp32"}
    assert {c[0].peak for c in cases} == {"none", "uniform", "zipf", "target"}
    assert {c[2] for c in cases} == {PROFILE, FACTOR, THRESHOLD}
    assert any((c[1].sum(axis=1) == 0).any() for c in cases)


def draw_lmhead_case(seed):
    rng = np.random.default_rng(30_000 + seed)
    B = int(rng.integers(1, 5))
    L = int(rng.integers(1, 65))
    H = int(rng.choice([8, 40, 72, 256, 520, 1024]))
    V = int(rng.choice([40, 300, 1000, 2050, 5000, 20000]))
    variant = ("auto", "solo", "pair", "slab")[rng.integers(4)]
    bn = int(rng.choice([256, 208]))
    frac = float(rng.uniform(0.2, 1.0))
    return B, L, H, V, variant, bn, frac


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(48))
def test_random_lmhead_case_matches_oracle(fd, orc, monkeypatch, seed):
    """The LM-head path on drawn shapes (H not a multiple of the K stage, V ragged against
    every tile), GEMM variants and tile widths: the stored logits within the fp32
    accumulation bound of the exact ones, and the fused confidences and tokens against the
    oracle on those same accumulators."""
    import torch
    from test_gpu_lmhead import bits, gemm_bound, gpu_logits, inputs

    B, L, H, V, variant, bn, frac = draw_lmhead_case(seed)
    if variant == "auto":
        monkeypatch.delenv("FDLLM_LMHEAD_GEMM", raising=False)
    else:
        monkeypatch.setenv("FDLLM_LMHEAD_GEMM", variant)  # slab only where B * L <= 32
    monkeypatch.setenv("FDLLM_LMHEAD_BN", str(bn))
    h, w, mask_np = inputs(B, L, H, V, seed=40_000 + seed, frac=frac)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    x32 = gpu_logits(fd, h, w, mask_np)
    mk = mask_np.astype(bool)
    rc, rt, bad = orc.confidence(x32, mask_np)
    assert bad == 0
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    assert np.array_equal(g_tok[mk], rt[mk])
    if mk.any():
        assert (np.abs(g_conf[mk] - rc[mk]) / rc[mk]).max() <= CONF_RTOL
    ref, mag = orc.lmhead_logits(bits(h), bits(w), mask=mask_np, with_abs=True)
    err = np.abs(x32[mk].astype(np.float64) - ref[mk])
    assert (err <= gemm_bound(mag[mk], ref[mk], H)).all()
    assert fd.fdllm_device_status() == 0


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(48))
def test_random_robust_case_matches_oracle(fd, orc, seed):
    """The calibration-robust rule on the drawn cases, with a drawn uniform allowance or a
    drawn per-position one (App. C), against the oracle's robust selector."""
    from test_gpu_robust import _check

    w, mask, _, _ = draw_case(100 + seed)
    rng = np.random.default_rng(50_000 + seed)
    param = float(rng.choice([0.5, 0.75, 1.0]))
    logits = syn.make_logits(w, seed=100 + seed, device="cuda")
    if rng.random() < 0.5:
        _check(fd, orc, logits, mask, param, float(rng.uniform(0.0, 0.3)))
    else:
        _check(fd, orc, logits, mask, param, 0.0, rng.uniform(0.0, 0.3, (w.B, w.L)))


def draw_large_shape_case(seed):
    """Many rows and long blocks on small vocabularies: B * L up to 65536 and L from 1 to
    1024 (both selection kernels, the reduction's mask compaction and work queue over many
    rows), at sizes the oracle finishes quickly."""
    rng = np.random.default_rng(90_000 + seed)
    dtype = ("bf16", "fp16", "fp32")[rng.integers(3)]
    q = 4 if dtype == "fp32" else 8
    V = int(rng.choice([8, 16, 24, 120, 1000]))
    V = (V + q - 1) // q * q
    L = int(rng.choice([1, 2, 31, 32, 33, 64, 100, 257, 512, 1024]))
    B = int(rng.integers(1, max(1, min(64, 65536 // L)) + 1))
    peak = ("none", "uniform", "target")[rng.integers(3)]
    lo, hi = (0.3, 4.0) if peak == "target" else (0.0, float(rng.uniform(2.0, 20.0)))
    w = syn.Workload("fuzz_large_%d" % seed, B, L, V, dtype, 1.0, peak, lo, hi)
    mrng = np.random.default_rng(seed)
    frac = mrng.uniform(0.0, 1.0, size=(B, 1))
    frac[mrng.random((B, 1)) < 0.2] = 0.0
    mask = (mrng.random((B, L)) < frac).astype(np.uint8)
    mode = int(rng.integers(3))
    if mode == THRESHOLD:
        param = float(rng.choice([0.3, 0.5, 0.9]))
    else:
        param = float(rng.choice([0.5, 0.75, 1.0, 2.0]))
    return w, mask, mode, param


@pytest.mark.gpu
@pytest.mark.parametrize("seed", range(64))
def test_random_large_shape_case_matches_oracle(fd, orc, seed):
    w, mask, mode, param = draw_large_shape_case(seed)
    logits = syn.make_logits(w, seed=seed, device="cuda")
    check_confidence(fd, orc, logits, mask)
    check_select(fd, orc, logits, mask, mode, param)


def test_large_shape_draws_cover_the_space():
    """The 64 large-shape draws reach both selection kernels and thousands of rows."""
    cases = [draw_large_shape_case(s) for s in range(64)]
    assert min(c[0].L for c in cases) <= 32 < max(c[0].L for c in cases)
    assert max(c[0].B * c[0].L for c in cases) >= 8192
    assert {c[0].dtype for c in cases} == {"bf16", "fp16", "fp32"}
