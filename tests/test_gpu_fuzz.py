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
from gpu_util import check_confidence, check_select

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
@pytest.mark.parametrize("seed", range(32))
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
