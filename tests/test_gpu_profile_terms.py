"""Heterogeneity-bonus diagnostics on the GPU against the oracle (same fp32 inputs)."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,L", [(1, 1), (5, 32), (3, 100), (2, 1024), (16, 64)])
def test_profile_terms_match_oracle(fd, orc, B, L):
    rng = np.random.default_rng(B * 1000 + L)
    c = np.clip(rng.beta(0.6, 0.25, (B, L)), 1e-6, 1.0).astype(np.float32)
    c[0, : min(L, 5)] = c[0, 0]  # ties
    mask_np = (rng.random((B, L)) < 0.8).astype(np.uint8)
    if B > 1:
        mask_np[-1] = 0
    delta = 0.25
    t = fd.fdllm_profile_terms(torch.from_numpy(c).cuda(), torch.from_numpy(mask_np).cuda(),
                               delta)
    ref = orc.profile_terms(c.astype(np.float64), mask_np)
    ref = dict(ref, f_eff=1.0 - delta + ref["B"])  # Remark adaptive-factor, on the oracle's B
    assert np.array_equal(t["order"].cpu().numpy(), ref["order"])
    for k in ("G", "F", "B", "f_eff"):
        g, r = t[k].cpu().numpy(), ref[k]
        assert np.array_equal(np.isnan(g), np.isnan(r))
        ok = ~np.isnan(r)
        np.testing.assert_allclose(g[ok], r[ok], rtol=0, atol=1e-12 * L)


def test_profile_terms_decomposition_on_gpu_confidences(fd):
    """G = F + B wherever the lower bound is positive, B >= 0 (fp64 on the GPU)."""
    rng = np.random.default_rng(3)
    c = (rng.integers(1, 257, (8, 32)) / 256).astype(np.float32)
    mask = torch.ones((8, 32), dtype=torch.uint8, device="cuda")
    t = fd.fdllm_profile_terms(torch.from_numpy(c).cuda(), mask)
    G, F, Bn = (t[k].cpu().numpy() for k in ("G", "F", "B"))
    cs = -np.sort(-c.astype(np.float64), axis=1)
    S = np.cumsum(cs, axis=1)
    n = np.arange(1, 33)
    active = S - (n - 1) > 0
    assert np.all(Bn >= -1e-12)
    assert np.allclose(G[active], F[active] + Bn[active], atol=1e-12)


@pytest.mark.parametrize("delta", [0.0, 0.25, 0.5])
def test_profile_rule_is_the_factor_rule_with_f_eff(fd, delta):
    """Remark adaptive-factor: where the lower bound is positive, G_n > delta exactly when
    (n+1)(1 - c_(n)) < f_eff(n) (dyadic confidences: no rounding at the comparisons)."""
    rng = np.random.default_rng(11)
    c = (rng.integers(128, 257, (8, 32)) / 256).astype(np.float32)
    mask = torch.ones((8, 32), dtype=torch.uint8, device="cuda")
    t = fd.fdllm_profile_terms(torch.from_numpy(c).cuda(), mask, delta)
    G, Fe = t["G"].cpu().numpy(), t["f_eff"].cpu().numpy()
    cs = -np.sort(-c.astype(np.float64), axis=1)
    n = np.arange(1, 33)
    active = np.cumsum(cs, axis=1) - (n - 1) > 0
    lhs = G > delta
    rhs = (n + 1) * (1.0 - cs) < Fe
    boundary = np.isclose(G, delta, atol=1e-12) | np.isclose((n + 1) * (1.0 - cs), Fe, atol=1e-12)
    keep = active & ~boundary
    assert keep.sum() > 50
    assert np.array_equal(lhs[keep], rhs[keep])
