"""Calibration-robust profile selection (App. C) on the GPU against the oracle."""
import numpy as np
import pytest
import torch

import fdllm_synth as syn
from gpu_util import MARGIN, oracle_threads

pytestmark = pytest.mark.gpu


def _check(fd, orc, logits, mask_np, param, eta, eta_pos=None):
    mask = torch.from_numpy(mask_np.copy()).cuda()
    ep = None if eta_pos is None else torch.from_numpy(eta_pos.astype(np.float32)).cuda()
    tok, commit, n = fd.fdllm_select_robust(logits, mask, param, eta, ep)
    torch.cuda.synchronize()
    g = [x.cpu().numpy() for x in (tok, commit, n, mask)]
    # the oracle sees the same fp32 allowances the GPU uses
    ep64 = None if eta_pos is None else eta_pos.astype(np.float32).astype(np.float64)
    ref = orc.select_robust(syn.host_bits(logits), mask_np, param,
                            float(np.float32(eta)), ep64, nthreads=oracle_threads())
    ok = ref["margin"] >= MARGIN
    assert np.array_equal(g[2][ok], ref["n"][ok]), (g[2], ref["n"])
    assert np.array_equal(g[1][ok], ref["commit"][ok])
    assert np.array_equal(g[3][ok], ref["mask"][ok])
    assert np.array_equal(g[0][ok], ref["tokens"][ok])
    # every row: the GPU decision is the rule applied to the GPU's own confidences
    conf, amax = fd.fdllm_confidence(logits, torch.from_numpy(mask_np).cuda())
    rg = orc.select_robust_from_conf(conf.cpu().numpy().astype(np.float64), amax.cpu().numpy(),
                                     mask_np, param, float(np.float32(eta)), ep64)
    same = rg["margin"] >= 1e-12
    assert np.array_equal(g[2][same], rg["n"][same])
    assert np.array_equal(g[1][same], rg["commit"][same])
    return int((~ok).sum())


@pytest.mark.parametrize("eta", [0.0, 0.01, 0.05, 0.2])
@pytest.mark.parametrize("name", ["target_b8_l32_bf16", "target_ties_b16_l64_fp32",
                                  "mixed_mask_b8_l32_bf16", "target_b8_l32_fp16"])
def test_robust_uniform_eta(fd, orc, name, eta):
    w = syn.WORKLOADS[name]
    logits = syn.make_logits(w, seed=606, device="cuda")
    mask_np = syn.make_mask(w, seed=606)
    for f in (1.0, 0.75):
        _check(fd, orc, logits, mask_np, f, eta)


@pytest.mark.parametrize("name", ["target_b8_l32_bf16", "target_ties_b16_l64_fp32",
                                  "target_b8_l32_fp16"])
def test_robust_per_position_eta(fd, orc, name):
    w = syn.WORKLOADS[name]
    logits = syn.make_logits(w, seed=707, device="cuda")
    mask_np = syn.make_mask(w, seed=707)
    eta_pos = np.random.default_rng(7).uniform(0.0, 0.1, (w.B, w.L))
    _check(fd, orc, logits, mask_np, 0.75, 0.0, eta_pos)


def test_robust_zero_eta_equals_profile(fd):
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=808, device="cuda")
    mask_np = syn.make_mask(w, seed=808)
    m1 = torch.from_numpy(mask_np.copy()).cuda()
    m2 = torch.from_numpy(mask_np.copy()).cuda()
    a = fd.fdllm_select(logits, m1, 0.75, fd.PROFILE)
    b = fd.fdllm_select_robust(logits, m2, 0.75, 0.0)
    for x, y in zip(list(a) + [m1], list(b) + [m2]):
        assert torch.equal(x, y)


def test_robust_full_size_serving_sample(fd, orc):
    w = syn.WORKLOADS["serving_b64_l32_bf16"]
    logits = syn.make_logits(w, seed=909, device="cuda")
    mask_np = syn.make_mask(w, seed=909)
    rows = [0, 9, 33, 63]
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_select_robust(logits, mask, 1.0, 0.02)
    torch.cuda.synchronize()
    ref = orc.select_robust(syn.host_bits(logits[rows]), mask_np[rows], 1.0,
                            float(np.float32(0.02)), None, nthreads=oracle_threads())
    for k, b in enumerate(rows):
        if ref["margin"][k] < MARGIN:
            continue
        assert n[b].item() == ref["n"][k]
        assert np.array_equal(commit[b].cpu().numpy(), ref["commit"][k])


def test_robust_negative_and_nan_allowances_read_as_zero(fd, orc):
    """Per-position allowances below 0 or NaN (outside App. C's eta >= 0) are read as 0:
    against the oracle, and bit for bit the decisions with those entries set to 0."""
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=909, device="cuda")
    mask_np = syn.make_mask(w, seed=909)
    rng = np.random.default_rng(9)
    eta_pos = rng.uniform(-0.2, 0.1, (w.B, w.L))
    eta_pos[::2, ::5] = np.nan
    _check(fd, orc, logits, mask_np, 0.75, 0.0, eta_pos)
    clean = np.where(np.isnan(eta_pos) | (eta_pos < 0.0), 0.0, eta_pos)
    outs = []
    for e in (eta_pos, clean):
        mask = torch.from_numpy(mask_np.copy()).cuda()
        ep = torch.from_numpy(e.astype(np.float32)).cuda()
        outs.append([x.cpu() for x in fd.fdllm_select_robust(logits, mask, 0.75, 0.0, ep)]
                    + [mask.cpu()])
    for x, y in zip(*outs):
        assert torch.equal(x, y)
