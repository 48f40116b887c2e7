"""Shared helpers of the GPU parity tests: run the CUDA path and the oracle on the same bytes
and compare them with the stated tolerances.

Tolerances (fixed by the selection's contract):
  * argmax tokens: bit-exact at every masked position (the max of identical inputs is exact);
  * confidences: within CONF_RTOL relative of the oracle's fp64 value;
  * n*, commit masks, committed tokens and the updated mask: bit-exact, except on rows whose
    oracle decision margin is below MARGIN (a rule quantity or a confidence gap that close to
    its boundary can flip under fp32 confidences); those rows are counted and returned, and
    the GPU decision on them is still checked against the oracle's rule applied to the GPU's
    own confidences.
"""
from __future__ import annotations

import numpy as np
import torch

import fdllm_synth

CONF_RTOL = 1e-5
MARGIN = 1e-5
ERR_NONFINITE = 3   # fdllm_status FDLLM_ERR_NONFINITE
ROW_NONFINITE = -1  # out_n of a row with unusable logits


def oracle_threads() -> int:
    import os
    return max(1, min(16, os.cpu_count() or 1))


def check_confidence(fd, orc, logits: torch.Tensor, mask_np: np.ndarray):
    """fdllm_confidence against the oracle at every masked position."""
    mask = torch.from_numpy(mask_np).cuda()
    conf, tok = fd.fdllm_confidence(logits, mask)
    torch.cuda.synchronize()
    host = fdllm_synth.host_bits(logits)
    rc, rt, rbad = orc.confidence(host, mask_np, nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    g_conf = conf.cpu().numpy().astype(np.float64)
    g_tok = tok.cpu().numpy()
    ref_bad = np.isnan(rc) & mk
    assert np.array_equal(np.isnan(g_conf) & mk, ref_bad), "non-finite rows differ"
    good = mk & ~ref_bad
    assert np.array_equal(g_tok[good], rt[good]), "argmax differs at %d positions" % int(
        np.sum(g_tok[good] != rt[good]))
    assert np.all(g_tok[ref_bad] == -1)
    if good.any():
        rel = np.abs(g_conf[good] - rc[good]) / rc[good]
        assert rel.max() <= CONF_RTOL, "max relative confidence error %.3g" % rel.max()
    # unmasked positions are never written
    assert np.all(np.isnan(g_conf[~mk])) and np.all(g_tok[~mk] == -1)
    return g_conf, g_tok, rc, rt


def check_select(fd, orc, logits: torch.Tensor, mask_np: np.ndarray, mode: int, param: float,
                 ref=None):
    """fdllm_select against the oracle; returns the number of low-margin rows."""
    B, L = mask_np.shape
    mask = torch.from_numpy(mask_np.copy()).cuda()
    assert fd.fdllm_device_status() == 0, "status word already set before this call"
    tok, commit, n = fd.fdllm_select(logits, mask, param, mode)
    status = fd.fdllm_device_status()  # synchronises; reads and clears the status word
    g = dict(tokens=tok.cpu().numpy(), commit=commit.cpu().numpy(), n=n.cpu().numpy(),
             mask=mask.cpu().numpy())
    if ref is None:
        host = fdllm_synth.host_bits(logits)
        ref = orc.select(host, mask_np, mode, param, nthreads=oracle_threads())
    # the status word reports non-finite rows exactly when the oracle has one
    assert status == (ERR_NONFINITE if (ref["n"] == ROW_NONFINITE).any() else 0), status
    low = ref["margin"] < MARGIN
    ok = ~low
    assert np.array_equal(g["n"][ok], ref["n"][ok]), (
        "n* differs on rows %s" % np.nonzero(g["n"] != ref["n"])[0][:10])
    assert np.array_equal(g["commit"][ok], ref["commit"][ok])
    assert np.array_equal(g["mask"][ok], ref["mask"][ok])
    assert np.array_equal(g["tokens"][ok], ref["tokens"][ok])
    # every row: the GPU decision is the rule applied to the GPU's own confidences
    conf, argmax = fd.fdllm_confidence(logits, torch.from_numpy(mask_np).cuda())
    rg = orc.select_from_conf(conf.cpu().numpy().astype(np.float64), argmax.cpu().numpy(),
                              mask_np, mode, param)
    same = rg["margin"] >= 1e-12
    assert np.array_equal(g["n"][same], rg["n"][same])
    assert np.array_equal(g["commit"][same], rg["commit"][same])
    assert np.array_equal(g["tokens"][same], rg["tokens"][same])
    # structural validity everywhere
    for b in range(B):
        m = int(mask_np[b].sum())
        if g["n"][b] >= 0:
            assert g["commit"][b].sum() == g["n"][b]
            assert (g["n"][b] == 0) == (m == 0)
            assert np.all(mask_np[b][g["commit"][b] == 1] == 1)
    return int(low.sum())
