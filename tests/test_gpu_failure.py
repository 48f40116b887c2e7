"""Failure detection on the GPU without a fault: a kernel wait that nothing completes must
run out after its limit, be reported as a device error, and leave the device usable."""
import time

import numpy as np
import pytest
import torch

import fdllm_synth as syn

pytestmark = pytest.mark.gpu
ERR_NONFINITE, ERR_DEVICE = 3, 6


def test_bounded_wait_runs_out_and_device_stays_usable(fd, orc):
    t0 = time.perf_counter()
    assert fd.fdllm_check_bounded_wait(0.02) == ERR_DEVICE
    elapsed = time.perf_counter() - t0
    assert 0.015 <= elapsed < 2.0
    assert fd.fdllm_check_bounded_wait(0.02) == ERR_DEVICE  # repeatable
    # the context is intact: a normal step still runs and its status is clean
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=11, device="cuda")
    mask_np = syn.make_mask(w, seed=11)
    tok, commit, n = fd.fdllm_select(logits, torch.from_numpy(mask_np.copy()).cuda(), 0.75,
                                     fd.PROFILE)
    torch.cuda.synchronize()
    assert fd.fdllm_device_status() == 0
    ref = orc.select(syn.host_bits(logits), mask_np, 0, 0.75)
    ok = ref["margin"] >= 1e-5
    assert np.array_equal(n.cpu().numpy()[ok], ref["n"][ok])


def test_bounded_wait_rejects_bad_limits(fd):
    assert fd.fdllm_check_bounded_wait(0.0) == 1
    assert fd.fdllm_check_bounded_wait(60.0) == 1


def test_clearing_an_error_resets_the_work_counter(fd, orc):
    """A launch that gave up a wait may stop fetching from its work queue before its last
    unit and so leave the counter mid-queue; the status read that reports the error clears
    both words, so that the next call on the workspace processes every unit.  The left-over
    state is written into a caller workspace from the host: no kernel is made to fail."""
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=13, device="cuda")
    mask_np = syn.make_mask(w, seed=13)
    ws = torch.zeros(fd.fdllm_workspace_bytes(w.B, w.L, w.V, fd.BF16), dtype=torch.uint8,
                     device="cuda")
    header = ws[:8].view(torch.int32)
    header.copy_(torch.tensor([1, 37], dtype=torch.int32))
    assert fd.fdllm_workspace_status(ws) == ERR_DEVICE
    assert header.cpu().tolist() == [0, 0]
    assert fd.fdllm_workspace_status(ws) == 0
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_select_ws(logits, mask, 0.75, fd.PROFILE, ws)
    torch.cuda.synchronize()
    assert fd.fdllm_workspace_status(ws) == 0 and header.cpu().tolist() == [0, 0]
    ref = orc.select(syn.host_bits(logits), mask_np, 0, 0.75)
    ok = ref["margin"] >= 1e-5
    assert ok.sum() >= w.B // 2
    assert np.array_equal(n.cpu().numpy()[ok], ref["n"][ok])
    assert np.array_equal(commit.cpu().numpy()[ok], ref["commit"][ok])


def test_status_bits_and_their_precedence(fd):
    """The status word's two bits, written into a caller workspace from the host: the
    non-finite bit alone reads as FDLLM_ERR_NONFINITE, together with the timeout bit as
    FDLLM_ERR_DEVICE (a failed step outranks a bad row); each read clears the header."""
    ws = torch.zeros(fd.fdllm_workspace_bytes(1, 1, 8, fd.BF16), dtype=torch.uint8,
                     device="cuda")
    header = ws[:8].view(torch.int32)
    for word, expect in ((2, ERR_NONFINITE), (3, ERR_DEVICE), (1, ERR_DEVICE), (0, 0)):
        header.copy_(torch.tensor([word, 0], dtype=torch.int32))
        assert fd.fdllm_workspace_status(ws) == expect, word
        assert header.cpu().tolist() == [0, 0]


def test_nonfinite_bit_does_not_fail_later_steps(fd, orc):
    """A set non-finite bit (a bad row in an earlier step, not yet read) leaves the next
    steps' decisions alone: only the timeout bit turns rows into device errors."""
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=17, device="cuda")
    mask_np = syn.make_mask(w, seed=17)
    ws = torch.zeros(fd.fdllm_workspace_bytes(w.B, w.L, w.V, fd.BF16), dtype=torch.uint8,
                     device="cuda")
    ws[:4].view(torch.int32).fill_(2)
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_select_ws(logits, mask, 0.75, fd.PROFILE, ws)
    assert fd.fdllm_workspace_status(ws) == ERR_NONFINITE
    ref = orc.select(syn.host_bits(logits), mask_np, 0, 0.75)
    ok = ref["margin"] >= 1e-5
    assert (n.cpu().numpy() >= 0).all()
    assert np.array_equal(n.cpu().numpy()[ok], ref["n"][ok])
    assert np.array_equal(commit.cpu().numpy()[ok], ref["commit"][ok])
