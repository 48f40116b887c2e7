"""The end-to-end input path: masked rows read by the GPU from pinned host memory."""
import numpy as np
import pytest
import torch

import fdllm_synth as syn

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["mixed_mask_b8_l32_bf16", "tie_groups_b16_l64_fp32"])
def test_gather_from_pinned_host_copies_masked_rows_only(fd, name):
    w = syn.WORKLOADS[name]
    x = syn.make_logits(w, seed=5, device="cpu", V=4096)
    h = x.pin_memory()
    mask_np = syn.make_mask(w, seed=5)
    mask = torch.from_numpy(mask_np).cuda()
    dst = torch.full(x.shape, 3.0, dtype=x.dtype, device="cuda")
    fd.fdllm_gather_masked_rows(h, mask, dst)
    torch.cuda.synchronize()
    got = dst.cpu()
    mk = torch.from_numpy(mask_np.astype(bool))
    assert torch.equal(got[mk], x[mk])
    assert (got[~mk] == 3.0).all()


def test_gather_from_device_and_rejects_pageable(fd):
    x = torch.randn(2, 8, 512, device="cuda").to(torch.bfloat16)
    mask = torch.tensor([[1, 0] * 4, [0, 1] * 4], dtype=torch.uint8, device="cuda")
    dst = fd.fdllm_gather_masked_rows(x, mask)
    torch.cuda.synchronize()
    mk = mask.bool()
    assert torch.equal(dst[mk], x[mk])
    with pytest.raises(ValueError):
        fd.fdllm_gather_masked_rows(x.cpu(), mask)


def test_host_select_through_pinned_path_matches_oracle(fd, orc):
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    x = syn.make_logits(w, seed=9, device="cpu", V=8192).pin_memory()
    mask_np = syn.make_mask(w, seed=9)
    h_mask = torch.from_numpy(mask_np.copy()).pin_memory()
    tok, commit, n = fd.fdllm_select(x, h_mask, 0.75, fd.PROFILE)
    ref = orc.select(syn.host_bits(x), mask_np, 0, 0.75)
    ok = ref["margin"] >= 1e-5
    assert np.array_equal(n.numpy()[ok], ref["n"][ok])
    assert np.array_equal(commit.numpy()[ok], ref["commit"][ok])
    assert np.array_equal(h_mask.numpy()[ok], ref["mask"][ok])
    c = ref["commit"].astype(bool) & ok[:, None]
    assert np.array_equal(tok.numpy()[c], ref["tokens"][c])
