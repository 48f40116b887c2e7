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


def _c_select_host(path):
    import ctypes
    lib = ctypes.CDLL(path)
    p, i, d = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
    lib.fdllm_select_host.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select_host.restype = i
    return lib


@pytest.mark.parametrize("where", ["pinned", "pageable", "device"])
@pytest.mark.parametrize("name,mode,param", [("mixed_mask_b8_l32_bf16", 0, 1.0),
                                             ("target_ties_b16_l64_fp32", 1, 1.0),
                                             ("target_b8_l32_fp16", 2, 0.9)])
def test_select_host_through_c_abi_equals_device_select(fd, orc, where, name, mode, param):
    """fdllm_select_host called through the C interface with host mask and outputs equals
    fdllm_select on device copies of the same inputs, bit for bit, wherever the logits
    live; positions it does not commit keep the caller's token values."""
    lib = _c_select_host(fd.library_path())
    w = syn.WORKLOADS[name]
    V = 4096 if where == "pageable" else w.V
    x = syn.make_logits(w, seed=21, device="cpu", V=V)
    mask_np = syn.make_mask(w, seed=21)
    dmask = torch.from_numpy(mask_np.copy()).cuda()
    ref = fd.fdllm_select(x.cuda(), dmask, param, mode)
    torch.cuda.synchronize()
    src = {"pinned": x.pin_memory(), "pageable": x, "device": x.cuda()}[where]
    dtype = {"bf16": 0, "fp32": 1, "fp16": 2}[w.dtype]
    h_mask = torch.from_numpy(mask_np.copy()).pin_memory()
    h_tok = torch.full((w.B, w.L), -7, dtype=torch.int32)
    h_commit = torch.full((w.B, w.L), 9, dtype=torch.uint8)
    h_n = torch.full((w.B,), -9, dtype=torch.int32)
    st = lib.fdllm_select_host(src.data_ptr(), dtype, w.B, w.L, V, h_mask.data_ptr(), param,
                               mode, h_tok.data_ptr(), h_commit.data_ptr(), h_n.data_ptr(),
                               torch.cuda.current_stream().cuda_stream)
    assert st == 0
    assert np.array_equal(h_n.numpy(), ref[2].cpu().numpy())
    assert np.array_equal(h_commit.numpy(), ref[1].cpu().numpy())
    assert np.array_equal(h_mask.numpy(), dmask.cpu().numpy())
    c = h_commit.numpy().astype(bool)
    assert np.array_equal(h_tok.numpy()[c], ref[0].cpu().numpy()[c])
    assert (h_tok.numpy()[~c] == -7).all()
    oref = orc.select(syn.host_bits(x), mask_np, mode, param)
    ok = oref["margin"] >= 1e-5
    assert np.array_equal(h_n.numpy()[ok], oref["n"][ok])


def test_host_select_reports_a_nonfinite_row(fd, orc):
    """Pinned host logits with a NaN in one masked position: through the host-buffer call
    that batch row reports FDLLM_ROW_NONFINITE and keeps its mask, the other rows match the
    oracle, and the library workspace's status word reads FDLLM_ERR_NONFINITE once."""
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    x = syn.make_logits(w, seed=19, device="cpu", V=4096)
    mask_np = np.ones((w.B, w.L), np.uint8)
    x[3, 7, 100] = float("nan")
    x = x.pin_memory()
    h_mask = torch.from_numpy(mask_np.copy()).pin_memory()
    tok, commit, n = fd.fdllm_select(x, h_mask, 0.75, fd.PROFILE)
    assert fd.fdllm_device_status() == 3  # FDLLM_ERR_NONFINITE
    assert fd.fdllm_device_status() == 0
    ref = orc.select(syn.host_bits(x), mask_np, 0, 0.75)
    assert n[3].item() == fd.ROW_NONFINITE == ref["n"][3]
    assert commit.numpy()[3].sum() == 0 and (h_mask.numpy()[3] == 1).all()
    ok = ref["margin"] >= 1e-5
    ok[3] = False
    assert ok.sum() >= 4
    assert np.array_equal(n.numpy()[ok], ref["n"][ok])
    assert np.array_equal(commit.numpy()[ok], ref["commit"][ok])


def test_c_program_selects_from_pinned_host_logits(fd, orc, cuda_lib_path, tmp_path):
    """The host-buffer step from a plain C program, as the README shows it: page-locked
    logits from cudaHostAlloc, one fdllm_select_host call, the results against the oracle."""
    import os
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    cuda = os.environ.get("CUDA_HOME", "/usr/local/cuda")
    if cc is None or not os.path.isdir(os.path.join(cuda, "include")):
        pytest.skip("no C compiler or CUDA headers")
    w = syn.WORKLOADS["target_b8_l32_bf16"]
    V = 4096
    x = syn.make_logits(w, seed=23, device="cpu", V=V)
    bits = syn.host_bits(x)  # uint16 bf16 patterns, [B, L, V]
    mask_np = syn.make_mask(w, seed=23)
    (tmp_path / "logits.bin").write_bytes(np.ascontiguousarray(bits).tobytes())
    (tmp_path / "mask.bin").write_bytes(mask_np.tobytes())
    src = tmp_path / "step.c"
    src.write_text(r'''
#include <stdio.h>
#include <stdlib.h>
#include <string.h>
#include <cuda_runtime.h>
#include "fdllm.h"
int main(int argc, char **argv)
{
    const int B = atoi(argv[1]), L = atoi(argv[2]), V = atoi(argv[3]);
    const size_t n = (size_t)B * L * V;
    uint16_t *logits = NULL;
    if (cudaHostAlloc((void **)&logits, n * 2, cudaHostAllocDefault) != cudaSuccess)
        return 2;
    FILE *f = fopen(argv[4], "rb");
    if (!f || fread(logits, 2, n, f) != n)
        return 3;
    fclose(f);
    uint8_t *mask = malloc((size_t)B * L), *commit = malloc((size_t)B * L);
    int32_t *tokens = malloc((size_t)B * L * 4), *nstar = malloc((size_t)B * 4);
    f = fopen(argv[5], "rb");
    if (!f || fread(mask, 1, (size_t)B * L, f) != (size_t)B * L)
        return 4;
    fclose(f);
    for (int i = 0; i < B * L; ++i)
        tokens[i] = -1;
    fdllm_status st = fdllm_select_host(logits, FDLLM_BF16, B, L, V, mask, 0.75, FDLLM_PROFILE,
                                        tokens, commit, nstar, 0);
    if (st != FDLLM_OK) {
        fprintf(stderr, "%s\n", fdllm_status_string(st));
        return 5;
    }
    if (fdllm_device_status(0) != FDLLM_OK)
        return 6;
    f = fopen(argv[6], "wb");
    fwrite(tokens, 4, (size_t)B * L, f);
    fwrite(commit, 1, (size_t)B * L, f);
    fwrite(nstar, 4, (size_t)B, f);
    fwrite(mask, 1, (size_t)B * L, f);
    fclose(f);
    cudaFreeHost(logits);
    return 0;
}
''')
    exe = tmp_path / "step"
    libdir = os.path.dirname(cuda_lib_path)
    cudalib = os.path.join(cuda, "lib64")
    include = os.path.join(os.path.dirname(libdir), "include")
    r = subprocess.run([cc, "-std=c99", "-O2", "-I", include,
                        "-I", os.path.join(cuda, "include"), str(src), "-o", str(exe),
                        "-L", libdir, "-lfdllm", "-L", cudalib, "-lcudart",
                        "-Wl,-rpath," + libdir, "-Wl,-rpath," + cudalib],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = tmp_path / "out.bin"
    p = subprocess.run([str(exe), str(w.B), str(w.L), str(V), str(tmp_path / "logits.bin"),
                        str(tmp_path / "mask.bin"), str(out)], capture_output=True, text=True)
    assert p.returncode == 0, (p.returncode, p.stderr)
    raw = out.read_bytes()
    BL = w.B * w.L
    tok = np.frombuffer(raw[:4 * BL], np.int32).reshape(w.B, w.L)
    commit = np.frombuffer(raw[4 * BL:5 * BL], np.uint8).reshape(w.B, w.L)
    nst = np.frombuffer(raw[5 * BL:5 * BL + 4 * w.B], np.int32)
    mask_out = np.frombuffer(raw[5 * BL + 4 * w.B:], np.uint8).reshape(w.B, w.L)
    ref = orc.select(bits, mask_np, 0, 0.75)
    ok = ref["margin"] >= 1e-5
    assert ok.sum() >= w.B // 2
    assert np.array_equal(nst[ok], ref["n"][ok])
    assert np.array_equal(commit[ok], ref["commit"][ok])
    assert np.array_equal(mask_out[ok], ref["mask"][ok])
    c = ref["commit"].astype(bool) & ok[:, None]
    assert np.array_equal(tok[c], ref["tokens"][c])
