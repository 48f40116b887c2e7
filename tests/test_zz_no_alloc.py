"""fdllm_select_static: the selection step on the library's fixed device scratch array.

Some callers cannot allocate device memory while they step: a serving process that
reserves all of its memory at start-up, or code running under an allocator that owns the
device.  fdllm_select_static serves them without any allocation.  These tests call it
through the C interface (ctypes, no Python wrapper in between) and require results equal to
fdllm_select's, bit for bit, on two calls in a row (the second call finds the first call's
leftovers in the shared array).  The file is named to be collected last.
"""
import ctypes

import numpy as np
import pytest
import torch

import fdllm_synth as syn

OK, ERR_WORKSPACE = 0, 5
STATIC_BYTES = 8 << 20


def _c_entry(path):
    lib = ctypes.CDLL(path)
    p, i, d = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
    lib.fdllm_select_static.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select_static.restype = i
    lib.fdllm_static_status.argtypes = [p]
    lib.fdllm_static_status.restype = i
    lib.fdllm_workspace_bytes.argtypes = [i, i, i, i]
    lib.fdllm_workspace_bytes.restype = ctypes.c_size_t
    return lib


@pytest.mark.gpu
@pytest.mark.parametrize("name,mode,param", [
    ("mixed_mask_b8_l32_bf16", 0, 0.75),
    ("target_ties_b16_l64_fp32", 1, 1.0),
    ("serving_b64_l32_bf16", 0, 1.0),
    ("target_b8_l32_fp16", 0, 0.75),
])
def test_static_scratch_matches_select_on_two_calls(fd, name, mode, param):
    lib = _c_entry(fd.library_path())
    w = syn.WORKLOADS[name]
    dtype = {"bf16": 0, "fp32": 1, "fp16": 2}[w.dtype]
    assert lib.fdllm_workspace_bytes(w.B, w.L, w.V, dtype) <= STATIC_BYTES
    logits = syn.make_logits(w, seed=77, device="cuda")
    mask_np = syn.make_mask(w, seed=77)

    ref_mask = torch.from_numpy(mask_np.copy()).cuda()
    ref = fd.fdllm_select(logits, ref_mask, param, mode)
    torch.cuda.synchronize()
    ref = [x.cpu().numpy() for x in ref] + [ref_mask.cpu().numpy()]

    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        mask = torch.from_numpy(mask_np.copy()).cuda()
        tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device="cuda")
        commit = torch.full((w.B, w.L), 7, dtype=torch.uint8, device="cuda")
        n = torch.full((w.B,), -9, dtype=torch.int32, device="cuda")
        st = lib.fdllm_select_static(logits.data_ptr(), dtype, w.B, w.L, w.V, mask.data_ptr(),
                                     param, mode, tok.data_ptr(), commit.data_ptr(),
                                     n.data_ptr(), stream)
        assert st == OK, "call %d returned %d" % (call, st)
        assert lib.fdllm_static_status(stream) == OK, "call %d: device error" % call
        torch.cuda.synchronize()
        got = [tok.cpu().numpy(), commit.cpu().numpy(), n.cpu().numpy(), mask.cpu().numpy()]
        for a, b, what in zip(ref, got, ("tokens", "commit", "n", "mask")):
            assert np.array_equal(a, b), "call %d: %s differs from fdllm_select" % (call, what)


def test_static_scratch_rejects_shapes_beyond_its_size(cuda_lib_path):
    """Checked on the host before any device work: fake, never-dereferenced addresses."""
    lib = _c_entry(cuda_lib_path)
    B, L, V, dtype = 64, 1024, 1 << 20, 1  # fp32 rows of 4 MiB: 32 MiB of unit partials
    assert lib.fdllm_workspace_bytes(B, L, V, dtype) > STATIC_BYTES
    a16 = 0x10000
    st = lib.fdllm_select_static(a16, dtype, B, L, V, a16, 1.0, 0, a16, a16, a16, None)
    assert st == ERR_WORKSPACE
