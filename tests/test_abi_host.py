"""The C interface on the host (no GPU): the library builds, loads, exports every function
include/fdllm.h declares, and rejects bad arguments before touching the device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fdllm.h")

OK, ERR_ARG, ERR_ALIGN, ERR_WORKSPACE = 0, 1, 2, 5


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fdllm_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib(cuda_lib_path):
    lib = ctypes.CDLL(cuda_lib_path)
    p, i, d, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_double, ctypes.c_size_t
    lib.fdllm_select.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_select_ws.argtypes = [p, i, i, i, i, p, d, i, p, p, p, p, sz, p]
    lib.fdllm_confidence.argtypes = [p, i, i, i, i, p, p, p, p]
    lib.fdllm_select_from_conf.argtypes = [p, p, i, i, p, d, i, p, p, p, p]
    lib.fdllm_workspace_bytes.argtypes = [i, i, i, i]
    lib.fdllm_workspace_bytes.restype = sz
    lib.fdllm_status_string.restype = ctypes.c_char_p
    return lib


def test_header_declares_the_interface():
    names = declared_functions()
    for must in ("fdllm_select", "fdllm_select_ws", "fdllm_workspace_bytes",
                 "fdllm_confidence", "fdllm_select_from_conf"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_version_and_status_strings(lib):
    assert lib.fdllm_version() >= 100
    for code in range(0, 7):
        assert lib.fdllm_status_string(code)


def test_workspace_bytes(lib):
    a = lib.fdllm_workspace_bytes(64, 32, 126464, 0)
    b = lib.fdllm_workspace_bytes(16, 1024, 126464, 1)
    assert a % 256 == 0 and b % 256 == 0 and b > a > 8 * 64 * 32
    assert lib.fdllm_workspace_bytes(0, 32, 126464, 0) == 0


# Fake device addresses: the argument checks reject these calls before any CUDA call.
A16 = 0x10000
A2 = 0x10002


@pytest.mark.parametrize("args,want", [
    ((A16, 0, 0, 32, 1024), ERR_ARG),          # B = 0
    ((A16, 0, 2, 0, 1024), ERR_ARG),           # L = 0
    ((A16, 0, 2, 1025, 1024), ERR_ARG),        # L > 1024
    ((A16, 0, 128, 1024, 1024), ERR_ARG),      # B * L > 65536
    ((A16, 0, 2, 32, 0), ERR_ARG),             # V = 0
    ((A16, 3, 2, 32, 1024), ERR_ARG),          # unknown dtype
    ((None, 0, 2, 32, 1024), ERR_ARG),         # null logits
    ((A2, 0, 2, 32, 1024), ERR_ALIGN),         # logits not 16-byte aligned
    ((A16, 0, 2, 32, 1001), ERR_ALIGN),        # V * 2 not a multiple of 16
    ((A16, 1, 2, 32, 1002), ERR_ALIGN),        # V * 4 not a multiple of 16
    ((A16, 2, 2, 32, 1001), ERR_ALIGN),        # fp16: V * 2 not a multiple of 16
])
def test_select_rejects_bad_shapes(lib, args, want):
    logits, dtype, B, L, V = args
    st = lib.fdllm_select(logits, dtype, B, L, V, A16, 1.0, 0, A16, A16, A16, None)
    assert st == want


@pytest.mark.parametrize("args,want", [
    ((A16, 0, 0, 32, 1024), ERR_ARG),          # B = 0
    ((A16, 0, 2, 1025, 1024), ERR_ARG),        # L > 1024
    ((None, 0, 2, 32, 1024), ERR_ARG),         # null logits
    ((A2, 0, 2, 32, 1024), ERR_ALIGN),         # logits not 16-byte aligned
    ((A16, 0, 2, 32, 1001), ERR_ALIGN),        # V * 2 not a multiple of 16
])
def test_select_host_rejects_bad_arguments_before_any_copy(lib, args, want):
    logits, dtype, B, L, V = args
    lib.fdllm_select_host.argtypes = lib.fdllm_select.argtypes
    assert lib.fdllm_select_host(logits, dtype, B, L, V, A16, 1.0, 0, A16, A16, A16,
                                 None) == want
    assert lib.fdllm_select_host(A16, 0, 2, 32, 1024, None, 1.0, 0, A16, A16, A16,
                                 None) == ERR_ARG
    assert lib.fdllm_select_host(A16, 0, 2, 32, 1024, A16, 1.0, 5, A16, A16, A16,
                                 None) == ERR_ARG


def test_select_rejects_bad_mode_param_and_outputs(lib):
    call = lambda mode, param, out=A16, mask=A16: lib.fdllm_select(
        A16, 0, 2, 32, 1024, mask, param, mode, out, A16, A16, None)
    assert call(3, 1.0) == ERR_ARG
    assert call(-1, 1.0) == ERR_ARG
    assert call(0, float("nan")) == ERR_ARG
    assert call(0, float("inf")) == ERR_ARG
    assert call(0, 1.0, out=None) == ERR_ARG
    assert call(0, 1.0, mask=None) == ERR_ARG


def test_select_ws_rejects_small_or_misaligned_workspace(lib):
    need = lib.fdllm_workspace_bytes(2, 32, 1024, 0)
    f = lambda ws, n: lib.fdllm_select_ws(A16, 0, 2, 32, 1024, A16, 1.0, 0, A16, A16, A16, ws,
                                          n, None)
    assert f(None, need) == ERR_WORKSPACE
    assert f(A16 + 16, need) == ERR_WORKSPACE
    assert f(A16, need - 1) == ERR_WORKSPACE


def test_confidence_and_select_from_conf_reject(lib):
    assert lib.fdllm_confidence(A2, 0, 2, 32, 1024, A16, A16, A16, None) == ERR_ALIGN
    assert lib.fdllm_confidence(A16, 0, 2, 32, 1024, None, A16, A16, None) == ERR_ARG
    assert lib.fdllm_select_from_conf(A16, A16, 2, 2000, A16, 1.0, 0, A16, A16, A16,
                                      None) == ERR_ARG
    assert lib.fdllm_select_from_conf(None, A16, 2, 32, A16, 1.0, 0, A16, A16, A16,
                                      None) == ERR_ARG


def test_select_robust_rejects(lib):
    p, i, d = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
    lib.fdllm_select_robust.argtypes = [p, i, i, i, i, p, d, d, p, p, p, p, p]
    f = lambda eta, B=2, logits=A16: lib.fdllm_select_robust(logits, 0, B, 32, 1024, A16, 1.0,
                                                             eta, None, A16, A16, A16, None)
    assert f(float("nan")) == ERR_ARG
    assert f(float("inf")) == ERR_ARG
    assert f(-0.05) == ERR_ARG  # App. C's allowance is >= 0
    assert f(0.1, B=0) == ERR_ARG
    assert f(0.1, logits=A2) == ERR_ALIGN


def test_decode_loop_rejects_before_any_device_call(lib):
    p, i, d = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
    fwd_t = ctypes.CFUNCTYPE(i, p, p, p, p, p)
    calls = []
    fwd = fwd_t(lambda *a: calls.append(a) or 0)
    lib.fdllm_decode_loop.argtypes = [i, i, i, i, i, d, i, fwd_t, p, p, p, p, i,
                                      ctypes.POINTER(i), p]
    steps = ctypes.c_int(-5)

    def f(B=2, gen=64, Lb=32, mode=0, forward=fwd, logits=A16, max_steps=100):
        return lib.fdllm_decode_loop(B, gen, Lb, 1024, 0, 1.0, mode, forward, None, logits,
                                     A16, A16, max_steps, ctypes.byref(steps), None)
    assert f(gen=48) == ERR_ARG                   # gen_len not a multiple of block_len
    assert f(gen=16) == ERR_ARG                   # gen_len < block_len
    assert f(Lb=2048, gen=4096) == ERR_ARG        # block_len > 1024
    assert f(B=0) == ERR_ARG
    assert f(mode=3) == ERR_ARG                   # the robust rule is not a loop mode
    assert f(max_steps=0) == ERR_ARG
    assert f(forward=fwd_t()) == ERR_ARG          # null forward pass
    assert f(logits=None) == ERR_ARG
    assert not calls and steps.value == -5


def test_lmhead_rejects_before_any_device_call(lib):
    p, i, d = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
    lib.fdllm_lmhead_select.argtypes = [p, p, i, i, i, i, p, d, i, p, p, p, p]
    lib.fdllm_lmhead_logits.argtypes = [p, p, i, i, i, i, p, p, p]

    def f(hidden=A16, w=A16, B=2, L=32, H=4096, V=126464, mask=A16, mode=0, param=1.0):
        return lib.fdllm_lmhead_select(hidden, w, B, L, H, V, mask, param, mode, A16, A16, A16,
                                       None)
    assert f(H=4100) == ERR_ALIGN          # rows of H bf16 not a multiple of 16 bytes
    assert f(hidden=A2) == ERR_ALIGN
    assert f(w=A2) == ERR_ALIGN
    assert f(H=0) == ERR_ARG
    assert f(V=0) == ERR_ARG
    assert f(L=1025) == ERR_ARG
    assert f(B=65, L=1024) == ERR_ARG      # B * L > 65536
    assert f(mask=None) == ERR_ARG
    assert f(mode=3) == ERR_ARG
    assert f(param=float("nan")) == ERR_ARG
    assert lib.fdllm_lmhead_logits(A16, A16, 2, 32, 64, 1000, A16, None, None) == ERR_ARG


def test_gather_masked_rows_rejects(lib):
    p, i = ctypes.c_void_p, ctypes.c_int
    lib.fdllm_gather_masked_rows.argtypes = [p, p, i, i, i, i, p, p]
    f = lambda src=A16, dst=A16, dtype=0, B=2, L=32, V=1024, mask=A16: \
        lib.fdllm_gather_masked_rows(src, dst, dtype, B, L, V, mask, None)
    assert f(src=None) == ERR_ARG
    assert f(mask=None) == ERR_ARG
    assert f(dtype=3) == ERR_ARG
    assert f(L=1025) == ERR_ARG
    assert f(V=1001) == ERR_ALIGN
    assert f(src=A2) == ERR_ALIGN
    assert f(dst=A2) == ERR_ALIGN


def test_vocab_reduce_rejects_before_any_device_call(lib):
    p, i = ctypes.c_void_p, ctypes.c_int
    lib.fdllm_vocab_reduce.argtypes = [p, i, i, i, i, p, p]
    A16 = 1 << 20  # a 16-byte aligned (never dereferenced) address
    assert lib.fdllm_vocab_reduce(A16, 0, 0, 32, 1024, A16, None) == ERR_ARG       # B < 1
    assert lib.fdllm_vocab_reduce(A16, 0, 2, 2000, 1024, A16, None) == ERR_ARG     # L > max
    assert lib.fdllm_vocab_reduce(A16, 0, 2, 32, 1024, None, None) == ERR_ARG      # no mask
    assert lib.fdllm_vocab_reduce(A16, 3, 2, 32, 1024, A16, None) == ERR_ARG       # dtype
    assert lib.fdllm_vocab_reduce(A16 + 2, 0, 2, 32, 1024, A16, None) == ERR_ALIGN  # base
    assert lib.fdllm_vocab_reduce(A16, 0, 2, 32, 1001, A16, None) == ERR_ALIGN     # V * 2


def test_profile_terms_rejects_before_any_device_call(lib):
    p, i, d = ctypes.c_void_p, ctypes.c_int, ctypes.c_double
    lib.fdllm_profile_terms.argtypes = [p, p, i, i, d, p, p, p, p, p, p]
    A16 = 1 << 20
    call = lambda B, L, delta, conf=A16, mask=A16: lib.fdllm_profile_terms(
        conf, mask, B, L, delta, None, None, None, None, None, None)
    assert call(0, 32, 0.0) == ERR_ARG
    assert call(2, 0, 0.0) == ERR_ARG
    assert call(2, 2000, 0.0) == ERR_ARG
    assert call(2, 32, 0.0, conf=None) == ERR_ARG
    assert call(2, 32, 0.0, mask=None) == ERR_ARG
    assert call(2, 32, float("nan")) == ERR_ARG
    assert call(2, 32, float("inf")) == ERR_ARG


def test_c_program_builds_against_the_header_and_links(cuda_lib_path, tmp_path):
    """A plain C99 program includes include/fdllm.h with -pedantic -Werror, takes the address
    of every declared function (so each must be exported with C linkage), links against the
    library and calls its host-only entry points."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    names = declared_functions()
    src = tmp_path / "abi.c"
    src.write_text(
        "#include <stdio.h>\n#include \"fdllm.h\"\n"
        "typedef void (*any_fn)(void);\n"
        "static any_fn table[] = {\n"
        + "".join("    (any_fn)%s,\n" % n for n in names)
        + "};\n"
        "int main(void)\n{\n"
        "    size_t ws = fdllm_workspace_bytes(64, 32, 126464, FDLLM_BF16);\n"
        "    printf(\"%d %zu %d %s\\n\", fdllm_version(), ws, (int)(sizeof table / sizeof *table),\n"
        "           fdllm_status_string(FDLLM_ERR_NONFINITE));\n"
        "    return fdllm_select(0, FDLLM_BF16, 1, 1, 8, 0, 0.75, FDLLM_PROFILE, 0, 0, 0, 0) ==\n"
        "               FDLLM_ERR_ARG ? 0 : 1;\n"
        "}\n")
    exe = tmp_path / "abi"
    libdir = os.path.dirname(cuda_lib_path)
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror",
                        "-Wno-cast-function-type", "-I", os.path.join(ROOT, "include"),
                        str(src), "-o", str(exe), "-L", libdir, "-lfdllm",
                        "-Wl,-rpath," + libdir], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out.stderr
    version, ws, count, text = out.stdout.split(" ", 3)
    assert int(version) >= 100 and int(ws) > 0 and int(count) == len(names)
    assert "non-finite" in text
