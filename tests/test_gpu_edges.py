"""Edge cases of the CUDA path against the oracle: empty and single-position rows, maximal
L and row counts, the smallest vocabulary, -inf and non-finite logits, all-equal logits,
maxima tied across CTA boundaries and in the ragged tail."""
import numpy as np
import pytest
import torch

import fdllm_synth as syn
from gpu_util import ERR_NONFINITE, check_confidence, check_select

pytestmark = pytest.mark.gpu
PROFILE, FACTOR, THRESHOLD = 0, 1, 2


def _bf16(x: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(x).to(torch.bfloat16).cuda()


def test_all_rows_unmasked(fd, orc):
    logits = torch.randn(4, 16, 1024, device="cuda", dtype=torch.bfloat16)
    mask = torch.zeros(4, 16, dtype=torch.uint8, device="cuda")
    tok, commit, n = fd.fdllm_select(logits, mask, 0.75, PROFILE)
    assert n.cpu().tolist() == [0, 0, 0, 0]
    assert commit.sum().item() == 0 and mask.sum().item() == 0
    assert torch.all(tok == -1)


@pytest.mark.parametrize("L", [1, 2, 31, 32, 33, 1024])
def test_row_lengths(fd, orc, L):
    w = syn.Workload("len", 2, L, 2048, "bf16", 1.0, "target", 0.3, 4.0)
    logits = syn.make_logits(w, seed=L, device="cuda")
    mask_np = np.ones((2, L), np.uint8)
    mask_np[1, ::3] = 0
    for mode, p in ((PROFILE, 0.75), (FACTOR, 0.75), (THRESHOLD, 0.9)):
        check_select(fd, orc, logits, mask_np, mode, p)


def test_max_rows_and_min_vocab(fd, orc):
    """B * L = 65536 rows of V = 8 bf16 (one 16-byte vector per row)."""
    B, L, V = 64, 1024, 8
    x = np.random.default_rng(1).normal(0, 2, (B, L, V)).astype(np.float32)
    logits = _bf16(x)
    mask_np = (np.random.default_rng(2).random((B, L)) < 0.5).astype(np.uint8)
    check_confidence(fd, orc, logits, mask_np)
    check_select(fd, orc, logits, mask_np, PROFILE, 0.75)


def test_fp32_min_vocab(fd, orc):
    x = np.random.default_rng(3).normal(0, 2, (3, 40, 4)).astype(np.float32)
    check_confidence(fd, orc, torch.from_numpy(x).cuda(), np.ones((3, 40), np.uint8))


def test_equal_logits_give_uniform_confidence(fd):
    V = 126464
    logits = torch.full((1, 3, V), 0.5, device="cuda", dtype=torch.bfloat16)
    conf, tok = fd.fdllm_confidence(logits, torch.ones(1, 3, dtype=torch.uint8, device="cuda"))
    assert torch.all(tok == 0)
    assert torch.allclose(conf.double(), torch.full_like(conf.double(), 1.0 / V), rtol=1e-5,
                          atol=0)


def test_nonfinite_rows(fd, orc):
    V = 4096
    x = np.random.default_rng(4).normal(0, 1, (3, 4, V)).astype(np.float32)
    x[0, 1, 100] = np.nan       # row 0 invalid
    x[1, 2, :] = -np.inf        # row 1 invalid (max is -inf)
    x[2, 0, ::2] = -np.inf      # row 2 fine: -inf entries contribute nothing
    x[2, 3, 4000] = np.inf      # ... but +inf makes row 2 invalid too
    logits = torch.from_numpy(x).cuda()
    mask_np = np.ones((3, 4), np.uint8)
    check_confidence(fd, orc, logits, mask_np)
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_select(logits, mask, 0.75, PROFILE)
    assert n.cpu().tolist() == [fd.ROW_NONFINITE] * 3
    assert commit.sum().item() == 0 and mask.sum().item() == 12
    # the workspace's status word says so too, and reading it clears it
    assert fd.fdllm_device_status() == ERR_NONFINITE
    assert fd.fdllm_device_status() == 0
    # -inf entries alone are fine
    x[2, 3, 4000] = 0.0
    x[0, 1, 100] = 0.0
    x[1, 2, :] = 0.0
    logits = torch.from_numpy(x).cuda()
    check_confidence(fd, orc, logits, mask_np)
    check_select(fd, orc, logits, mask_np, PROFILE, 0.75)


def test_nonfinite_rows_reported_by_every_status_word(fd):
    """A NaN in one masked row: the caller workspace's and the static array's status words
    report FDLLM_ERR_NONFINITE after the step (the other row still commits), and a clean
    step afterwards reads FDLLM_OK."""
    B, L, V = 2, 8, 4096
    x = np.random.default_rng(6).normal(0, 1, (B, L, V)).astype(np.float32)
    x[1, 5, 7] = np.nan
    mask_np = np.ones((B, L), np.uint8)
    ws = torch.zeros(fd.fdllm_workspace_bytes(B, L, V, fd.FP32), dtype=torch.uint8,
                     device="cuda")
    for bad in (True, False):
        logits = torch.from_numpy(x).cuda()
        expect = ERR_NONFINITE if bad else 0
        _, _, n = fd.fdllm_select_ws(logits, torch.from_numpy(mask_np.copy()).cuda(), 0.75,
                                     PROFILE, ws)
        assert fd.fdllm_workspace_status(ws) == expect
        assert n[0].item() >= 1 and (n[1].item() == fd.ROW_NONFINITE) == bad
        _, _, n = fd.fdllm_select_static(logits, torch.from_numpy(mask_np.copy()).cuda(), 0.75,
                                         PROFILE)
        assert fd.fdllm_static_status() == expect
        assert n[0].item() >= 1 and (n[1].item() == fd.ROW_NONFINITE) == bad
        assert fd.fdllm_static_status() == 0
        x[1, 5, 7] = 0.0


def test_decode_loop_stops_on_a_nonfinite_row(fd):
    """A forward pass that leaves a NaN in a masked row: that row commits nothing, so the
    loop ends after the step with FDLLM_ERR_NONFINITE instead of running to max_steps
    (which would read as FDLLM_ERR_DEVICE)."""
    B, gen, Lb, V = 2, 64, 32, 4096
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")

    def forward(state, mask, out, stream):
        syn.synth_block_logits_gpu(out, mask, B, Lb, V, 3, step_ptr=state, peak_max=16.0,
                                   stream_ptr=stream)
        with torch.cuda.stream(torch.cuda.ExternalStream(stream)):
            logits[1, 4, 9].fill_(float("nan"))

    with pytest.raises(fd.FdllmError) as err:
        fd.fdllm_decode_loop(forward, logits, gen, 1.0, PROFILE, max_steps=10 * gen)
    assert err.value.status == ERR_NONFINITE
    assert fd.fdllm_device_status() == ERR_NONFINITE
    assert fd.fdllm_device_status() == 0


@pytest.mark.parametrize("dtype", ["bf16", "fp16", "fp32"])
def test_large_magnitude_logits(fd, orc, dtype):
    """Logits far from 0: a row shifted by a large constant (softmax is shift-invariant), rows
    filled with the type's most negative finite value (a common masking value), the largest
    finite value tied twice, and (fp32, bf16) maxima on both sides of 2^30, where the sum
    switches from the scaled FMA form to counting the maxima, up to 1e30 and beyond."""
    np_t = {"bf16": np.float32, "fp16": np.float16, "fp32": np.float32}[dtype]
    info = {"bf16": torch.finfo(torch.bfloat16), "fp16": torch.finfo(torch.float16),
            "fp32": torch.finfo(torch.float32)}[dtype]
    lo, hi = float(info.min), float(info.max)
    V = 126464 if dtype != "fp16" else 8192
    rng = np.random.default_rng(12)
    x = rng.normal(0.0, 1.0, (2, 8, V))
    x[0, 0] = x[0, 0] * 0.05 + (3.0e4 if dtype == "fp32" else 600.0)   # shifted, tight
    x[0, 1] = lo                                                       # c = 1 / V
    x[0, 2] = lo
    x[0, 2, [5, V // 2, V - 1]] = rng.normal(0.0, 1.0, 3)              # a few ordinary values
    x[0, 3, [7, V - 9]] = hi                                           # tied largest value
    x[0, 4] = x[0, 4] - (3.0e4 if dtype == "fp32" else 600.0)          # shifted down
    x[0, 5, V // 3] = hi / 2
    x[0, 6] = -x[0, 6] ** 2 * 1e3                                      # wide negative spread
    x[0, 6, 11] = 0.5
    x[0, 7] = lo / 4
    x[0, 7, [1, V // 3 + 1]] = lo / 8                                  # tied, all far below 0
    if dtype != "fp16":
        b = 2.0 ** 30
        below = float(np.nextafter(np.float32(b), np.float32(0)))      # b - 64
        x[1, 0, 3] = b                                                 # exactly the switch
        x[1, 0, 9] = below                                             # e^-64 below it
        x[1, 1] = -b
        x[1, 1, ::7] = lo
        x[1, 2, [0, 4000]] = below                                     # tied, scaled form
        x[1, 3] = rng.normal(0.0, 1.0, V) * 1e30
        x[1, 4] = -2.0 * b
        x[1, 4, [17, V - 5]] = -b                                      # max -2^30, tied
        x[1, 5, ::1000] = hi
        x[1, 6] = x[1, 6] * 4.0 + 1e8                                  # rounding residual 8
        x[1, 7] = x[1, 7] * 2.0 ** 24 + 2.0 ** 29                      # residual up to 32
    else:
        x[1, :4] = x[1, :4] * 8.0 + 60000.0 * np.sign(x[1, :4])
    x = np.clip(x, lo, hi).astype(np_t)
    logits = _bf16(x) if dtype == "bf16" else torch.from_numpy(x).cuda()
    mask_np = np.ones((2, 8), np.uint8)
    conf, tok, rc, rt = check_confidence(fd, orc, logits, mask_np)
    assert abs(conf[0, 1] * V - 1.0) <= 1e-5 and tok[0, 1] == 0
    assert abs(conf[0, 3] - 0.5) <= 1e-6 and tok[0, 3] == 7
    check_select(fd, orc, logits, mask_np, PROFILE, 0.75)


def test_argmax_ties_across_chunks_and_ctas(fd, orc):
    """Equal maxima far apart in a row (different chunks and, at this size, different CTAs),
    and maxima in the last, ragged chunk: the lowest index must win."""
    V = 126464
    rng = np.random.default_rng(5)
    x = rng.normal(0, 1, (2, 6, V)).astype(np.float32)
    x[0, 0, [V - 1, 70000, 9000]] = 20.0
    x[0, 1, [V - 1]] = 20.0
    x[0, 2, [0, V - 1]] = 20.0
    x[0, 3, [8191, 8192, 16384]] = 20.0
    x[0, 4, [V - 8, V - 7]] = 20.0
    x[0, 5, :] = 3.0
    x[1] = x[0, ::-1]
    for dt in ("bf16", "fp32"):
        logits = _bf16(x) if dt == "bf16" else torch.from_numpy(x).cuda()
        _, g_tok, _, _ = check_confidence(fd, orc, logits, np.ones((2, 6), np.uint8))
        assert g_tok[0, :5].tolist() == [9000, V - 1, 0, 8191, V - 8]
        assert g_tok[0, 5] == 0


def test_large_rows_many_ctas_fp32(fd, orc):
    """Few long rows: every row spans many CTAs, so the split-row combination decides."""
    w = syn.Workload("long", 1, 3, 1 << 20, "fp32", 1.0, "target", 0.3, 4.0)
    logits = syn.make_logits(w, seed=6, device="cuda")
    check_confidence(fd, orc, logits, np.ones((1, 3), np.uint8))


def test_bad_arguments_raise(fd):
    logits = torch.randn(2, 4, 1000, device="cuda", dtype=torch.bfloat16)
    mask = torch.ones(2, 4, dtype=torch.uint8, device="cuda")
    with pytest.raises(fd.FdllmError) as e:
        fd.fdllm_select(logits, mask, 1.0, 7)
    assert e.value.status == 1
    with pytest.raises(fd.FdllmError) as e:
        fd.fdllm_select(logits, mask, float("nan"), 0)
    assert e.value.status == 1


def test_misaligned_logits_rejected(fd):
    base = torch.randn(2 * 4 * 1000 + 8, device="cuda", dtype=torch.bfloat16)
    logits = base[1:1 + 2 * 4 * 1000].view(2, 4, 1000)
    mask = torch.ones(2, 4, dtype=torch.uint8, device="cuda")
    with pytest.raises(fd.FdllmError) as e:
        fd.fdllm_select(logits, mask, 1.0, PROFILE)
    assert e.value.status == 2
    with pytest.raises(fd.FdllmError) as e:
        fd.fdllm_select(torch.randn(2, 4, 999, device="cuda", dtype=torch.bfloat16), mask, 1.0,
                        PROFILE)
    assert e.value.status == 2


@pytest.mark.parametrize("first_masked", [2048, 60000, 65500])
def test_masked_rows_only_far_into_the_batch(fd, orc, first_masked):
    """Every masked row lies beyond the first 2048 rows (beyond the producer's own scan for
    its first unit): the units are then found through the CTA's compaction; results match."""
    B, L, V = 2048, 32, 1024
    w = syn.Workload("far", B, L, V, "bf16", 1.0, "target", 0.3, 4.0)
    logits = syn.make_logits(w, seed=first_masked, device="cuda")
    mask = np.zeros((B, L), np.uint8)
    flat = mask.reshape(-1)
    rng = np.random.default_rng(first_masked)
    rows = rng.choice(np.arange(first_masked, B * L), size=min(300, B * L - first_masked),
                      replace=False)
    flat[rows] = 1
    check_confidence(fd, orc, logits, mask)
    assert check_select(fd, orc, logits, mask, 0, 0.75) <= 2


@pytest.mark.parametrize("dtype,L", [("bf16", 8), ("fp32", 96)])
def test_argmax_ties_on_unit_boundaries(fd, orc, dtype, L):
    """Equal maxima on both sides of a unit boundary, under both unit plans: a small step
    (8 bf16 rows, 2 MB: 64 KB units of 32768 logits) and a large one (96 fp32 rows, 48 MB:
    128 KB units of 32768 logits).  The boundary's left neighbour must win, and the rows'
    confidences match the oracle."""
    V = 126464
    per_unit = 32768  # logits per unit in both plans (64 KB of bf16, 128 KB of fp32)
    rng = np.random.default_rng(17)
    x = rng.normal(0, 1, (1, L, V)).astype(np.float32)
    for j in range(min(L, 3)):
        edge = per_unit * (j + 1)
        x[0, j, [edge - 1, edge]] = 25.0            # straddles unit j | j + 1
        x[0, j, edge + 5] = 25.0
    x[0, 3, [per_unit, 2 * per_unit - 1]] = 30.0    # both ends of one unit
    logits = _bf16(x) if dtype == "bf16" else torch.from_numpy(x).cuda()
    mask_np = np.ones((1, L), np.uint8)
    conf, tok, rc, rt = check_confidence(fd, orc, logits, mask_np)
    for j in range(min(L, 3)):
        assert tok[0, j] == per_unit * (j + 1) - 1
    assert tok[0, 3] == per_unit
    check_select(fd, orc, logits, mask_np, PROFILE, 0.75)


@pytest.mark.parametrize("B,L,offset,density", [
    (5, 7, 1, 0.6),       # 35 rows: a partial mask word, mask pointer not 16-byte aligned
    (5, 7, 0, 0.6),
    (128, 32, 0, 0.05),   # 4096 rows, sparse: most first units lie beyond the producer's scan
    (128, 32, 3, 0.5),
    (4097, 1, 0, 0.1),
    (64, 64, 0, 1.0),
])
def test_mask_reading_unaligned_and_partial_words(fd, orc, B, L, offset, density):
    """Masks at any byte offset (the reduction and the selection read them byte by byte),
    row counts that are not a multiple of 32, and sparse masks whose masked rows lie beyond
    the producer's first-unit scan, against the oracle."""
    V = 1024
    w = syn.Workload("mask_edge", B, L, V, "bf16", 1.0, "target", 0.3, 4.0)
    logits = syn.make_logits(w, seed=B * 7 + L + offset, device="cuda")
    rng = np.random.default_rng(B + L + offset)
    mask_np = (rng.random((B, L)) < density).astype(np.uint8)
    store = torch.zeros(B * L + 64, dtype=torch.uint8, device="cuda")
    mask = store[offset:offset + B * L].view(B, L)
    mask.copy_(torch.from_numpy(mask_np))
    assert (mask.data_ptr() % 16 == 0) == (offset == 0)
    conf, tok = fd.fdllm_confidence(logits, mask)
    torch.cuda.synchronize()
    rc, rt, _ = orc.confidence(syn.host_bits(logits), mask_np)
    mk = mask_np.astype(bool)
    assert np.array_equal(tok.cpu().numpy()[mk], rt[mk])
    assert (np.abs(conf.cpu().numpy()[mk] - rc[mk]) / rc[mk]).max() <= 1e-5
    out = fd.fdllm_select(logits, mask, 0.75, PROFILE)
    torch.cuda.synchronize()
    ref = orc.select(syn.host_bits(logits), mask_np, PROFILE, 0.75)
    ok = ref["margin"] >= 1e-5
    assert np.array_equal(out[2].cpu().numpy()[ok], ref["n"][ok])
    assert np.array_equal(mask.cpu().numpy()[ok], ref["mask"][ok])


def _select_from_conf_case(fd, orc, conf_np, mode, param):
    B, L = conf_np.shape
    mask_np = (conf_np > 0).astype(np.uint8)
    tok_np = np.arange(B * L, dtype=np.int32).reshape(B, L)
    mask = torch.from_numpy(mask_np.copy()).cuda()
    t, c, n = fd.fdllm_select_from_conf(torch.from_numpy(conf_np).cuda(),
                                        torch.from_numpy(tok_np).cuda(), mask, param, mode)
    torch.cuda.synchronize()
    ref = orc.select_from_conf(conf_np.astype(np.float64), tok_np, mask_np, mode, param)
    return n.cpu().numpy(), c.cpu().numpy(), mask.cpu().numpy(), ref


@pytest.mark.parametrize("tau", [0.3, 0.9, 0.1, 1.0 / 3.0, 0.875, 1.0, 1.0000001, 0.0, -1.0,
                                 2.0])
def test_threshold_decides_exactly_at_float_boundaries(fd, orc, tau):
    """The threshold rule on fp32 confidences one ulp below, at and above the float nearest
    tau (tau itself is rarely representable): c >= tau is decided exactly as the oracle
    decides it on the same values in fp64, including tau at or beyond the ends of (0, 1]."""
    t32 = np.float32(tau)
    vals = [np.nextafter(t32, np.float32(-np.inf)), t32, np.nextafter(t32, np.float32(np.inf))]
    vals = [v for v in vals if 0.0 < v <= 1.0] or [np.float32(0.5)]
    rows = []
    for v in vals:   # each row: the boundary value first, then fillers far below
        rows.append([v, np.float32(0.01), np.float32(0.02), 0.0])
        rows.append([np.float32(0.9999), v, 0.0, v])
    conf_np = np.array(rows, np.float32)
    n, c, m, ref = _select_from_conf_case(fd, orc, conf_np, THRESHOLD, tau)
    assert np.array_equal(n, ref["n"]), (tau, conf_np, n, ref["n"])
    assert np.array_equal(c, ref["commit"]) and np.array_equal(m, ref["mask"])


@pytest.mark.parametrize("mode", [PROFILE, FACTOR])
@pytest.mark.parametrize("f", [-1e30, -5.0, 0.0, 1e-12, 0.75, 1.0, 1.5, 1499.0, 2000.0, 1e30])
def test_profile_and_factor_at_extreme_parameters(fd, orc, mode, f):
    """Any finite f: far beyond the range where (n+1)(1 - c) <= 1025 can change a decision
    (f clamped to +-1500 in the kernels' fixed point) every prefix is accepted or none is;
    in between, the decisions equal the oracle's on the same fp32 confidences (dyadic
    values, exact in both arithmetics)."""
    rng = np.random.default_rng(int(abs(f)) % 1000 + mode)
    conf_np = (rng.integers(1, 257, (6, 32)) / 256.0).astype(np.float32)
    conf_np[rng.random((6, 32)) < 0.2] = 0.0   # unmasked
    conf_np[0, :] = np.float32(1.0)            # all certain
    conf_np[1, :5] = np.float32(0.5)           # flat
    n, c, m, ref = _select_from_conf_case(fd, orc, conf_np, mode, f)
    ok = ref["margin"] >= 1e-12
    assert np.array_equal(n[ok], ref["n"][ok]), (f, n, ref["n"])
    assert np.array_equal(c[ok], ref["commit"][ok])
    if abs(f) >= 1500:
        m_rows = (conf_np > 0).sum(axis=1)
        assert np.array_equal(n, m_rows if f > 0 else np.minimum(m_rows, 1))
