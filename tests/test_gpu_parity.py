"""CUDA path vs the CPU oracle on identical seeded inputs, through the C interface.

Covers step a1 alone (fdllm_confidence), steps a2-a5 alone (fdllm_select_from_conf) and the
whole step (fdllm_select / fdllm_select_ws) on the selection workloads at sizes the oracle
finishes in seconds: several 16 KB chunks per row, rows split across CTAs, ragged last
chunks, partially masked and empty rows, every mode.
"""
import numpy as np
import pytest
import torch

import fdllm_synth as syn
from gpu_util import check_confidence, check_select

pytestmark = pytest.mark.gpu

W = syn.WORKLOADS
PROFILE, FACTOR, THRESHOLD = 0, 1, 2


def _mask(B, L, seed, frac=0.7, empty_rows=()):
    rng = np.random.default_rng(seed)
    m = (rng.random((B, L)) < frac).astype(np.uint8)
    for b in empty_rows:
        m[b] = 0
    return m


@pytest.mark.parametrize("dtype", ["bf16", "fp16", "fp32"])
@pytest.mark.parametrize("V", [8, 1000, 8200, 20000, 126464])
@pytest.mark.parametrize("B,L", [(1, 1), (3, 7), (2, 33), (4, 64)])
def test_confidence_shapes(fd, orc, dtype, V, B, L):
    if dtype == "fp32" and V % 4:
        pytest.skip("V*4 not a multiple of 16")
    w = syn.Workload("shape", B, L, V, dtype, 1.0, "uniform", 0.0, 14.0)
    logits = syn.make_logits(w, seed=V * 7 + L, device="cuda")
    check_confidence(fd, orc, logits, _mask(B, L, seed=V + B, empty_rows=(0,) if B > 2 else ()))


@pytest.mark.parametrize("name", ["single_block_b1_l32_bf16", "mixed_mask_b8_l32_bf16",
                                  "tie_groups_b16_l64_fp32", "target_b8_l32_bf16",
                                  "target_ties_b16_l64_fp32", "target_b8_l32_fp16"])
def test_confidence_workloads_full_vocab(fd, orc, name):
    w = W[name]
    logits = syn.make_logits(w, seed=101, device="cuda")
    check_confidence(fd, orc, logits, syn.make_mask(w, seed=101))


@pytest.mark.parametrize("mode,param", [(PROFILE, 1.0), (PROFILE, 0.75), (PROFILE, 0.5),
                                        (PROFILE, 2.0), (FACTOR, 1.0), (FACTOR, 0.75),
                                        (FACTOR, 0.5), (FACTOR, 2.0), (THRESHOLD, 0.9),
                                        (THRESHOLD, 0.5)])
@pytest.mark.parametrize("name", ["single_block_b1_l32_bf16", "mixed_mask_b8_l32_bf16",
                                  "target_b8_l32_bf16", "target_b8_l32_fp16"])
def test_select_workloads(fd, orc, name, mode, param):
    w = W[name]
    logits = syn.make_logits(w, seed=202, device="cuda")
    low = check_select(fd, orc, logits, syn.make_mask(w, seed=202), mode, param)
    assert low <= max(1, w.B // 8)


@pytest.mark.parametrize("name", ["tie_groups_b16_l64_fp32", "target_ties_b16_l64_fp32"])
def test_equal_confidence_groups_profile_equals_factor(fd, orc, name):
    """Rows of a tie group are byte-identical, so their confidences are identical on the GPU
    too; where the committed prefix is flat, profile(delta = 0) and factor(f = 1) agree
    (Cor. factor-reduction)."""
    w = W[name]
    logits = syn.make_logits(w, seed=303, device="cuda")
    mask_np = syn.make_mask(w, seed=303)
    conf, _, _, _ = check_confidence(fd, orc, logits, mask_np)
    g = conf.reshape(w.B, w.L // 8, 8)
    assert np.all(g == g[..., :1]), "tie groups must give bit-identical confidences"
    check_select(fd, orc, logits, mask_np, PROFILE, 1.0)
    check_select(fd, orc, logits, mask_np, FACTOR, 1.0)
    _, _, n_p = fd.fdllm_select(logits, torch.from_numpy(mask_np).cuda(), 1.0, PROFILE)
    _, _, n_f = fd.fdllm_select(logits, torch.from_numpy(mask_np).cuda(), 1.0, FACTOR)
    n_p, n_f = n_p.cpu().numpy(), n_f.cpu().numpy()
    for b in range(w.B):
        c = np.sort(conf[b])[::-1]
        k = int(n_p[b])
        if np.all(c[:k] == c[0]):  # flat over the committed prefix and its successor set
            assert n_p[b] >= n_f[b]
            if k < len(c) and c[k] == c[0]:
                assert n_p[b] == n_f[b]


@pytest.mark.parametrize("mode,param", [(PROFILE, 0.75), (FACTOR, 0.75), (THRESHOLD, 0.9)])
def test_select_from_conf_matches_oracle_exactly(fd, orc, mode, param):
    """Steps a2-a5 on given fp32 confidences: the oracle sees the same values widened to
    fp64, so decisions agree bit for bit (no margin exclusion needed)."""
    rng = np.random.default_rng(9)
    for B, L in ((5, 32), (3, 1), (2, 1024), (7, 100), (4, 64)):
        c = rng.beta(0.6, 0.25, (B, L)).astype(np.float32)
        c = np.clip(c, np.float32(1e-6), np.float32(1.0))
        c[0, : min(L, 4)] = c[0, 0]  # ties
        mask_np = (rng.random((B, L)) < 0.8).astype(np.uint8)
        mask_np[-1] = 0  # an empty row
        tok = rng.integers(0, 126464, (B, L)).astype(np.int32)
        mask = torch.from_numpy(mask_np.copy()).cuda()
        out_tok, commit, n = fd.fdllm_select_from_conf(torch.from_numpy(c).cuda(),
                                                       torch.from_numpy(tok).cuda(), mask,
                                                       param, mode)
        ref = orc.select_from_conf(c.astype(np.float64), tok, mask_np, mode, param)
        same = ref["margin"] >= 1e-12
        assert np.array_equal(n.cpu().numpy()[same], ref["n"][same])
        assert np.array_equal(commit.cpu().numpy()[same], ref["commit"][same])
        assert np.array_equal(out_tok.cpu().numpy()[same], ref["tokens"][same])
        assert np.array_equal(mask.cpu().numpy()[same], ref["mask"][same])


def test_select_ws_matches_select(fd, orc):
    w = W["mixed_mask_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=404, device="cuda")
    mask_np = syn.make_mask(w, seed=404)
    ws = torch.zeros(fd.fdllm_workspace_bytes(w.B, w.L, w.V, fd.BF16), dtype=torch.uint8,
                     device="cuda")
    outs = []
    for use_ws in (False, True, True):
        mask = torch.from_numpy(mask_np.copy()).cuda()
        if use_ws:
            r = fd.fdllm_select_ws(logits, mask, 0.75, PROFILE, ws)
        else:
            r = fd.fdllm_select(logits, mask, 0.75, PROFILE)
        outs.append([x.cpu().numpy() for x in r] + [mask.cpu().numpy()])
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            assert np.array_equal(a, b)
    assert fd.fdllm_workspace_status(ws) == 0
    assert fd.fdllm_device_status() == 0


def test_deterministic_rerun(fd):
    w = W["target_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=505, device="cuda")
    mask = torch.from_numpy(syn.make_mask(w, seed=505)).cuda()
    c1, t1 = fd.fdllm_confidence(logits, mask)
    c2, t2 = fd.fdllm_confidence(logits, mask)
    assert torch.equal(c1.view(torch.int32), c2.view(torch.int32)) and torch.equal(t1, t2)


def test_fp16_nonfinite_ties_and_extremes(fd, orc):
    """fp16 rows: a NaN, a +inf maximum, all -inf, -inf entries, the largest finite half
    (65504), subnormals, and maxima tied within and across 16-byte vectors."""
    B, L, V = 2, 8, 4096
    rng = np.random.default_rng(5)
    x = rng.normal(0.0, 2.0, (B, L, V)).astype(np.float16)
    x[0, 0, 17] = np.nan
    x[0, 1, 100] = np.inf
    x[0, 2, :] = -np.inf
    x[0, 3, ::3] = -np.inf
    x[0, 4, 5] = 65504.0
    x[0, 4, 4000] = 65504.0                    # tied maximum, later index
    x[0, 5, :] = np.float16(6e-8)              # all subnormal and equal: c = 1/V, x_hat = 0
    x[1, 0, 8:16] = 30.0                       # a tie inside one vector and the next
    x[1, 1, 4095] = 40.0                       # maximum in the last element
    logits = torch.from_numpy(x).cuda()
    mask = np.ones((B, L), np.uint8)
    check_confidence(fd, orc, logits, mask)
    check_select(fd, orc, logits, mask, PROFILE, 0.75)


def test_vocab_reduce_alone_leaves_the_library_consistent(fd, orc):
    """fdllm_vocab_reduce (the reduction kernel by itself, for timing) resets its work counter:
    selections and confidences after it still match the oracle."""
    w = W["mixed_mask_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=808, device="cuda")
    mask_np = syn.make_mask(w, seed=808)
    m = torch.from_numpy(mask_np).cuda()
    for _ in range(3):
        fd.fdllm_vocab_reduce(logits, m)
    check_confidence(fd, orc, logits, mask_np)
    fd.fdllm_vocab_reduce(logits, m)
    check_select(fd, orc, logits, mask_np, PROFILE, 0.75)
    assert fd.fdllm_device_status() == 0


def test_concurrent_streams_with_own_workspaces(fd):
    """Two selection streams, each with its own caller workspace, launched with no ordering
    between them (the documented way to run concurrent steps): every repetition gives each
    stream exactly the decisions of the same call run alone."""
    wa, wb = W["mixed_mask_b8_l32_bf16"], W["target_b8_l32_bf16"]
    logits = [syn.make_logits(wa, seed=606, device="cuda"),
              syn.make_logits(wb, seed=607, device="cuda")]
    masks_np = [syn.make_mask(wa, seed=606), syn.make_mask(wb, seed=607)]
    shapes = [(wa.B, wa.L), (wb.B, wb.L)]
    ref = []
    for x, m_np, (B, L) in zip(logits, masks_np, shapes):
        m = torch.from_numpy(m_np.copy()).cuda()
        tok = torch.full((B, L), -1, dtype=torch.int32, device="cuda")
        r = fd.fdllm_select(x, m, 0.75, PROFILE, tok)
        torch.cuda.synchronize()
        ref.append([t.cpu().numpy() for t in r] + [m.cpu().numpy()])
    ws = [torch.zeros(fd.fdllm_workspace_bytes(w.B, w.L, w.V, fd.BF16), dtype=torch.uint8,
                      device="cuda") for w in (wa, wb)]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    for _ in range(20):
        masks = [torch.from_numpy(m.copy()).cuda() for m in masks_np]
        toks = [torch.full(s, -1, dtype=torch.int32, device="cuda") for s in shapes]
        torch.cuda.synchronize()
        res = []
        for i in range(2):
            with torch.cuda.stream(streams[i]):
                res.append(fd.fdllm_select_ws(logits[i], masks[i], 0.75, PROFILE, ws[i],
                                              out_tokens=toks[i], stream=streams[i]))
        torch.cuda.synchronize()
        for i in range(2):
            got = [t.cpu().numpy() for t in res[i]] + [masks[i].cpu().numpy()]
            for a, b in zip(ref[i], got):
                assert np.array_equal(a, b)
    for w in ws:
        assert fd.fdllm_workspace_status(w) == 0


@pytest.mark.parametrize("masked_rows", [0, 1, 5, 76, 77, 152])
def test_work_counter_reset_by_the_last_fetch(fd, orc, masked_rows):
    """The reduction puts its work counter back to zero with the launch's last fetch, for
    any number of units against the grid (none, fewer than the CTAs, about one per CTA,
    more): a dense selection right after still matches the oracle."""
    w = W["mixed_mask_b8_l32_bf16"]
    logits = syn.make_logits(w, seed=909, device="cuda")
    sparse = np.zeros((w.B, w.L), np.uint8)
    sparse.reshape(-1)[np.random.default_rng(masked_rows).choice(w.B * w.L, masked_rows,
                                                                  replace=False)] = 1
    for _ in range(3):
        fd.fdllm_vocab_reduce(logits, torch.from_numpy(sparse).cuda())
        fd.fdllm_select(logits, torch.from_numpy(sparse.copy()).cuda(), 0.75, PROFILE)
    check_select(fd, orc, logits, np.ones((w.B, w.L), np.uint8), PROFILE, 0.75)
    assert fd.fdllm_device_status() == 0
