"""The LM-head path (fdllm_lmhead_*: a tcgen05 GEMM whose epilogue reduces the logits)
against the oracle.

Two layers, each with a tolerance fixed by its arithmetic:
  1. The GEMM.  fdllm_lmhead_logits stores the fp32 accumulators.  Against the oracle's exact
     fp64 products: |x_gpu - x| <= gamma_H * sum_k |h_k w_vk| + 2^-24 |x|, the classical
     bound of a length-H dot product of exact bf16 x bf16 products accumulated in fp32, with
     gamma_H = H u / (1 - H u) and u = 2^-23 (one ulp per addition: the tensor cores'
     accumulation is not assumed to round to nearest).
  2. The fused reduction.  The reduce epilogue sees the same accumulators, so it is compared
     with the oracle run on the stored fp32 logits at the selection's own bar: argmax
     bit-exact, confidence within 1e-5 relative, decisions bit-exact except rows with
     decision margin < 1e-5.
Then, end to end against the exact logits: every GPU confidence within exp(2 E) - 1 + 1e-5
of the exact one and every GPU token within 2 E of the exact maximum logit, E the row's
largest layer-1 bound.
"""
import numpy as np
import pytest
import torch

import fdllm_synth as syn
import oracle
from gpu_util import CONF_RTOL, MARGIN, oracle_threads

pytestmark = pytest.mark.gpu

U = 2.0 ** -23


@pytest.fixture(params=[(g, bn) for bn in (256, 208) for g in ("solo", "pair")],
                ids=lambda p: "%s-n%d" % p)
def cluster(request, monkeypatch):
    """Every tile GEMM variant: one CTA per W tile, or a CTA-pair MMA (M = 256), with
    vocabulary tiles of 256 or 208 entries."""
    mode, bn = request.param
    monkeypatch.setenv("FDLLM_LMHEAD_GEMM", mode)
    monkeypatch.setenv("FDLLM_LMHEAD_BN", str(bn))
    return request.param


def bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def inputs(B, L, H, V, seed, frac=0.75, beta=(0.0, 20.0)):
    h, w, _ = syn.make_lmhead_inputs(B, L, H, V, seed, beta[0], beta[1], device="cuda")
    rng = np.random.default_rng(seed)
    mask_np = (rng.random((B, L)) < frac).astype(np.uint8)
    return h, w, mask_np


def gemm_bound(mag, x, H):
    gamma = H * U / (1.0 - H * U)
    return gamma * mag + 2.0 ** -24 * np.abs(x)


SHAPES = [
    # (B, L, H, V): ragged vocabulary tiles, ragged row tiles, a hidden size that is not a
    # multiple of the 64-element stage (zero-filled K tail), V below one tile.
    (2, 8, 128, 300),
    (4, 64, 512, 5000),
    (1, 3, 72, 40),
    (3, 100, 256, 2048),
    (4, 100, 128, 1000),   # three row tiles: an odd count for the cluster pairs
    (2, 40, 192, 3000),    # three K-blocks: the pair's last two-block stage half past H
    (2, 40, 64, 500),      # one K-block: the pair's only stage half past H
]


@pytest.mark.parametrize("B,L,H,V", SHAPES)
def test_gemm_within_fp32_accumulation_bound(fd, orc, cluster, B, L, H, V):
    h, w, mask_np = inputs(B, L, H, V, seed=B * 1000 + V)
    x = fd.fdllm_lmhead_logits(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    xg = x.cpu().numpy().astype(np.float64)
    ref, mag = orc.lmhead_logits(bits(h), bits(w), mask=mask_np, with_abs=True,
                                 nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    err = np.abs(xg[mk] - ref[mk])
    assert (err <= gemm_bound(mag[mk], ref[mk], H)).all(), err.max()
    assert np.isnan(xg[~mk]).all()  # unmasked rows untouched


def gpu_logits(fd, h, w, mask_np):
    x = fd.fdllm_lmhead_logits(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    return np.nan_to_num(x.cpu().numpy(), nan=0.0).astype(np.float32)


@pytest.mark.parametrize("B,L,H,V", SHAPES)
def test_fused_confidence_matches_oracle_on_the_same_accumulators(fd, orc, cluster, B, L, H,
                                                                  V):
    h, w, mask_np = inputs(B, L, H, V, seed=7 + V)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    x32 = gpu_logits(fd, h, w, mask_np)
    rc, rt, bad = orc.confidence(x32, mask_np, nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    assert bad == 0
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    assert np.array_equal(g_tok[mk], rt[mk])
    rel = np.abs(g_conf[mk] - rc[mk]) / rc[mk]
    assert rel.max() <= CONF_RTOL, rel.max()
    assert np.isnan(g_conf[~mk]).all() and (g_tok[~mk] == -1).all()


@pytest.mark.parametrize("k", [12, 26, 122])
def test_fused_confidence_at_large_magnitude(fd, orc, cluster, k):
    """Hidden states scaled by 2^k (exact in bf16): logits near 1e5 (k = 12), where the fp32
    reference M log2e carries a rounding residual up to 4e-3; near 2^30 (k = 26), residuals
    up to 64 and both forms of the epilogue's sum; up to 2^126.3 (k = 122), the maxima
    counted."""
    B, L, H, V = 2, 32, 256, 3000
    h, w, mask_np = inputs(B, L, H, V, seed=31 + k)
    h = h * (2.0 ** k)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    x32 = gpu_logits(fd, h, w, mask_np)
    mk = mask_np.astype(bool)
    assert np.isfinite(x32[mk]).all()
    if k >= 26:
        assert (np.abs(x32[mk]).max(axis=-1) >= 2.0 ** 30).any()
    rc, rt, bad = orc.confidence(x32, mask_np, nthreads=oracle_threads())
    assert bad == 0
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    assert np.array_equal(g_tok[mk], rt[mk])
    rel = np.abs(g_conf[mk] - rc[mk]) / rc[mk]
    assert rel.max() <= CONF_RTOL, rel.max()


@pytest.mark.parametrize("mode,param", [(oracle.PROFILE, 1.0), (oracle.PROFILE, 0.75),
                                        (oracle.FACTOR, 1.0), (oracle.THRESHOLD, 0.9)])
@pytest.mark.parametrize("B,L,H,V", [(4, 32, 512, 5000), (8, 64, 256, 3000)])
def test_fused_select_matches_oracle(fd, orc, cluster, B, L, H, V, mode, param):
    h, w, mask_np = inputs(B, L, H, V, seed=11 + L)
    x32 = gpu_logits(fd, h, w, mask_np)
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_lmhead_select(h, w, mask, param, mode)
    torch.cuda.synchronize()
    ref = orc.select(x32, mask_np, mode, param, nthreads=oracle_threads())
    ok = ref["margin"] >= MARGIN
    assert ok.mean() > 0.8
    assert np.array_equal(n.cpu().numpy()[ok], ref["n"][ok])
    assert np.array_equal(commit.cpu().numpy()[ok], ref["commit"][ok])
    assert np.array_equal(mask.cpu().numpy()[ok], ref["mask"][ok])
    t = tok.cpu().numpy()
    c = ref["commit"].astype(bool) & ok[:, None]
    assert np.array_equal(t[c], ref["tokens"][c])


@pytest.mark.parametrize("B,L,H,V", [(4, 64, 512, 5000), (2, 32, 4096, 8192)])
def test_fused_confidence_against_exact_logits(fd, orc, cluster, B, L, H, V):
    h, w, mask_np = inputs(B, L, H, V, seed=21 + H)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    ref, mag = orc.lmhead_logits(bits(h), bits(w), mask=mask_np, with_abs=True,
                                 nthreads=oracle_threads())
    rc, rt, _ = orc.confidence(ref, mask_np, nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    E = gemm_bound(mag, ref, H).max(axis=-1)
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    rel = np.abs(g_conf[mk] - rc[mk]) / rc[mk]
    assert (rel <= np.expm1(2 * E[mk]) + CONF_RTOL).all()
    x_at_tok = np.take_along_axis(ref, np.maximum(g_tok, 0)[..., None], axis=-1)[..., 0]
    assert (x_at_tok[mk] >= ref.max(axis=-1)[mk] - 2 * E[mk]).all()
    # the planted peaks make most argmaxes unambiguous: those must agree exactly
    clear = mk & (np.sort(ref, axis=-1)[..., -1] - np.sort(ref, axis=-1)[..., -2] > 4 * E)
    assert clear.sum() > 0.5 * mk.sum()
    assert np.array_equal(g_tok[clear], rt[clear])


def test_llada_shape_sampled_rows(fd, orc, cluster):
    # LLaDA-8B head: H = 4096, V = 126464; the serving batch B = 64, L = 32 with 75 % masked.
    B, L, H, V = 64, 32, syn.LLADA_HIDDEN, syn.LLADA_VOCAB
    h, w, mask_np = inputs(B, L, H, V, seed=99)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    rows = [(0, 0), (5, 17), (31, 31), (63, 12), (40, 3)]
    rows = [(b, l) for b, l in rows if mask_np[b, l]][:4]
    hs = torch.stack([h[b, l] for b, l in rows])[None]          # [1, k, H]
    one = np.ones((1, len(rows)), np.uint8)
    ref, mag = orc.lmhead_logits(bits(hs), bits(w), mask=one, with_abs=True,
                                 nthreads=oracle_threads())
    rc, rt, _ = orc.confidence(ref, one, nthreads=oracle_threads())
    E = gemm_bound(mag, ref, H).max(axis=-1)[0]
    for i, (b, l) in enumerate(rows):
        gc, gt = float(conf[b, l]), int(tok[b, l])
        assert abs(gc - rc[0, i]) / rc[0, i] <= np.expm1(2 * E[i]) + CONF_RTOL
        assert ref[0, i, gt] >= ref[0, i].max() - 2 * E[i]
    # every masked position got a confidence in (0, 1] and a token in range
    mk = mask_np.astype(bool)
    c = conf.cpu().numpy()[mk]
    t = tok.cpu().numpy()[mk]
    assert ((c > 0) & (c <= 1)).all() and ((t >= 0) & (t < V)).all()


def test_empty_mask_and_repeat(fd, cluster):
    B, L, H, V = 2, 16, 128, 1000
    h, w, _ = inputs(B, L, H, V, seed=3)
    mask = torch.zeros((B, L), dtype=torch.uint8, device="cuda")
    tok, commit, n = fd.fdllm_lmhead_select(h, w, mask, 1.0)
    torch.cuda.synchronize()
    assert (n == 0).all().item() and (commit == 0).all().item()
    m1 = torch.ones((B, L), dtype=torch.uint8, device="cuda")
    m2 = m1.clone()
    a = fd.fdllm_lmhead_select(h, w, m1, 0.75)
    b = fd.fdllm_lmhead_select(h, w, m2, 0.75)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(x, y)
    assert torch.equal(m1, m2)
    assert fd.fdllm_device_status() == 0


@pytest.mark.parametrize("H", [8, 16, 40])
def test_hidden_sizes_below_one_stage(fd, orc, H):
    """H smaller than the 64-element stage: the TMA boxes reach past the rows' end and read
    zeros there."""
    B, L, V = 2, 8, 700
    h, w, mask_np = inputs(B, L, H, V, seed=H)
    x = fd.fdllm_lmhead_logits(h, w, torch.from_numpy(mask_np).cuda())
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    ref, mag = orc.lmhead_logits(bits(h), bits(w), mask=mask_np, with_abs=True)
    mk = mask_np.astype(bool)
    xg = x.cpu().numpy().astype(np.float64)
    assert (np.abs(xg[mk] - ref[mk]) <= gemm_bound(mag[mk], ref[mk], H)).all()
    rc, rt, _ = orc.confidence(np.nan_to_num(x.cpu().numpy(), nan=0.0), mask_np)
    assert np.array_equal(tok.cpu().numpy()[mk], rt[mk])
    assert (np.abs(conf.cpu().numpy()[mk] - rc[mk]) / rc[mk]).max() <= CONF_RTOL


# ----------------------------------------------------------------------------- slab variant
SLAB_SHAPES = [
    # (B, L, H, V) with B * L <= 32: a ragged last tile, V below one tile, tiles of every
    # height the host picks on 152 SMs (96 for small V, 112 at V = 34048, 120 at 36480, 104
    # for LLaDA's head: 1216 tiles, eight per CTA), and the head itself.
    (1, 32, 256, 5000),
    (1, 3, 72, 40),
    (2, 8, 128, 300),
    (1, 17, 512, 20000),
    (4, 8, 64, 129),
    (1, 20, 128, 34048),
    (2, 7, 192, 36480),
    (1, 32, 4096, syn.LLADA_VOCAB),
]


@pytest.fixture
def slab(monkeypatch):
    """The swapped-operand variant (W as the M = 128 side, vocabulary tiles of up to 128
    entries dealt round-robin over the CTAs)."""
    monkeypatch.setenv("FDLLM_LMHEAD_GEMM", "slab")


@pytest.mark.parametrize("B,L,H,V", SLAB_SHAPES)
def test_slab_gemm_within_fp32_accumulation_bound(fd, orc, slab, B, L, H, V):
    h, w, mask_np = inputs(B, L, H, V, seed=B * 100 + V)
    x = fd.fdllm_lmhead_logits(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    xg = x.cpu().numpy().astype(np.float64)
    ref, mag = orc.lmhead_logits(bits(h), bits(w), mask=mask_np, with_abs=True,
                                 nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    err = np.abs(xg[mk] - ref[mk])
    assert (err <= gemm_bound(mag[mk], ref[mk], H)).all(), err.max()
    assert np.isnan(xg[~mk]).all()


@pytest.mark.parametrize("B,L,H,V", SLAB_SHAPES)
def test_slab_fused_confidence_matches_oracle_on_the_same_accumulators(fd, orc, slab, B, L,
                                                                       H, V):
    h, w, mask_np = inputs(B, L, H, V, seed=5 + V)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    x32 = gpu_logits(fd, h, w, mask_np)
    rc, rt, bad = orc.confidence(x32, mask_np, nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    assert bad == 0
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    assert np.array_equal(g_tok[mk], rt[mk])
    rel = np.abs(g_conf[mk] - rc[mk]) / rc[mk]
    assert rel.max() <= CONF_RTOL, rel.max()
    assert np.isnan(g_conf[~mk]).all() and (g_tok[~mk] == -1).all()


@pytest.mark.parametrize("mode,param", [(oracle.PROFILE, 1.0), (oracle.PROFILE, 0.75),
                                        (oracle.FACTOR, 1.0), (oracle.THRESHOLD, 0.9)])
def test_slab_select_matches_oracle(fd, orc, slab, mode, param):
    B, L, H, V = 1, 32, 512, 30000
    h, w, mask_np = inputs(B, L, H, V, seed=13, frac=0.9)
    x32 = gpu_logits(fd, h, w, mask_np)
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_lmhead_select(h, w, mask, param, mode)
    torch.cuda.synchronize()
    ref = orc.select(x32, mask_np, mode, param, nthreads=oracle_threads())
    ok = ref["margin"] >= MARGIN
    assert np.array_equal(n.cpu().numpy()[ok], ref["n"][ok])
    assert np.array_equal(commit.cpu().numpy()[ok], ref["commit"][ok])
    assert np.array_equal(mask.cpu().numpy()[ok], ref["mask"][ok])
    t = tok.cpu().numpy()
    c = ref["commit"].astype(bool) & ok[:, None]
    assert np.array_equal(t[c], ref["tokens"][c])


@pytest.mark.parametrize("k", [12, 26, 122])
def test_slab_confidence_at_large_magnitude(fd, orc, slab, k):
    B, L, H, V = 1, 32, 256, 3000
    h, w, mask_np = inputs(B, L, H, V, seed=31 + k)
    h = h * (2.0 ** k)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    x32 = gpu_logits(fd, h, w, mask_np)
    mk = mask_np.astype(bool)
    assert np.isfinite(x32[mk]).all()
    rc, rt, bad = orc.confidence(x32, mask_np, nthreads=oracle_threads())
    assert bad == 0
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    assert np.array_equal(g_tok[mk], rt[mk])
    assert (np.abs(g_conf[mk] - rc[mk]) / rc[mk]).max() <= CONF_RTOL


def test_slab_empty_mask_and_bit_identical_repeats(fd, slab):
    B, L, H, V = 2, 16, 128, 1000
    h, w, _ = inputs(B, L, H, V, seed=3)
    mask = torch.zeros((B, L), dtype=torch.uint8, device="cuda")
    tok, commit, n = fd.fdllm_lmhead_select(h, w, mask, 1.0)
    torch.cuda.synchronize()
    assert (n == 0).all().item() and (commit == 0).all().item()
    m = torch.ones((B, L), dtype=torch.uint8, device="cuda")
    c1, t1 = fd.fdllm_lmhead_confidence(h, w, m)
    c2, t2 = fd.fdllm_lmhead_confidence(h, w, m)
    torch.cuda.synchronize()
    assert torch.equal(c1.view(torch.int32), c2.view(torch.int32)) and torch.equal(t1, t2)
    assert fd.fdllm_device_status() == 0


def test_slab_agrees_with_the_tile_variant(fd, orc, monkeypatch):
    """The same rows through the slab variant and the 128-row tile variant: argmax equal where
    the top two logits are apart by more than both GEMMs' error, confidences within it."""
    B, L, H, V = 1, 32, 1024, 50000
    h, w, mask_np = inputs(B, L, H, V, seed=77)
    m = torch.from_numpy(mask_np).cuda()
    out = {}
    for mode in ("slab", "solo"):
        monkeypatch.setenv("FDLLM_LMHEAD_GEMM", mode)
        c, t = fd.fdllm_lmhead_confidence(h, w, m)
        torch.cuda.synchronize()
        out[mode] = (c.cpu().numpy().astype(np.float64), t.cpu().numpy())
    ref, mag = orc.lmhead_logits(bits(h), bits(w), mask=mask_np, with_abs=True,
                                 nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    E = gemm_bound(mag, ref, H).max(axis=-1)
    srt = np.sort(ref, axis=-1)
    clear = mk & (srt[..., -1] - srt[..., -2] > 4 * E)
    assert clear.sum() > 0.5 * mk.sum()
    assert np.array_equal(out["slab"][1][clear], out["solo"][1][clear])
    rel = np.abs(out["slab"][0][mk] - out["solo"][0][mk]) / out["solo"][0][mk]
    assert (rel <= np.expm1(4 * E[mk]) + 2 * CONF_RTOL).all()


def test_automatic_tiling_small_batch(fd, orc, monkeypatch):
    """No variant forced: at most 32 rows with V = 19456 (152 tiles of 128, one per CTA on
    152 SMs) is where the host takes the slab variant by itself; any other SM count may take
    another variant, which must agree with the oracle all the same."""
    monkeypatch.delenv("FDLLM_LMHEAD_GEMM", raising=False)
    monkeypatch.delenv("FDLLM_LMHEAD_BN", raising=False)
    B, L, H, V = 1, 32, 256, 19456
    h, w, mask_np = inputs(B, L, H, V, seed=8)
    conf, tok = fd.fdllm_lmhead_confidence(h, w, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    x32 = gpu_logits(fd, h, w, mask_np)
    rc, rt, bad = orc.confidence(x32, mask_np, nthreads=oracle_threads())
    mk = mask_np.astype(bool)
    assert bad == 0
    g_conf, g_tok = conf.cpu().numpy().astype(np.float64), tok.cpu().numpy()
    assert np.array_equal(g_tok[mk], rt[mk])
    assert (np.abs(g_conf[mk] - rc[mk]) / rc[mk]).max() <= CONF_RTOL


@pytest.mark.parametrize("variant", ["solo", "pair", "slab"])
@pytest.mark.parametrize("bad", [float("nan"), float("inf")])
def test_nonfinite_hidden_state_flags_only_its_row(fd, monkeypatch, variant, bad):
    """A NaN or an infinity in one masked position's hidden state makes that position's
    logits unusable: its batch row reports FDLLM_ROW_NONFINITE, commits nothing and keeps its
    mask, the status word reads FDLLM_ERR_NONFINITE, and every other batch row decides
    exactly as on the clean input (a row's logits depend on its own hidden state only)."""
    monkeypatch.setenv("FDLLM_LMHEAD_GEMM", variant)
    B, L, H, V = 2, 16, 256, 3000
    h, w, mask_np = inputs(B, L, H, V, seed=41, frac=1.0)
    bad_h = h.clone()
    bad_h[1, 5, 17] = bad
    outs = []
    for hid, expect in ((h, 0), (bad_h, 3)):
        mask = torch.from_numpy(mask_np.copy()).cuda()
        tok, commit, n = fd.fdllm_lmhead_select(hid, w, mask, 0.75)
        assert fd.fdllm_device_status() == expect
        outs.append((tok.cpu().numpy(), commit.cpu().numpy(), n.cpu().numpy(),
                     mask.cpu().numpy()))
    (t0, c0, n0, m0), (t1, c1, n1, m1) = outs
    assert n1[1] == fd.ROW_NONFINITE and c1[1].sum() == 0
    assert np.array_equal(m1[1], mask_np[1])
    assert n0[1] >= 1 and n1[0] == n0[0] >= 1
    assert np.array_equal(c1[0], c0[0]) and np.array_equal(m1[0], m0[0])
    assert np.array_equal(t1[0][c1[0] == 1], t0[0][c0[0] == 1])
