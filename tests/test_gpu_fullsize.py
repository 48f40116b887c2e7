"""Parity at full workload sizes, in the launch configuration bench.py times.

The GPU runs whole batches; the oracle checks sampled batch rows one by one (rows are
independent, so a sample is checked exactly as in the full run).  The long-sequence loop
runs selection + commit until no mask remains and checks the invariants of every step plus
oracle parity on sampled steps.
"""
import numpy as np
import pytest
import torch

import fdllm_synth as syn
from gpu_util import CONF_RTOL, MARGIN, oracle_threads

pytestmark = pytest.mark.gpu
PROFILE, FACTOR = 0, 1


def _check_rows(fd, orc, logits, mask_np, rows, mode, param, tol_low=1):
    """GPU step on the whole batch; oracle on `rows`.  Returns low-margin row count."""
    mask = torch.from_numpy(mask_np.copy()).cuda()
    tok, commit, n = fd.fdllm_select(logits, mask, param, mode)
    conf, amax = fd.fdllm_confidence(logits, torch.from_numpy(mask_np).cuda())
    torch.cuda.synchronize()
    g_tok, g_commit, g_n, g_mask = (x.cpu().numpy() for x in (tok, commit, n, mask))
    g_conf, g_amax = conf.cpu().numpy().astype(np.float64), amax.cpu().numpy()
    host = syn.host_bits(logits[rows])
    ref = orc.select(host, mask_np[rows], mode, param, nthreads=oracle_threads())
    low = 0
    for k, b in enumerate(rows):
        mk = mask_np[b].astype(bool)
        assert np.array_equal(g_amax[b][mk], ref["tok"][k][mk]), "argmax row %d" % b
        rel = np.abs(g_conf[b][mk] - ref["conf"][k][mk]) / ref["conf"][k][mk]
        assert rel.max(initial=0.0) <= CONF_RTOL, "confidence row %d: %.3g" % (b, rel.max())
        if ref["margin"][k] < MARGIN:
            low += 1
            continue
        assert g_n[b] == ref["n"][k], "n* row %d" % b
        assert np.array_equal(g_commit[b], ref["commit"][k]), "commit row %d" % b
        assert np.array_equal(g_mask[b], ref["mask"][k]), "mask row %d" % b
        assert np.array_equal(g_tok[b][g_commit[b] == 1], ref["tokens"][k][g_commit[b] == 1])
    assert low <= tol_low
    return low


def test_serving_b64_full_size(fd, orc):
    w = syn.WORKLOADS["serving_b64_l32_bf16"]
    logits = syn.make_logits(w, seed=1234, device="cuda")
    mask_np = syn.make_mask(w, seed=1234)
    rows = [0, 1, 17, 31, 32, 50, 62, 63]
    _check_rows(fd, orc, logits, mask_np, rows, PROFILE, 1.0)
    _check_rows(fd, orc, logits, mask_np, rows, FACTOR, 0.75)


def test_serving_b64_graph_replay_matches_direct(fd):
    """The bench replays a captured CUDA graph; it must compute what direct calls compute."""
    w = syn.WORKLOADS["serving_b64_l32_bf16"]
    bufs = [syn.make_logits(w, seed=1234 + i, device="cuda") for i in range(2)]
    mask0 = torch.from_numpy(syn.make_mask(w, seed=1234)).cuda()
    direct = []
    for i in range(2):
        m = mask0.clone()
        direct.append([x.clone() for x in fd.fdllm_select(bufs[i], m, 1.0, PROFILE)] + [m])
    mask = mask0.clone()
    tok = torch.full((w.B, w.L), -1, dtype=torch.int32, device="cuda")
    commit = torch.empty((w.B, w.L), dtype=torch.uint8, device="cuda")
    n = torch.empty((w.B,), dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    outs = []
    with torch.cuda.stream(s):
        fd.fdllm_select(bufs[0], mask, 1.0, PROFILE, tok, commit, n, stream=s)  # warm
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for i in range(2):
            mask.copy_(mask0)
            tok.fill_(-1)
            fd.fdllm_select(bufs[i], mask, 1.0, PROFILE, tok, commit, n, stream=s)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    # after a replay the outputs hold the second step's results
    for a, b in zip(direct[1], [tok, commit, n, mask]):
        assert torch.equal(a, b)


def test_full_sequence_first_step_full_size(fd, orc):
    """B = 16, L = 1024, fp32, V = 126464 (8.3 GB of logits): the first step."""
    w = syn.WORKLOADS["full_seq_b16_l1024_fp32"]
    logits = syn.make_logits(w, seed=55, device="cuda")
    mask_np = syn.make_mask(w, seed=55)
    _check_rows(fd, orc, logits, mask_np, [3, 15], PROFILE, 1.0)
    del logits
    torch.cuda.empty_cache()


@pytest.mark.parametrize("mode", [PROFILE, FACTOR])
def test_full_sequence_loop_until_done(fd, orc, mode):
    """Selection + commit until no mask remains (B = 16, L = 1024, fp32, logits regenerated
    from (seed, step) every step), checked three ways:
      * every step, every row: >= 1 commit per row with masked positions left, commits only
        at masked positions, the mask updated by exactly the commits; all rows finish
        within L steps;
      * every step, two complete row trajectories: the GPU's decision equals the oracle's
        rule applied to the GPU's confidences on the GPU's mask state;
      * every 64th step, all rows: the confidences and argmax of 8 sampled masked positions
        per row against the oracle on the same logits; and one row's whole decision
        against the oracle from the logits."""
    w = syn.WORKLOADS["full_seq_b16_l1024_fp32"]
    B, L = w.B, w.L
    traj = (3, 11)
    rng = np.random.default_rng(7)
    mask = torch.ones((B, L), dtype=torch.uint8, device="cuda")
    tokens = torch.full((B, L), -1, dtype=torch.int32, device="cuda")
    commit = torch.empty((B, L), dtype=torch.uint8, device="cuda")
    n = torch.empty((B,), dtype=torch.int32, device="cuda")
    conf = torch.empty((B, L), dtype=torch.float32, device="cuda")
    amax = torch.empty((B, L), dtype=torch.int32, device="cuda")
    committed_total = np.zeros(B, np.int64)
    step = 0
    while True:
        before = mask.cpu().numpy()
        if before.sum() == 0:
            break
        assert step < L, "loop did not finish within L steps"
        logits = syn.make_logits(w, seed=99, device="cuda", step=step)
        fd.fdllm_confidence(logits, mask, conf, amax)
        fd.fdllm_select(logits, mask, 1.0, mode, tokens, commit, n)
        after, c, nn = mask.cpu().numpy(), commit.cpu().numpy(), n.cpu().numpy()
        live = before.sum(1) > 0
        assert np.all(nn[live] >= 1) and np.all(nn[~live] == 0)
        assert np.array_equal(c.sum(1), nn)
        assert np.all(before[c == 1] == 1) and np.array_equal(after, before & (1 - c))
        committed_total += nn
        # two trajectories: the rule on the GPU's own confidences, every step
        g_conf = conf.cpu().numpy().astype(np.float64)
        g_amax = amax.cpu().numpy()
        rows = list(traj)
        rg = orc.select_from_conf(g_conf[rows], g_amax[rows], before[rows], mode, 1.0)
        for k, b in enumerate(rows):
            if rg["margin"][k] >= 1e-12:
                assert nn[b] == rg["n"][k], "step %d row %d" % (step, b)
                assert np.array_equal(c[b], rg["commit"][k]), "step %d row %d" % (step, b)
        if step % 64 == 0:
            # sampled confidences of every row against the oracle on the same bytes
            picks = []
            for b in range(B):
                pos = np.nonzero(before[b])[0]
                if pos.size:
                    for l in rng.choice(pos, size=min(8, pos.size), replace=False):
                        picks.append((b, int(l)))
            bi = torch.tensor([p[0] for p in picks], device="cuda")
            li = torch.tensor([p[1] for p in picks], device="cuda")
            sample = logits[bi, li][None]  # [1, k, V]
            rc, rt, _ = orc.confidence(syn.host_bits(sample), np.ones((1, len(picks)), np.uint8),
                                       nthreads=oracle_threads())
            gc = np.array([g_conf[b, l] for b, l in picks])
            gt = np.array([g_amax[b, l] for b, l in picks])
            assert np.array_equal(gt, rt[0])
            assert (np.abs(gc - rc[0]) / rc[0]).max() <= CONF_RTOL
            # one row's whole decision from the logits
            b = (step // 64) % B
            ref = orc.select(syn.host_bits(logits[b:b + 1]), before[b:b + 1], mode, 1.0,
                             nthreads=oracle_threads())
            if ref["margin"][0] >= MARGIN:
                assert nn[b] == ref["n"][0] and np.array_equal(c[b], ref["commit"][0])
        del logits
        step += 1
    assert np.all(committed_total == L)
    assert np.all(tokens.cpu().numpy() >= 0)
    torch.cuda.empty_cache()
