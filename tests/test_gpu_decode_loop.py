"""The device-resident decode loop (Algorithm 1's outer loop as one CUDA graph with a
conditional WHILE node) against the oracle's loop, on the counter-based synthetic forward
pass that both sides implement from the same published definition.

Tolerance: the committed sequence and the steps per block are compared bit-exactly.  A row
whose decision margin at some step is below MARGIN could flip that decision under fp32
confidences, and one flipped decision can change a block's step count and with it every
later step's logits; so each case first picks, from the oracle alone, the first seed whose
generation has no such row (all rows of every step at margin >= MARGIN).
"""
import numpy as np
import pytest
import torch

import fdllm_synth as syn
import oracle
from gpu_util import MARGIN, oracle_threads

pytestmark = pytest.mark.gpu


def forward_for(B, Lb, V, seed, peak):
    def forward(state, mask, out, stream):
        syn.synth_block_logits_gpu(out, mask, B, Lb, V, seed, step_ptr=state, peak_max=peak,
                                   stream_ptr=stream)
    return forward


def clean_seed(orc, B, gen, Lb, V, mode, param, peak, first=1, tries=12):
    for seed in range(first, first + tries):
        ref = orc.decode_loop(B, gen, Lb, V, mode, param, seed, peak, 10 * gen,
                              nthreads=oracle_threads())
        if ref["margin"].min() >= MARGIN:
            return seed, ref
    pytest.fail("no seed without near-boundary decisions in %d tries" % tries)


@pytest.mark.parametrize("B,L,V,step", [(2, 8, 4096, 0), (3, 32, 1000, 7), (1, 5, 126464, 2**20)])
def test_synth_gpu_bytes_match_oracle(fd, orc, B, L, V, step):
    mask_np = (np.arange(B * L).reshape(B, L) % 3 != 1).astype(np.uint8)
    mask = torch.from_numpy(mask_np).cuda()
    out = torch.full((B, L, V), 7.0, dtype=torch.bfloat16, device="cuda")
    st = torch.tensor([step], dtype=torch.int32, device="cuda")
    syn.synth_block_logits_gpu(out.data_ptr(), mask.data_ptr(), B, L, V, 4242,
                               step_ptr=st.data_ptr(), peak_max=16.0,
                               stream_ptr=torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    got = syn.host_bits(out)
    ref = orc.synth_block_logits(B, L, V, 4242, step, 16.0, mask=mask_np)
    mk = mask_np.astype(bool)
    assert np.array_equal(got[mk], ref[mk])
    assert (got[~mk] == syn.host_bits(torch.tensor([7.0], dtype=torch.bfloat16))[0]).all()


CASES = [
    # (B, gen_len, block_len, V, mode, param, peak)
    (4, 64, 32, 4096, oracle.PROFILE, 1.0, 16.0),
    (4, 64, 32, 4096, oracle.PROFILE, 0.6, 16.0),
    (3, 48, 16, 2048, oracle.FACTOR, 1.0, 16.0),
    (3, 48, 16, 2048, oracle.THRESHOLD, 0.9, 16.0),
    (2, 40, 8, 1000, oracle.PROFILE, 1.0, 12.0),     # V * 2 bytes = 2000, a ragged last unit
    (1, 96, 32, 8192, oracle.PROFILE, 0.95, 18.0),
    (2, 256, 128, 2048, oracle.PROFILE, 1.0, 16.0),  # blocks beyond 32: the CTA-per-row select
    (1, 512, 512, 1024, oracle.FACTOR, 1.0, 16.0),   # one 512-position block
]


@pytest.mark.parametrize("B,gen,Lb,V,mode,param,peak", CASES)
def test_decode_loop_matches_oracle(fd, orc, B, gen, Lb, V, mode, param, peak):
    seed, ref = clean_seed(orc, B, gen, Lb, V, mode, param, peak)
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")
    seq, nfe, steps = fd.fdllm_decode_loop(forward_for(B, Lb, V, seed, peak), logits, gen,
                                           param, mode, max_steps=10 * gen)
    torch.cuda.synchronize()
    assert steps == ref["steps"] == int(ref["nfe"].sum())
    assert np.array_equal(nfe.cpu().numpy(), ref["nfe"])
    assert np.array_equal(seq.cpu().numpy(), ref["seq"])


def test_decode_loop_llada_vocab(fd, orc):
    B, gen, Lb, V, peak = 2, 64, 32, syn.LLADA_VOCAB, 20.0
    seed, ref = clean_seed(orc, B, gen, Lb, V, oracle.PROFILE, 1.0, peak, tries=4)
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")
    seq, nfe, steps = fd.fdllm_decode_loop(forward_for(B, Lb, V, seed, peak), logits, gen, 1.0,
                                           oracle.PROFILE)
    assert steps == ref["steps"]
    assert np.array_equal(nfe.cpu().numpy(), ref["nfe"])
    assert np.array_equal(seq.cpu().numpy(), ref["seq"])


def test_decode_loop_twice_in_a_row(fd, orc):
    B, gen, Lb, V, peak = 3, 64, 16, 2048, 16.0
    seed, ref = clean_seed(orc, B, gen, Lb, V, oracle.PROFILE, 1.0, peak)
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")
    fwd = forward_for(B, Lb, V, seed, peak)
    a = fd.fdllm_decode_loop(fwd, logits, gen, 1.0, oracle.PROFILE)
    b = fd.fdllm_decode_loop(fwd, logits, gen, 1.0, oracle.PROFILE)
    for x, y in ((a[0], b[0]), (a[1], b[1])):
        assert torch.equal(x, y)
    assert a[2] == b[2] == ref["steps"]
    assert np.array_equal(a[0].cpu().numpy(), ref["seq"])


def test_decode_loop_threshold_above_one_takes_block_len_steps(fd):
    B, gen, Lb, V = 4, 64, 32, 4096
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")
    seq, nfe, steps = fd.fdllm_decode_loop(forward_for(B, Lb, V, 3, 16.0), logits, gen, 1.5,
                                           oracle.THRESHOLD)
    assert steps == gen and (nfe.cpu().numpy() == Lb).all()
    assert (seq >= 0).all().item() and (seq < V).all().item()


def test_decode_loop_step_bound_reports_device_error(fd):
    B, gen, Lb, V = 2, 64, 16, 2048
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(fd.FdllmError) as e:
        fd.fdllm_decode_loop(forward_for(B, Lb, V, 3, 16.0), logits, gen, 1.5,
                             oracle.THRESHOLD, max_steps=20)
    assert e.value.status == fd.ERR_DEVICE
    # The library stays usable afterwards.
    seq, nfe, steps = fd.fdllm_decode_loop(forward_for(B, Lb, V, 3, 16.0), logits, gen, 1.5,
                                           oracle.THRESHOLD)
    assert steps == gen


def test_decode_loop_forward_failure_is_reported(fd):
    B, gen, Lb, V = 2, 32, 16, 2048
    logits = torch.empty((B, Lb, V), dtype=torch.bfloat16, device="cuda")

    def failing(state, mask, out, stream):
        return 3

    with pytest.raises(fd.FdllmError) as e:
        fd.fdllm_decode_loop(failing, logits, gen, 1.0, oracle.PROFILE)
    assert e.value.status == fd.ERR_ARG
    seq, nfe, steps = fd.fdllm_decode_loop(forward_for(B, Lb, V, 3, 16.0), logits, gen, 1.5,
                                           oracle.THRESHOLD)
    assert steps == gen


# ----------------------------------------------------------------------------- LM head loop
def lm_inputs(H, V):
    _, w, _ = syn.make_lmhead_inputs(1, 1, H, V, seed=V, device="cuda")
    return w


@pytest.mark.parametrize("B,L,H,V", [(2, 8, 256, 3000), (3, 5, 72, 1000)])
def test_synth_hidden_gpu_bytes_match_oracle(fd, orc, B, L, H, V):
    w = lm_inputs(H, V)
    mask_np = (np.arange(B * L).reshape(B, L) % 4 != 2).astype(np.uint8)
    mask = torch.from_numpy(mask_np).cuda()
    out = torch.full((B, L, H), 5.0, dtype=torch.bfloat16, device="cuda")
    st = torch.tensor([9], dtype=torch.int32, device="cuda")
    syn.synth_block_hidden_gpu(out.data_ptr(), mask.data_ptr(), B, L, H, V, w.data_ptr(), 77,
                               step_ptr=st.data_ptr(), beta_max=18.0,
                               stream_ptr=torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    got = syn.host_bits(out)
    ref = orc.synth_block_hidden(syn.host_bits(w), B, L, 77, 9, 18.0, mask=mask_np)
    mk = mask_np.astype(bool)
    assert np.array_equal(got[mk], ref[mk])


def hidden_forward(B, Lb, H, V, w, seed, beta):
    def forward(state, mask, out, stream):
        syn.synth_block_hidden_gpu(out, mask, B, Lb, H, V, w.data_ptr(), seed, step_ptr=state,
                                   beta_max=beta, stream_ptr=stream)
    return forward


@pytest.mark.parametrize("mode,param,Lb,gen", [(oracle.PROFILE, 1.0, 16, 32),
                                                (oracle.PROFILE, 0.75, 16, 32),
                                                (oracle.FACTOR, 1.0, 16, 32),
                                                (oracle.PROFILE, 1.0, 64, 128),
                                                (oracle.FACTOR, 1.0, 96, 192)])
def test_decode_loop_lmhead_against_host_loop_and_oracle(fd, orc, mode, param, Lb, gen):
    """The device-resident loop with the LM head equals a host-driven loop of
    fdllm_lmhead_select calls (same kernels: bit-exact), and every step of the host loop
    matches the oracle run on that step's tensor-core accumulators (margin >= 1e-5).  Blocks
    of 16 positions take the slab GEMM (B * L <= 32), blocks of 64 and 96 the tile GEMM and,
    past 32 positions, the CTA-per-row selection."""
    B, H, V, seed, beta = 2, 256, 3000, 5, 20.0
    w = lm_inputs(H, V)
    hidden = torch.empty((B, Lb, H), dtype=torch.bfloat16, device="cuda")
    seq_d, nfe_d, steps_d = fd.fdllm_decode_loop_lmhead(
        hidden_forward(B, Lb, H, V, w, seed, beta), hidden, w, gen, param, mode)
    torch.cuda.synchronize()

    stream = torch.cuda.current_stream().cuda_stream
    seq = np.full((B, gen), -1, np.int32)
    nfe, step, checked = [], 0, 0
    tok = torch.empty((B, Lb), dtype=torch.int32, device="cuda")
    commit = torch.empty((B, Lb), dtype=torch.uint8, device="cuda")
    n = torch.empty((B,), dtype=torch.int32, device="cuda")
    for blk in range(gen // Lb):
        mask = torch.ones((B, Lb), dtype=torch.uint8, device="cuda")
        k = 0
        while bool(mask.any().item()):
            syn.synth_block_hidden_gpu(hidden.data_ptr(), mask.data_ptr(), B, Lb, H, V,
                                       w.data_ptr(), seed, step=step, beta_max=beta,
                                       stream_ptr=stream)
            before = mask.cpu().numpy()
            x32 = fd.fdllm_lmhead_logits(hidden, w, mask)
            fd.fdllm_lmhead_select(hidden, w, mask, param, mode, tok, commit, n)
            torch.cuda.synchronize()
            x32 = np.nan_to_num(x32.cpu().numpy(), nan=0.0).astype(np.float32)
            ref = orc.select(x32, before, mode, param, nthreads=oracle_threads())
            c = commit.cpu().numpy()
            for b in range(B):
                if ref["margin"][b] >= MARGIN:
                    assert n[b].item() == ref["n"][b] and np.array_equal(c[b], ref["commit"][b])
                    checked += 1
            t = tok.cpu().numpy()
            seq[:, blk * Lb:(blk + 1) * Lb][c == 1] = t[c == 1]
            step += 1
            k += 1
        nfe.append(k)
    assert checked > 0
    assert steps_d == step
    assert list(nfe_d.cpu().numpy()) == nfe
    assert np.array_equal(seq_d.cpu().numpy(), seq)


def test_decode_loop_lmhead_stops_on_a_nonfinite_hidden_state(fd):
    """A forward pass that leaves a NaN in a masked position's hidden state: its row commits
    nothing, so the loop with the LM head ends after that step with FDLLM_ERR_NONFINITE
    instead of running to max_steps."""
    B, gen, Lb, H, V = 2, 32, 16, 256, 3000
    w = lm_inputs(H, V)
    hidden = torch.empty((B, Lb, H), dtype=torch.bfloat16, device="cuda")
    synth = hidden_forward(B, Lb, H, V, w, 5, 20.0)

    def forward(state, mask, out, stream):
        synth(state, mask, out, stream)
        with torch.cuda.stream(torch.cuda.ExternalStream(stream)):
            hidden[0, 3, 11].fill_(float("nan"))

    with pytest.raises(fd.FdllmError) as err:
        fd.fdllm_decode_loop_lmhead(forward, hidden, w, gen, 1.0, oracle.PROFILE,
                                    max_steps=10 * gen)
    assert err.value.status == 3  # FDLLM_ERR_NONFINITE
    assert fd.fdllm_device_status() == 3
    assert fd.fdllm_device_status() == 0
