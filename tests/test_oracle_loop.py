"""The oracle's multi-step block loop (Algorithm 1's outer loop) and its counter-based
synthetic forward pass, pinned on the CPU.

Pins:
  * the generator against an independent pure-Python evaluation of its definition
    (SplitMix64 finaliser, Irwin-Hall(4) noise, one planted peak, bf16 round to nearest
    even) and against the moments that definition implies;
  * the loop against rules whose step counts are fixed by the mathematics: a threshold above
    every confidence commits one position per step (block_len steps per block, Alg. 1's
    fallback n* = 1); a factor bound above (L + 1) accepts every prefix (one step per block);
  * the loop's bookkeeping (block offsets, global step counter, re-masking) against a
    brute-force replay built from single oracle selections.
"""
import numpy as np
import pytest

import oracle

M64 = (1 << 64) - 1
GOLD = 0x9E3779B97F4A7C15


def mix(z):
    z &= M64
    z ^= z >> 30
    z = (z * 0xBF58476D1CE4E5B9) & M64
    z ^= z >> 27
    z = (z * 0x94D049BB133111EB) & M64
    z ^= z >> 31
    return z


def bf16_bits(x32: np.float32) -> int:
    u = int(np.array([x32], np.float32).view(np.uint32)[0])
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) & 0xFFFF


def py_synth(B, L, V, seed, step, peak_max):
    out = np.zeros((B, L, V), np.uint16)
    scale = np.float32(np.sqrt(3.0) / 131072.0)
    pscale = np.float32(peak_max / 16777216.0)
    for b in range(B):
        for l in range(L):
            k = mix(seed ^ mix(((step * GOLD) & M64) ^ mix((b << 32) | l)))
            p = mix(k ^ 0xD1B54A32D192ED03)
            pidx = p % V
            height = np.float32(np.float32(p >> 40) * pscale)
            for v in range(V):
                h = mix(k + (v + 1) * GOLD)
                s = sum(2 * ((h >> (16 * j)) & 0xFFFF) + 1 for j in range(4)) - 262144
                x = np.float32(np.float32(s) * scale)
                if v == pidx:
                    x = np.float32(x + height)
                out[b, l, v] = bf16_bits(x)
    return out


def bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def test_synth_matches_its_definition(orc):
    for seed, step in ((7, 0), (12345, 3), (2**40 + 11, 17)):
        got = orc.synth_block_logits(2, 3, 40, seed, step, 16.0)
        assert np.array_equal(got, py_synth(2, 3, 40, seed, step, 16.0))


def test_synth_skips_unmasked_rows(orc):
    mask = np.array([[1, 0, 1], [0, 1, 0]], np.uint8)
    full = orc.synth_block_logits(2, 3, 64, 5, 2, 12.0)
    part = orc.synth_block_logits(2, 3, 64, 5, 2, 12.0, mask=mask)
    mk = mask.astype(bool)
    assert np.array_equal(part[mk], full[mk]) and not part[~mk].any()


def test_synth_moments_and_peak(orc):
    V = 8192
    x = bits_to_f32(orc.synth_block_logits(2, 4, V, 99, 0, 0.0)).reshape(-1, V)
    # Irwin-Hall(4) rescaled: mean 0, variance 1, support [-2 sqrt 3, 2 sqrt 3].
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    assert np.abs(x).max() <= 2 * np.sqrt(3.0) + 1e-2
    # With a peak of up to 16 the planted index is the row maximum whenever height > 7.
    y = bits_to_f32(orc.synth_block_logits(2, 4, V, 99, 0, 16.0)).reshape(-1, V)
    d = y - x
    assert ((d != 0).sum(axis=1) <= 1).all()
    assert (d >= 0).all() and d.max() > 7.0


@pytest.mark.parametrize("B,gen,Lb,V", [(2, 16, 8, 512), (3, 24, 8, 1024)])
def test_threshold_above_one_commits_one_per_step(orc, B, gen, Lb, V):
    r = orc.decode_loop(B, gen, Lb, V, oracle.THRESHOLD, 1.5, 3, 16.0, 10 * gen)
    assert (r["nfe"] == Lb).all() and r["steps"] == gen
    assert (r["seq"] >= 0).all() and (r["seq"] < V).all()


@pytest.mark.parametrize("B,gen,Lb,V", [(2, 16, 8, 512), (4, 64, 32, 1024)])
def test_factor_bound_above_block_commits_everything(orc, B, gen, Lb, V):
    # (n + 1)(1 - c) <= n + 1 <= Lb + 1 < f for every prefix n.
    r = orc.decode_loop(B, gen, Lb, V, oracle.FACTOR, float(Lb + 2), 5, 16.0, 10 * gen)
    assert (r["nfe"] == 1).all() and r["steps"] == gen // Lb
    assert (r["seq"] >= 0).all()


def replay(orc, B, gen, Lb, V, mode, param, seed, peak, max_steps):
    """Alg. 1's outer loop assembled from single oracle selections."""
    seq = np.full((B, gen), -1, np.int32)
    nfe = np.zeros(gen // Lb, np.int32)
    step = 0
    for blk in range(gen // Lb):
        mask = np.ones((B, Lb), np.uint8)
        while mask.any() and step < max_steps:
            bits = orc.synth_block_logits(B, Lb, V, seed, step, peak, mask=mask)
            r = orc.select(bits, mask, mode, param)
            c = r["commit"].astype(bool)
            seq[:, blk * Lb:(blk + 1) * Lb][c] = r["tokens"][c]
            mask = r["mask"]
            step += 1
            nfe[blk] += 1
    return seq, nfe, step


@pytest.mark.parametrize("mode,param", [(oracle.PROFILE, 1.0), (oracle.PROFILE, 0.7),
                                        (oracle.FACTOR, 1.0), (oracle.THRESHOLD, 0.9)])
def test_loop_matches_replay_of_single_selections(orc, mode, param):
    B, gen, Lb, V, seed, peak = 3, 24, 8, 512, 11, 14.0
    r = orc.decode_loop(B, gen, Lb, V, mode, param, seed, peak, 1000)
    seq, nfe, steps = replay(orc, B, gen, Lb, V, mode, param, seed, peak, 1000)
    assert np.array_equal(r["seq"], seq) and np.array_equal(r["nfe"], nfe)
    assert r["steps"] == steps == nfe.sum()
    assert (r["seq"] >= 0).all() and ((1 <= nfe) & (nfe <= Lb)).all()


def test_loop_stops_at_max_steps(orc):
    r = orc.decode_loop(2, 32, 8, 512, oracle.THRESHOLD, 1.5, 3, 16.0, 11)
    assert r["steps"] == 11
    assert list(r["nfe"]) == [8, 3, 0, 0]
    filled = r["seq"] >= 0
    assert filled[:, :8].all() and (filled[:, 8:16].sum(axis=1) == 3).all()
    assert not filled[:, 16:].any()


def py_synth_hidden(w_bits, B, L, seed, step, beta_max):
    V, H = w_bits.shape
    f32 = np.float32
    out = np.zeros((B, L, H), np.uint16)
    wf = bits_to_f32(w_bits)
    scale_n = f32(np.sqrt(3.0) / 131072.0)
    bscale = f32(beta_max / 16777216.0)
    for b in range(B):
        for l in range(L):
            k = mix(seed ^ mix(((step * GOLD) & M64) ^ mix((b << 32) | l)))
            p = mix(k ^ 0xD1B54A32D192ED03)
            t = p % V
            beta = f32(f32(p >> 40) * bscale)
            lanes = []
            for i in range(32):
                acc = f32(0.0)
                for j in range(i, H, 32):
                    acc = f32(acc + f32(wf[t, j] * wf[t, j]))
                lanes.append(acc)
            o = 16
            while o:
                lanes = [f32(lanes[i] + lanes[i ^ o]) for i in range(32)]
                o >>= 1
            scale = f32(beta / lanes[0])
            for j in range(H):
                h = mix(k + (j + 1) * GOLD)
                sv = sum(2 * ((h >> (16 * q)) & 0xFFFF) + 1 for q in range(4)) - 262144
                z = f32(f32(sv) * scale_n)
                out[b, l, j] = bf16_bits(f32(z + f32(scale * wf[t, j])))
    return out


def test_synth_hidden_matches_its_definition(orc):
    import torch
    g = torch.Generator().manual_seed(4)
    w = (torch.randn((50, 40), generator=g) / 6).to(torch.bfloat16)
    wb = w.view(torch.int16).numpy().view(np.uint16)
    for seed, step in ((7, 0), (99, 5)):
        got = orc.synth_block_hidden(wb, 2, 3, seed, step, 20.0)
        assert np.array_equal(got, py_synth_hidden(wb, 2, 3, seed, step, 20.0))


def test_synth_hidden_plants_the_target(orc):
    import fdllm_synth as syn
    _, w, _ = syn.make_lmhead_inputs(1, 1, 256, 2000, seed=1)
    wb = w.view(torch_int16()).numpy().view(np.uint16)
    h = orc.synth_block_hidden(wb, 2, 8, 11, 0, 16.0)
    x = orc.lmhead_logits(h, wb)
    # the planted index carries beta ~ U[0, 16) above N(0, ~1) noise: the argmax for tall peaks
    k_hits = (x.max(-1) > 8.0).sum()
    assert k_hits > 0
    noise = np.sort(x, axis=-1)[..., :-1]
    assert abs(noise.mean()) < 0.05 and abs(noise.std() - 1.0) < 0.15


def torch_int16():
    import torch
    return torch.int16
