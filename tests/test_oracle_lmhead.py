"""The oracle's LM-head logits (exact fp64 products of bf16 inputs), pinned on the CPU
against closed forms and an independent library evaluation."""
import numpy as np
import torch

BF16_ONE = 0x3F80


def bits(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def test_identity_head_returns_the_hidden_state(orc):
    H = 64
    h = torch.randn((2, 3, H)).to(torch.bfloat16)
    w = np.zeros((H, H), np.uint16)
    w[np.arange(H), np.arange(H)] = BF16_ONE
    out = orc.lmhead_logits(bits(h), w)
    assert np.array_equal(out, h.to(torch.float64).numpy())


def test_single_column_power_of_two(orc):
    # w[v] = 2^(v - 3) e_k: logit_v = h_k 2^(v - 3) exactly.
    H, V, k = 16, 8, 5
    h = torch.randn((1, 4, H)).to(torch.bfloat16)
    w = torch.zeros((V, H), dtype=torch.float32)
    w[:, k] = torch.tensor([2.0 ** (v - 3) for v in range(V)])
    out = orc.lmhead_logits(bits(h), bits(w.to(torch.bfloat16)))
    hk = h.to(torch.float64)[0, :, k].numpy()
    assert np.array_equal(out[0], hk[:, None] * np.array([2.0 ** (v - 3) for v in range(V)]))


def test_matches_library_matmul_and_bounds(orc):
    g = torch.Generator().manual_seed(3)
    h = torch.randn((3, 5, 96), generator=g).to(torch.bfloat16)
    w = (torch.randn((70, 96), generator=g) / 10).to(torch.bfloat16)
    out, mag = orc.lmhead_logits(bits(h), bits(w), with_abs=True, nthreads=2)
    ref = torch.einsum("blh,vh->blv", h.to(torch.float64), w.to(torch.float64)).numpy()
    assert np.allclose(out, ref, rtol=0, atol=1e-12)
    absref = torch.einsum("blh,vh->blv", h.to(torch.float64).abs(),
                          w.to(torch.float64).abs()).numpy()
    assert np.allclose(mag, absref, rtol=1e-14, atol=0)
    assert (mag >= np.abs(out)).all()


def test_scaling_by_two_is_exact_and_unmasked_rows_untouched(orc):
    g = torch.Generator().manual_seed(4)
    h = torch.randn((2, 4, 32), generator=g).to(torch.bfloat16)
    w = torch.randn((24, 32), generator=g).to(torch.bfloat16)
    mask = np.array([[1, 0, 1, 1], [0, 0, 1, 0]], np.uint8)
    a = orc.lmhead_logits(bits(h), bits(w), mask=mask)
    b = orc.lmhead_logits(bits((h.float() * 2).to(torch.bfloat16)), bits(w), mask=mask)
    assert np.array_equal(b, 2 * a)
    assert not a[mask == 0].any() and a[mask == 1].any()


def test_planted_recipe_puts_the_peak_on_the_target(orc):
    import fdllm_synth as syn
    h, w, t = syn.make_lmhead_inputs(2, 8, 256, 512, seed=5, beta_lo=12.0, beta_hi=16.0)
    x = orc.lmhead_logits(bits(h), bits(w))
    assert (x.argmax(-1) == t.numpy()).all()
    others = np.where(np.arange(512)[None, None, :] == t.numpy()[..., None], np.nan, x)
    # w_v . h = w_v . z + beta w_v . w_t / |w_t|^2 with w_v . w_t ~ N(0, 1/H) for v != t:
    # variance 1 + E[beta^2] / H, E[beta^2] = (16^3 - 12^3) / (3 * 4) for beta ~ U[12, 16].
    sd = np.sqrt(1.0 + (16.0 ** 3 - 12.0 ** 3) / 12.0 / 256)
    assert abs(np.nanmean(others)) < 0.05 and abs(np.nanstd(others) - sd) < 0.1
