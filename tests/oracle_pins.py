"""Checks that pin the CPU oracle to what the paper and the mathematics fix.

Every check takes an ``oracle.Oracle`` and raises AssertionError when the oracle disagrees
with an independent statement: a library routine (torch float64 logsumexp / argmax), a
closed form, brute force over all candidate subsets, the paper's propositions and
corollaries, or values worked out by hand (tests/golden).  None of them re-types the
oracle's own formula.  ``test_oracle_pins.py`` runs them on the committed oracle and
``test_oracle_mutants.py`` runs them on copies with planted mistakes, each of which must
fail at least one check.
"""
from __future__ import annotations

import itertools
import json
import math
import os

import numpy as np
import torch

PROFILE, FACTOR, THRESHOLD = 0, 1, 2
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "hand_worked_profiles.json")


# ----------------------------------------------------------------------------- helpers
def bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 (round to nearest even, by torch) as raw uint16 bits."""
    t = torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def widen(arr: np.ndarray) -> torch.Tensor:
    """Exact float64 view of fp32, fp16 or bf16-bits logits, via torch's own conversion."""
    if arr.dtype == np.uint16:
        return torch.from_numpy(arr.view(np.int16).copy()).view(torch.bfloat16).to(torch.float64)
    return torch.from_numpy(arr).to(torch.float64)


def run_profiles(o, profiles, mode, param, pos=None):
    """Run select_from_conf on a batch of confidence lists (one batch row each).

    Returns (n [B], committed position sets)."""
    B = len(profiles)
    L = max(1, max(len(p) for p in profiles))
    conf = np.zeros((B, L))
    mask = np.zeros((B, L), np.uint8)
    tok = np.arange(B * L, dtype=np.int32).reshape(B, L)
    for b, p in enumerate(profiles):
        places = range(len(p)) if pos is None else pos[b]
        for c, l in zip(p, places):
            conf[b, l] = c
            mask[b, l] = 1
    r = o.select_from_conf(conf, tok, mask, mode, param)
    sets = [set(np.nonzero(r["commit"][b])[0].tolist()) for b in range(B)]
    return r["n"], sets, r


def G_of_subset(cs):
    k = len(cs)
    return max(0.0, sum(cs) - (k - 1)) - (1.0 - min(cs))


# ----------------------------------------------------------------------------- pins
def pin_confidence_vs_torch(o):
    """c = exp(M - logsumexp) and x_hat = first argmax, against torch float64 (Sec. 3)."""
    rng = np.random.default_rng(11)
    for dt in ("fp32", "bf16", "fp16"):
        for V in (1, 2, 7, 1000, 4099):
            B, L = 3, 5
            x = rng.normal(0.0, 3.0, (B, L, V)).astype(np.float32)
            if V > 2:
                x[0, 1, 1::2] = -np.inf          # -inf entries contribute nothing
                x[1, 2, : V // 2] = x[1, 2, V // 2]  # repeated values
            arr = bf16_bits(x) if dt == "bf16" else (x.astype(np.float16) if dt == "fp16"
                                                     else x)
            mask = (rng.random((B, L)) < 0.7).astype(np.uint8)
            mask[0, 1] = mask[1, 2] = 1
            conf, tok, bad = o.confidence(arr, mask)
            assert bad == 0
            t = widen(arr)
            ref_c = torch.exp(t.max(-1).values - torch.logsumexp(t, -1)).numpy()
            ref_t = torch.argmax(t, -1).numpy()
            mk = mask.astype(bool)
            np.testing.assert_allclose(conf[mk], ref_c[mk], rtol=1e-12, atol=0)
            assert np.array_equal(tok[mk], ref_t[mk])
            assert np.all(tok[~mk] == -1)


def pin_half_widening(o):
    """The fp16 widening: every one of the 65536 half bit patterns against numpy's own
    float16 -> float64 conversion (NaN patterns: NaN)."""
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    got = o.half_to_double(bits)
    ref = bits.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


def pin_confidence_closed_forms(o):
    """Equal logits give c = 1/V, x_hat = 0; two-valued rows give the two-term closed form."""
    for V in (1, 2, 5, 4096, 126464):
        x = np.full((1, 1, V), 0.37, np.float32)
        conf, tok, _ = o.confidence(x, np.ones((1, 1), np.uint8))
        assert math.isclose(conf[0, 0], 1.0 / V, rel_tol=1e-12) and tok[0, 0] == 0
    V = 1000
    for a, b, k in ((2.0, -1.0, 17), (-3.0, 0.5, 0), (-3.0, 0.5, 9), (10.0, 10.0 - 0.25, 999)):
        x = np.full((1, 1, V), b, np.float32)
        x[0, 0, k] = a
        conf, tok, _ = o.confidence(x, np.ones((1, 1), np.uint8))
        fa, fb = float(np.float32(a)), float(np.float32(b))
        if fa > fb:
            c = 1.0 / (1.0 + (V - 1) * math.exp(fb - fa))
            want = k
        else:
            c = 1.0 / ((V - 1) + math.exp(fa - fb))
            want = 0 if k != 0 else 1
        assert math.isclose(conf[0, 0], c, rel_tol=1e-12), (a, b, k, conf[0, 0], c)
        assert tok[0, 0] == want
    # exact ties of the maximum: lowest index wins, c = 1 / (ties + rest)
    x = np.full((1, 1, 64), -2.0, np.float32)
    x[0, 0, [40, 3, 17]] = 1.5
    conf, tok, _ = o.confidence(x, np.ones((1, 1), np.uint8))
    assert tok[0, 0] == 3
    assert math.isclose(conf[0, 0], 1.0 / (3 + 61 * math.exp(-3.5)), rel_tol=1e-12)


def pin_extreme_magnitudes(o):
    """Finite logits of any magnitude: rows of the dtype's most negative finite value give
    c = 1/V and x_hat = 0; the largest finite value tied twice over very negative logits
    gives exactly 1/2 at the first of them; a spread far beyond exp's range leaves only the
    maximum (c = 1); a constant shift by a power of two is exact in fp32 and leaves c
    unchanged.  (A sum of exp(x) not re-based to the maximum overflows on every case.)"""
    V = 300
    f32 = np.finfo(np.float32)
    for dt, lo, hi in (("fp32", float(f32.min), float(f32.max)),
                       ("fp16", -65504.0, 65504.0),
                       ("bf16", -3.3895313892515355e38, 3.3895313892515355e38)):
        def run(x):
            a = x.astype(np.float16) if dt == "fp16" else x.astype(np.float32)
            if dt == "bf16":
                a = bf16_bits(a)
            return o.confidence(a[None, None], np.ones((1, 1), np.uint8))
        conf, tok, bad = run(np.full(V, lo))
        assert bad == 0 and math.isclose(conf[0, 0], 1.0 / V, rel_tol=1e-12) and tok[0, 0] == 0
        x = np.full(V, lo / 2)
        x[[7, 200]] = hi
        conf, tok, _ = run(x)
        assert conf[0, 0] == 0.5 and tok[0, 0] == 7
        x = np.linspace(lo / 4, hi / 4, V)
        conf, tok, _ = run(x)
        assert conf[0, 0] == 1.0 and tok[0, 0] == V - 1
    # a row shifted by 2^20 against the same row shifted back (both shifts exact in fp32)
    x = np.random.default_rng(3).normal(0.0, 2.0, V).astype(np.float32)
    xs = x + np.float32(2.0 ** 20)
    xr = xs - np.float32(2.0 ** 20)
    c1, t1, _ = o.confidence(xs[None, None], np.ones((1, 1), np.uint8))
    c2, t2, _ = o.confidence(xr[None, None], np.ones((1, 1), np.uint8))
    assert math.isclose(c1[0, 0], c2[0, 0], rel_tol=1e-12) and t1[0, 0] == t2[0, 0]


def pin_nonfinite(o):
    """NaN anywhere, or a max of +inf / -inf, marks the row invalid; other rows unaffected."""
    x = np.zeros((1, 5, 16), np.float32)
    x[0, 0, 3] = np.nan
    x[0, 1, 7] = np.inf
    x[0, 2, :] = -np.inf
    x[0, 3, ::2] = -np.inf
    x[0, 4, 5] = 2.0
    conf, tok, bad = o.confidence(x, np.ones((1, 5), np.uint8))
    assert bad == 3
    assert np.all(np.isnan(conf[0, :3])) and np.all(tok[0, :3] == -1)
    assert math.isclose(conf[0, 3], 1.0 / 8, rel_tol=1e-12) and tok[0, 3] == 1
    assert tok[0, 4] == 5
    r = o.select_from_conf(conf, tok, np.ones((1, 5), np.uint8), PROFILE, 1.0)
    assert r["n"][0] == -1 and r["commit"].sum() == 0 and r["mask"].sum() == 5


def pin_hand_worked(o):
    """Values worked out by hand from the paper's definitions (tests/golden)."""
    with open(GOLDEN) as fh:
        cases = json.load(fh)["cases"]
    modes = {"profile": PROFILE, "factor": FACTOR, "threshold": THRESHOLD}
    for case in cases:
        c = np.array(case["c_sorted"])
        Ln, Un, Gn = o.frechet_scan(c)
        np.testing.assert_allclose(Ln, case["L"], atol=1e-12)
        np.testing.assert_allclose(Un, case["U"], atol=1e-12)
        np.testing.assert_allclose(Gn, case["G"], atol=1e-12)
        # positions listed in reverse so the sort is exercised
        rev = list(reversed(range(len(c))))
        for key, want in case["nstar"].items():
            name, p = key.split()
            n, sets, _ = run_profiles(o, [list(c)], modes[name], float(p.split("=")[1]),
                                      pos=[rev])
            assert n[0] == want, (case["name"], key, n[0], want)
            ranked = sorted(zip(c, rev), key=lambda cp: (-cp[0], cp[1]))
            assert sets[0] == {p for _, p in ranked[:want]}, (case["name"], key)


def _random_profiles(rng, count, m_max, dyadic=None):
    out = []
    for _ in range(count):
        m = int(rng.integers(1, m_max + 1))
        if dyadic:
            c = rng.integers(1, dyadic + 1, m) / dyadic
        else:
            c = rng.beta(0.6, 0.25, m)
            c = np.clip(c, 1e-6, 1.0)
        out.append(list(map(float, c)))
    return out


def pin_bruteforce_subsets(o):
    """n* = largest |S| with an admissible subset S (brute force over all subsets), and the
    committed set attains the best score at that size (Sec. 3 rule, Alg. 1)."""
    rng = np.random.default_rng(5)
    profiles = _random_profiles(rng, 160, 8, dyadic=64)
    for f in (1.0, 0.75, 0.5, 0.25):
        delta = 1.0 - f
        n, sets, _ = run_profiles(o, profiles, PROFILE, f)
        nf, setsf, _ = run_profiles(o, profiles, FACTOR, f)
        for b, c in enumerate(profiles):
            m = len(c)
            best = {k: max(G_of_subset([c[i] for i in S])
                           for S in itertools.combinations(range(m), k))
                    for k in range(1, m + 1)}
            ks = [k for k in range(1, m + 1) if best[k] > delta]
            want = max(ks) if ks else 1
            assert n[b] == want, (c, f, n[b], want)
            got = sorted(sets[b])
            assert len(got) == want
            if ks:
                assert G_of_subset([c[i] for i in got]) == best[want]
            # factor: (|S|+1)(1 - min_S c) < f for some S of size k
            kf = [k for k in range(1, m + 1)
                  if any((k + 1) * (1.0 - min(c[i] for i in S)) < f
                         for S in itertools.combinations(range(m), k))]
            assert nf[b] == (max(kf) if kf else 1), (c, f)
    # threshold: S = {i : c_i >= tau}, else the single most confident (lowest position)
    for tau in (0.5, 0.75, 0.9, 1.0):
        n, sets, _ = run_profiles(o, profiles, THRESHOLD, tau)
        for b, c in enumerate(profiles):
            S = {i for i, ci in enumerate(c) if ci >= tau}
            if not S:
                top = max(c)
                S = {min(i for i, ci in enumerate(c) if ci == top)}
            assert sets[b] == S and n[b] == len(S), (c, tau)


def pin_equal_confidence_reduction(o):
    """Cor. factor-reduction: on flat profiles Frechet(delta) == Factor(f = 1 - delta) for
    delta in [0, 1] (dyadic confidences, so every boundary case is exact)."""
    profiles = [[k / 1024.0] * m for k in range(4, 1025, 4) for m in range(1, 13)]
    for delta in (0.0, 0.125, 0.25, 0.5, 0.75, 1.0):
        n_p, sets_p, _ = run_profiles(o, profiles, PROFILE, 1.0 - delta)
        n_f, sets_f, _ = run_profiles(o, profiles, FACTOR, 1.0 - delta)
        assert np.array_equal(n_p, n_f), delta
        assert sets_p == sets_f
        # Eq. equal_conf_threshold: accepted iff c > 1 - (1 - delta)/(n+1)
        for b, p in enumerate(profiles):
            c, m = p[0], len(p)
            acc = [n for n in range(1, m + 1) if c > 1.0 - (1.0 - delta) / (n + 1)]
            assert n_p[b] == (max(acc) if acc else 1), (c, m, delta)


def pin_heterogeneity_bonus(o):
    """Prop. heterogeneity-bonus: G_n = F_n + B_n when L_n > 0, with B_n >= 0 and B_n = 0
    iff the prefix is flat; in general G_n >= F_n + B_n (the max with zero only raises L_n)."""
    rng = np.random.default_rng(7)
    profiles = _random_profiles(rng, 300, 16, dyadic=256)
    profiles += [[0.5] * 6, [1.0] * 3, [0.75, 0.75, 0.5]]
    for p in profiles:
        c = np.array(sorted(p, reverse=True))
        Ln, Un, Gn = o.frechet_scan(c)
        for n in range(1, len(c) + 1):
            F = (n + 1) * c[n - 1] - n
            Bn = float(np.sum(c[: n - 1] - c[n - 1]))
            assert Bn >= 0.0
            assert (Bn == 0.0) == bool(np.all(c[:n] == c[n - 1]))
            if Ln[n - 1] > 0:
                assert Gn[n - 1] == F + Bn, (c, n)
            else:
                assert Gn[n - 1] >= F + Bn, (c, n)


def pin_matched_dominance(o):
    """Cor. matched-factor-dominance: factor(f = 1 - delta) accepting n implies Frechet(delta)
    accepting n, so n*_profile >= n*_factor; Frechet accepts and factor rejects whenever
    F_n <= delta < F_n + B_n."""
    rng = np.random.default_rng(3)
    profiles = _random_profiles(rng, 400, 32)
    for delta in np.linspace(0.0, 1.0, 11):
        n_p, _, _ = run_profiles(o, profiles, PROFILE, 1.0 - delta)
        n_f, _, _ = run_profiles(o, profiles, FACTOR, 1.0 - delta)
        assert np.all(n_p >= n_f), delta
    for p in profiles[:150]:
        c = np.array(sorted(p, reverse=True))
        _, _, Gn = o.frechet_scan(c)
        for delta in (0.0, 0.1, 0.25, 0.5):
            for n in range(1, len(c) + 1):
                F = (n + 1) * c[n - 1] - n
                Bn = float(np.sum(c[: n - 1] - c[n - 1]))
                if F + 1e-12 <= delta < F + Bn - 1e-12:
                    assert Gn[n - 1] > delta
                    assert not ((n + 1) * (1 - c[n - 1]) < 1 - delta)


def pin_greedy_equivalence(o):
    """Thm. frechet-greedy on random joint distributions over V^n (V = 3, n <= 3): whenever
    L_n > U_n for the marginals, the tuple of marginal argmaxes is the unique joint mode."""
    rng = np.random.default_rng(13)
    hits = 0
    for trial in range(6000):
        n = 2 + trial % 2
        P = rng.dirichlet(np.full(3 ** n, 0.08)).reshape((3,) * n)
        marg = [P.sum(axis=tuple(a for a in range(n) if a != i)) for i in range(n)]
        xs = tuple(int(np.argmax(mg)) for mg in marg)
        c = np.array(sorted((float(mg.max()) for mg in marg), reverse=True))
        Ln, Un, _ = o.frechet_scan(c)
        if Ln[-1] > Un[-1]:
            hits += 1
            others = np.delete(P.reshape(-1), np.ravel_multi_index(xs, P.shape))
            assert P[xs] > others.max(), (P, xs)
    assert hits > 300, hits


def pin_monotone_prefix(o):
    """G_n is non-increasing and (n+1)(1 - c_(n)) non-decreasing, so every accepted set is a
    prefix and n* (a max, Sec. 3) equals the first rejected size minus one."""
    rng = np.random.default_rng(17)
    profiles = _random_profiles(rng, 300, 40)
    for p in profiles:
        c = np.array(sorted(p, reverse=True))
        _, _, Gn = o.frechet_scan(c)
        assert np.all(np.diff(Gn) <= 1e-12)
    for f in (1.0, 0.75, 0.3):
        n, _, _ = run_profiles(o, profiles, PROFILE, f)
        for b, p in enumerate(profiles):
            c = np.array(sorted(p, reverse=True))
            _, _, Gn = o.frechet_scan(c)
            first_fail = next((k for k in range(len(c)) if not Gn[k] > 1.0 - f), len(c))
            assert n[b] == max(first_fail, 1)


def pin_special_cases(o):
    """m = 1 -> n* = 1 in every mode; all c = 1 -> n* = m (profile delta < 1, factor f > 0);
    all c < 1/2 -> profile n* = 1 for delta >= 0; empty rows commit nothing."""
    rng = np.random.default_rng(19)
    singles = [[float(x)] for x in rng.random(50)]
    for mode, param in ((PROFILE, 1.0), (PROFILE, 0.75), (FACTOR, 0.75), (FACTOR, 2.0),
                        (THRESHOLD, 0.9), (THRESHOLD, 0.1)):
        n, sets, _ = run_profiles(o, singles, mode, param)
        assert np.all(n == 1) and all(s == {0} for s in sets)
    ones = [[1.0] * m for m in range(1, 20)]
    for f in (0.01, 0.5, 1.0):
        n, _, _ = run_profiles(o, ones, PROFILE, f)
        assert list(n) == list(range(1, 20))
        n, _, _ = run_profiles(o, ones, FACTOR, f)
        assert list(n) == list(range(1, 20))
    low = [list(map(float, rng.uniform(0.0, 0.499, int(rng.integers(1, 30))))) for _ in range(80)]
    for f in (1.0, 0.75, 0.0):
        n, _, _ = run_profiles(o, low, PROFILE, f)
        assert np.all(n == 1)
    conf = np.zeros((3, 4))
    mask = np.zeros((3, 4), np.uint8)
    mask[1, 2] = 1
    conf[1, 2] = 0.3
    tok = np.full((3, 4), 5, np.int32)
    r = o.select_from_conf(conf, tok, mask, PROFILE, 1.0)
    assert list(r["n"]) == [0, 1, 0] and r["commit"].sum() == 1 and r["commit"][1, 2] == 1


def pin_reveal_and_ties(o):
    """Alg. 1 reveal: committed positions take their token and leave the mask; nothing else
    is written.  Equal confidences at the commit boundary go to the lower position."""
    B, L = 2, 8
    conf = np.zeros((B, L))
    mask = np.zeros((B, L), np.uint8)
    tok = (np.arange(B * L, dtype=np.int32) * 7).reshape(B, L)
    conf[0, [5, 2, 7, 0]] = [0.9, 0.9, 0.9, 0.2]
    mask[0, [5, 2, 7, 0]] = 1
    conf[1, [1, 6]] = [0.95, 0.99]
    mask[1, [1, 6]] = 1
    sentinel = np.full((B, L), -77, np.int32)
    # threshold 0.95 -> row 0 has no passing position: fallback to the lowest of the ties
    r = o.select_from_conf(conf, tok, mask, THRESHOLD, 0.95, out_tokens=sentinel)
    assert np.nonzero(r["commit"][0])[0].tolist() == [2]
    assert np.nonzero(r["commit"][1])[0].tolist() == [1, 6]
    for b in range(B):
        for l in range(L):
            if r["commit"][b, l]:
                assert r["tokens"][b, l] == tok[b, l] and r["mask"][b, l] == 0
            else:
                assert r["tokens"][b, l] == -77 and r["mask"][b, l] == mask[b, l]
    # factor f = 0.5 on three equal 0.9's: (n+1)*0.1 < 0.5 for n <= 3 -> all three
    r = o.select_from_conf(conf, tok, mask, FACTOR, 0.5)
    assert np.nonzero(r["commit"][0])[0].tolist() == [2, 5, 7]
    # factor f = 0.35: n = 2 accepted (0.3), n = 3 rejected (0.4) -> positions 2 and 5
    r = o.select_from_conf(conf, tok, mask, FACTOR, 0.35)
    assert np.nonzero(r["commit"][0])[0].tolist() == [2, 5]


def pin_end_to_end(o):
    """Whole step on logits: confidences from torch float64, then the brute-force rule."""
    rng = np.random.default_rng(23)
    B, L, V = 4, 6, 300
    x = rng.normal(0.0, 1.0, (B, L, V)).astype(np.float32)
    for b in range(B):
        for l in range(L):
            x[b, l, rng.integers(V)] += rng.uniform(4.0, 14.0)
    mask = (rng.random((B, L)) < 0.8).astype(np.uint8)
    t = widen(x)
    c_ref = torch.exp(t.max(-1).values - torch.logsumexp(t, -1)).numpy()
    for f in (1.0, 0.75):
        r = o.select(x, mask, PROFILE, f)
        for b in range(B):
            pos = [l for l in range(L) if mask[b, l]]
            if not pos:
                assert r["n"][b] == 0
                continue
            c = [float(c_ref[b, l]) for l in pos]
            ks = [k for k in range(1, len(c) + 1)
                  if max(G_of_subset(S) for S in itertools.combinations(c, k)) > 1.0 - f]
            assert r["n"][b] == (max(ks) if ks else 1)


def _robust_profiles(rng, count, m_max, dyadic, eta_lo=0.0):
    out = []
    for _ in range(count):
        m = int(rng.integers(1, m_max + 1))
        lo = int(np.ceil(eta_lo * dyadic))
        out.append(list(map(float, rng.integers(max(lo, 1), dyadic + 1, m) / dyadic)))
    return out


def _run_robust(o, profiles, param, eta, eta_pos=None):
    B = len(profiles)
    L = max(len(p) for p in profiles)
    conf = np.zeros((B, L))
    mask = np.zeros((B, L), np.uint8)
    tok = np.arange(B * L, dtype=np.int32).reshape(B, L)
    for b, p in enumerate(profiles):
        conf[b, :len(p)] = p
        mask[b, :len(p)] = 1
    r = o.select_robust_from_conf(conf, tok, mask, param, eta, eta_pos)
    return r["n"], [set(np.nonzero(r["commit"][b])[0].tolist()) for b in range(B)], r


def pin_robust_zero_eta_is_profile(o):
    """App. C with eta = 0 is the plain profile rule (c_low = c_hat)."""
    rng = np.random.default_rng(29)
    profiles = _random_profiles(rng, 200, 24)
    for f in (1.0, 0.75, 0.5):
        n_r, s_r, _ = _run_robust(o, profiles, f, 0.0)
        n_p, s_p, _ = run_profiles(o, profiles, PROFILE, f)
        assert np.array_equal(n_r, n_p) and s_r == s_p


def pin_robust_negative_allowance_is_zero(o):
    """App. C takes allowances eta >= 0; the library reads a negative or NaN per-position
    allowance as 0, so rows whose allowances are all negative or NaN decide as the plain
    profile rule, and a row mixing such entries with zeros does too."""
    rng = np.random.default_rng(31)
    profiles = _random_profiles(rng, 120, 24)
    L = max(len(p) for p in profiles)
    eta_pos = -rng.uniform(0.01, 2.0, (len(profiles), L))
    eta_pos[::3, ::2] = np.nan
    eta_pos[1::3, 1::2] = 0.0
    for f in (1.0, 0.75):
        n_r, s_r, _ = _run_robust(o, profiles, f, 0.0, eta_pos)
        n_p, s_p, _ = run_profiles(o, profiles, PROFILE, f)
        assert np.array_equal(n_r, n_p) and s_r == s_p


def pin_robust_calibration_penalty(o):
    """Cor. calibration-penalty: with uniform eta and no clipping (every c_hat >= eta),
    G^(eta)_n = G_hat_n - (n+1) eta where the robust lower bound is active, and both sides
    reject otherwise (delta >= 0), so n*_robust = max{n : G_hat_n - (n+1) eta > delta}.
    Dyadic values keep every comparison exact."""
    rng = np.random.default_rng(31)
    for eta in (1 / 64, 1 / 16, 3 / 32):
        profiles = _robust_profiles(rng, 150, 12, 256, eta_lo=eta)
        for f in (1.0, 0.75, 0.5):
            delta = 1.0 - f
            n_r, _, _ = _run_robust(o, profiles, f, eta)
            for b, p in enumerate(profiles):
                c = np.array(sorted(p, reverse=True))
                _, _, G = o.frechet_scan(c)
                acc = [n for n in range(1, len(c) + 1) if G[n - 1] - (n + 1) * eta > delta]
                assert n_r[b] == (max(acc) if acc else 1), (p, eta, f)


def _G_low(cs):
    k = len(cs)
    return max(0.0, sum(cs) - (k - 1)) - (1.0 - min(cs))


def pin_robust_bruteforce(o):
    """Eq. robust_L_U over all subsets with per-position allowances: n* is the largest size
    with an admissible subset, and the committed set attains the best robust score."""
    rng = np.random.default_rng(37)
    B, m = 120, 7
    profiles = [list(map(float, rng.integers(1, 65, m) / 64)) for _ in range(B)]
    eta_pos = rng.integers(0, 9, (B, m)) / 64
    for f in (1.0, 0.75):
        delta = 1.0 - f
        n_r, sets, _ = _run_robust(o, profiles, f, 0.0, eta_pos)
        for b, p in enumerate(profiles):
            low = [max(0.0, p[i] - eta_pos[b, i]) for i in range(m)]
            best = {k: max(_G_low([low[i] for i in S])
                           for S in itertools.combinations(range(m), k))
                    for k in range(1, m + 1)}
            ks = [k for k in range(1, m + 1) if best[k] > delta]
            want = max(ks) if ks else 1
            assert n_r[b] == want, (p, eta_pos[b], f)
            if ks:
                assert _G_low([low[i] for i in sorted(sets[b])]) == best[want]


def pin_robust_monotone_and_clipped(o):
    """A larger allowance never commits more (uniform eta); when every confidence is at or
    below eta all lower confidences are 0 and the progress convention commits the lowest
    position."""
    rng = np.random.default_rng(41)
    profiles = _random_profiles(rng, 200, 20)
    prev = None
    for eta in (0.0, 0.01, 0.05, 0.1, 0.3):
        n_r, _, _ = _run_robust(o, profiles, 1.0, eta)
        if prev is not None:
            assert np.all(n_r <= prev)
        prev = n_r
    low = [[0.2, 0.1, 0.3], [0.05]]
    n_r, sets, _ = _run_robust(o, low, 0.75, 0.3)
    assert list(n_r) == [1, 1] and sets == [{0}, {0}]


def pin_bonus_terms(o):
    """Eq. heterogeneity_decomp: F_n and B_n against the hand-worked profiles, and
    G_n = F_n + B_n whenever L_n > 0 with B_n >= 0 (zero iff the prefix is flat)."""
    with open(GOLDEN) as fh:
        cases = json.load(fh)["cases"]
    for case in cases:
        F, Bn = o.bonus_terms(np.array(case["c_sorted"]))
        np.testing.assert_allclose(F, case["F"], atol=1e-12)
        np.testing.assert_allclose(Bn, case["Bn"], atol=1e-12)
    rng = np.random.default_rng(43)
    for p in _random_profiles(rng, 200, 16, dyadic=256):
        c = np.array(sorted(p, reverse=True))
        Ln, _, Gn = o.frechet_scan(c)
        F, Bn = o.bonus_terms(c)
        assert np.all(Bn >= 0)
        for n in range(1, len(c) + 1):
            assert (Bn[n - 1] == 0) == bool(np.all(c[:n] == c[n - 1]))
            if Ln[n - 1] > 0:
                assert Gn[n - 1] == F[n - 1] + Bn[n - 1]
    # the row-level terms follow the selection's order
    conf = np.array([[0.3, 0.9, 0.0, 0.9, 0.7]])
    mask = np.array([[1, 1, 0, 1, 1]], np.uint8)
    t = o.profile_terms(conf, mask)
    assert t["order"][0].tolist() == [1, 3, 4, 0, -1]
    _, _, G = o.frechet_scan(np.array([0.9, 0.9, 0.7, 0.3]))
    np.testing.assert_allclose(t["G"][0, :4], G, atol=0)
    assert np.isnan(t["G"][0, 4]) and np.isnan(t["B"][0, 4])



MARGINS = os.path.join(os.path.dirname(GOLDEN), "decision_margins.json")


def _select_any(o, conf, mask, rule, param, eta=None, eta_pos=None):
    tok = np.arange(conf.size, dtype=np.int32).reshape(conf.shape)
    if rule == "robust":
        return o.select_robust_from_conf(conf, tok, mask, param, 0.0 if eta is None else eta,
                                         eta_pos)
    mode = {"profile": PROFILE, "factor": FACTOR, "threshold": THRESHOLD}[rule]
    return o.select_from_conf(conf, tok, mask, mode, param)


def pin_decision_margin_hand_worked(o):
    """The decision margin (the distance that decides which rows parity may excuse) on
    profiles whose margin is worked out by hand (tests/golden/decision_margins.json): the
    rule quantity at n* and n* + 1, the rank gap, a tie block straddling n* with its
    neighbour above or below closest, the progress fallback, n* = m, and the robust rule's
    distance to a clipping point.  Every value is a multiple of 1/64, so the comparison is
    exact."""
    with open(MARGINS) as fh:
        cases = json.load(fh)["cases"]
    for case in cases:
        conf = np.array([case["conf_by_pos"]], np.float64)
        mask = (conf > 0).astype(np.uint8)
        r = _select_any(o, conf, mask, case["rule"], case["param"], case.get("eta"))
        assert r["n"][0] == case["nstar"], (case["name"], r["n"][0])
        assert np.nonzero(r["commit"][0])[0].tolist() == case["commit_pos"], case["name"]
        assert r["margin"][0] == case["margin"], (case["name"], r["margin"][0], case["margin"])


def _tie_profile(rng, m, grid=256):
    """m dyadic confidences in [8, 248] / grid with planted equal groups (ties across
    positions), so that tie blocks often straddle the boundary."""
    k = int(rng.integers(1, m + 1))
    levels = rng.choice(np.arange(8, grid - 7), size=k, replace=False) / grid
    c = levels[rng.integers(0, k, m)]
    return c


def pin_decision_margin_stability(o):
    """What the margin means: no perturbation that moves every confidence by less than
    margin / (n* + 2), and moves equal confidences together (bit-identical inputs give
    bit-identical confidences on both sides), can change n* or the committed set.  The rule
    quantity at rank n moves by at most (n + 1) times the perturbation (sorting is
    1-Lipschitz in the largest change; L_n sums n confidences, U_n one), so the decisions at
    n* and n* + 1 keep their sides, the rules' monotonicity in n carries them to every other
    n, and gaps above twice the perturbation keep the committed ranks (whole tie blocks
    move as one) in place.  For the robust rule the groups are equal lower confidences and
    the perturbation is applied to c_hat, which stays on its side of its clipping point.
    Checked on random dyadic profiles with planted ties, for every rule, with the
    perturbations that push every group up, every group down, or neighbouring groups apart
    and together."""
    rng = np.random.default_rng(61)
    rules = [("profile", (1.0, 0.875, 0.75, 0.5)), ("factor", (0.5, 1.0, 1.5, 2.0)),
             ("threshold", (0.5, 0.75, 0.875)), ("robust", (1.0, 0.75))]
    checked = 0
    for trial in range(600):
        rule, params = rules[trial % len(rules)]
        param = float(params[rng.integers(len(params))])
        m = int(rng.integers(1, 9))
        L = m + int(rng.integers(0, 3))
        c_hat = _tie_profile(rng, m)
        pos = rng.permutation(L)[:m]
        conf = np.zeros((1, L))
        conf[0, pos] = c_hat
        mask = (conf > 0).astype(np.uint8)
        eta_pos = None
        if rule == "robust":
            eta_pos = np.zeros((1, L))
            eta_pos[0, pos] = rng.integers(0, 9, m) / 256 if trial % 8 < 4 else 6 / 256
            if trial % 3 == 0:  # some allowances just above or below their confidence
                near = rng.random(m) < 0.5
                eta_pos[0, pos[near]] = c_hat[near] + rng.integers(-2, 3, near.sum()) / 256
        r0 = _select_any(o, conf, mask, rule, param, eta_pos=eta_pos)
        M, nstar = float(r0["margin"][0]), int(r0["n"][0])
        if not M > 0:
            continue
        eps = min(0.999 * M / (nstar + 2), 4 / 256)
        low = conf[0] if eta_pos is None else np.maximum(conf[0] - eta_pos[0], 0.0)
        # groups: equal (lower) confidences move together; clipped positions stay clipped
        keys = {}
        group = np.full(L, -1)
        for l in pos:
            key = low[l] if low[l] > 0 else ("clip", int(l))
            group[l] = keys.setdefault(key, len(keys))
        order = sorted(keys.items(), key=lambda kv: -(kv[0] if not isinstance(kv[0], tuple)
                                                       else 0.0))
        rank_of = {g: i for i, (_, g) in enumerate(order)}
        signs = [np.ones(len(keys)), -np.ones(len(keys)),
                 np.array([(-1.0) ** rank_of[g] for g in range(len(keys))]),
                 np.array([-((-1.0) ** rank_of[g]) for g in range(len(keys))]),
                 rng.choice([-1.0, 1.0], len(keys))]
        for sg in signs:
            pert = conf.copy()
            pert[0, pos] += eps * sg[group[pos]]
            r1 = _select_any(o, pert, mask, rule, param, eta_pos=eta_pos)
            assert r1["n"][0] == nstar, (rule, param, c_hat, eps, M)
            assert np.array_equal(r1["commit"], r0["commit"]), (rule, param, c_hat, eps, M)
        checked += 1
    assert checked > 400


ALL_PINS = [
    pin_confidence_vs_torch, pin_confidence_closed_forms, pin_nonfinite, pin_hand_worked,
    pin_bruteforce_subsets, pin_equal_confidence_reduction, pin_heterogeneity_bonus,
    pin_matched_dominance, pin_greedy_equivalence, pin_monotone_prefix, pin_special_cases,
    pin_reveal_and_ties, pin_end_to_end, pin_robust_zero_eta_is_profile,
    pin_robust_calibration_penalty, pin_robust_bruteforce, pin_robust_monotone_and_clipped,
    pin_robust_negative_allowance_is_zero,
    pin_bonus_terms, pin_half_widening, pin_extreme_magnitudes,
    pin_decision_margin_hand_worked, pin_decision_margin_stability,
]
