"""Pins of the oracle's detector suite: the per-token scores of the pivot
r = u (Aaronson, the U-score, Li et al.'s optimal Gumbel score, Lattimore's
truncated power law; App. D) and the segment p-values (the exact Gamma tail of
S_A and the Chernoff bound on the U-score; App. D.2, App. E)."""
from __future__ import annotations

import math

import mpmath
import numpy as np
import pytest
from scipy import stats

import oracle

W_GRID = np.unique(np.concatenate([np.linspace(0, 2 ** 32 - 1, 200001).astype(np.uint64),
                                   np.arange(0, 4096, dtype=np.uint64),
                                   (2 ** 32 - 1 - np.arange(0, 4096, dtype=np.uint64))]))


def _ids(n, seed):
    rng = np.random.default_rng(seed)
    return (rng.integers(0, 2 ** 63, n, dtype=np.uint64), rng.integers(0, 2 ** 63, n, dtype=np.uint64),
            rng.integers(0, 2 ** 31, n, dtype=np.uint32))


# ---------------------------------------------------------------- p-values

@pytest.mark.parametrize("S", [0.0, 0.3, 1.0, 7.5, 40.0])
def test_gamma_tail_single_token_is_exp(S):
    # M = 1: P(Exp(1) >= S) = e^-S
    assert oracle.gamma_tail_logp(1, S) == pytest.approx(-S, abs=1e-15)


@pytest.mark.parametrize("M,ratio", [(2, 0.5), (5, 1.0), (16, 1.3), (64, 2.0), (128, 0.8), (300, 1.0),
                                     (1000, 1.5), (20, 12.0)])
def test_gamma_tail_matches_the_regularised_upper_incomplete_gamma(M, ratio):
    # extreme watermarked tails included (ln p down to ~ -200)
    S = ratio * M
    mpmath.mp.dps = 50
    want = float(mpmath.log(mpmath.gammainc(M, S, mpmath.inf, regularized=True)))
    assert oracle.gamma_tail_logp(M, S) == pytest.approx(want, rel=1e-11, abs=1e-12)


@pytest.mark.parametrize("M", [1 << 18, 1 << 20, (1 << 24) + 5])
@pytest.mark.parametrize("c", [-1.5, 0.0, 3.0])
def test_gamma_tail_of_long_segments_matches_scipy(M, c):
    # segments of 2^18 .. 2^24 tokens, S within a few standard deviations of M, against scipy's
    # regularised upper incomplete gamma (which agrees with mpmath to 1e-13 where mpmath
    # converges).  The oracle's running log-term is compensated; what remains is its
    # log-sum-exp accumulator, rescaled at each of the ~S rising terms with one rounding each:
    # ~1e-8 at 2^24 tokens, far inside the GPU parity tolerance of 2e-6
    sp = pytest.importorskip("scipy.special")
    S = M + c * math.sqrt(M) + 0.31
    want = math.log(sp.gammaincc(M, S))
    assert oracle.gamma_tail_logp(M, S) == pytest.approx(want, rel=1e-10, abs=5e-8)


def test_gamma_tail_p_values_are_uniform_under_the_null():
    # S_A of M independent Exp(1) scores: the p-value is U(0,1) (App. D.2)
    rng = np.random.default_rng(1)
    M = 37
    S = rng.exponential(1.0, (4000, M)).sum(1)
    p = np.exp([oracle.gamma_tail_logp(M, s) for s in S])
    assert stats.kstest(p, "uniform").pvalue > 1e-3


def _irwin_hall_tail(M, x):
    # P(U_1 + ... + U_M >= x), exact (Irwin-Hall), in rationals
    from fractions import Fraction
    x = Fraction(x)
    cdf = sum((-1) ** k * math.comb(M, k) * (x - k) ** M for k in range(0, int(x) + 1)) / math.factorial(M)
    return float(1 - cdf)


@pytest.mark.parametrize("M,frac", [(1, 0.9), (3, 0.7), (6, 0.8), (10, 0.66), (12, 0.9)])
def test_chernoff_u_bound_is_the_minimum_and_bounds_the_exact_tail(M, frac):
    S = frac * M
    got = oracle.chernoff_u_logp(M, S)
    lam = np.linspace(1e-6, 200, 400001)
    f = M * np.log(np.expm1(lam) / lam) - lam * S
    assert got <= f.min() + 1e-12                 # no worse than a fine grid
    assert got >= f.min() - 1e-6                  # and the grid's spacing bounds the gap
    exact = _irwin_hall_tail(M, S)
    assert got >= math.log(exact) - 1e-12         # Chernoff is an upper bound on the tail


def test_chernoff_u_bound_trivial_below_half_and_infinite_at_the_top():
    for M in (1, 7, 50):
        assert oracle.chernoff_u_logp(M, 0.5 * M) == 0.0
        assert oracle.chernoff_u_logp(M, 0.2 * M) == 0.0
        assert oracle.chernoff_u_logp(M, float(M)) == -math.inf


# ---------------------------------------------------------------- per-token scores

def test_aaronson_and_u_scores_are_the_pivot_transforms():
    for w in (0, 1, 12345, 2 ** 31 - 1, 2 ** 31, 2 ** 32 - 2, 2 ** 32 - 1):
        u = (w + 0.5) / 2 ** 32
        assert oracle.score_kind(w, oracle.AARONSON) == pytest.approx(-math.log1p(-u), rel=1e-13)
        assert oracle.score_kind(w, oracle.U_SCORE) == pytest.approx(u, rel=1e-15)


@pytest.mark.parametrize("delta", [0.1, 0.3, 0.5, 0.62, 0.9])
def test_li_score_is_a_null_likelihood_ratio(delta):
    # h* = ln(dP_Delta*/dP_0) of the pivot, so E_null[exp(h*)] = 1; h* -> ln(k + [q > 0]) as r -> 1
    w = W_GRID
    u = (w.astype(np.float64) + 0.5) / 2 ** 32
    h = np.array([oracle.score_kind(int(x), oracle.LI, delta) for x in w])
    assert np.trapezoid(np.exp(h), u) == pytest.approx(1.0, abs=2e-4)
    k = math.floor(1 / (1 - delta))
    q = 1 - k * (1 - delta)
    assert h[-1] == pytest.approx(math.log(k + (1 if q > 1e-12 else 0)), abs=1e-6)
    assert np.all(np.diff(h) >= -1e-12)  # increasing in r


def test_li_score_closed_form_when_one_over_one_minus_delta_is_integer():
    # Delta = 1/2, 2/3, 3/4: q = 0 and h* = ln k + (Delta/(1-Delta)) ln r
    for delta, k in ((0.5, 2), (2 / 3, 3), (0.75, 4)):
        for w in (5, 2 ** 20, 2 ** 31 + 7, 2 ** 32 - 9):
            r = (w + 0.5) / 2 ** 32
            want = math.log(k) + delta / (1 - delta) * math.log(r)
            assert oracle.score_kind(w, oracle.LI, delta) == pytest.approx(want, rel=1e-9, abs=1e-12)


@pytest.mark.parametrize("eps", [1e-4, 1e-2, 0.2, 1.0])
def test_power_law_score_is_centred_and_truncated(eps):
    w = W_GRID
    u = (w.astype(np.float64) + 0.5) / 2 ** 32
    h = np.array([oracle.score_kind(int(x), oracle.PL, eps) for x in w])
    # E_null[h] = 0 (the centring 2 - sqrt(eps)): the integral of min(eps^-1/2, (1-r)^-1/2) is 2 - sqrt(eps)
    assert np.trapezoid(h, u) == pytest.approx(0.0, abs=5e-4)
    assert h.max() == pytest.approx(eps ** -0.5 - (2 - eps ** 0.5), rel=1e-12)
    r = 0.3
    w0 = int(r * 2 ** 32)
    want = min(eps ** -0.5, (1 - (w0 + 0.5) / 2 ** 32) ** -0.5) - (2 - eps ** 0.5)
    assert oracle.score_kind(w0, oracle.PL, eps) == pytest.approx(want, rel=1e-12)


def test_detector_pass_sums_and_p_values_per_segment():
    n = 3000
    rng = np.random.default_rng(3)
    tok = rng.integers(0, 128256, n, dtype=np.int32)
    key, ctx, pos = _ids(n, 4)
    seg = np.array([0, 1, 2, 130, 1000, 1000, 2999, 3000], np.int64)
    for kind, param in ((oracle.AARONSON, 0), (oracle.U_SCORE, 0), (oracle.LI, 0.4), (oracle.PL, 0.05)):
        sc, sums, logp = oracle.wm_detect(tok, key, ctx, pos, seg, kind, param)
        for g in range(len(seg) - 1):
            a, b = seg[g], seg[g + 1]
            assert sums[g] == pytest.approx(sc[a:b].sum(), rel=1e-12, abs=1e-12)
            M = b - a
            if M == 0:
                assert logp[g] == 0.0
            elif kind == oracle.AARONSON:
                assert logp[g] == oracle.gamma_tail_logp(M, sums[g])
            elif kind == oracle.U_SCORE:
                assert logp[g] == oracle.chernoff_u_logp(M, sums[g])
            else:
                assert math.isnan(logp[g])
        w = [oracle.word(int(key[t]), int(ctx[t]), int(pos[t]), int(tok[t])) for t in range(0, n, 97)]
        assert np.allclose(sc[::97], [oracle.score_kind(x, kind, param) for x in w], rtol=1e-15)
