"""Closed forms that pin the oracle (test infrastructure only).

Each function restates a quantity the paper fixes, in plain numpy/scipy, for
small vocabularies (O(V^2) loops are fine here):

* ``accept_k1``       single-draft coupling probability of the exponential race,
                      sum_i 1 / sum_j max(p_j/p_i, q_j/q_i): the list-matching
                      bound of App. B.3 at B = 1, which for one draft is the exact
                      probability that argmin E/q = argmin E/p.
* ``alpha``           alpha_i = p_i sum_j (q_j/q_i - p_j/p_i)_+   (Thm B.2).
* ``accept_iid``      1 - sum_i p_i (alpha_i / (1 + alpha_i))^K.  Thm B.2 states
                      it as a lower bound; for the multi-arrival list of the
                      direct finite-support MPFR algorithm it is exact (given
                      Y = i and E_{i,1} = e, every other token adds
                      Poisson(e (q_j/q_i - p_j/p_i)_+) arrivals ahead of i).
* ``accept_distinct`` the same conditioning for the K smallest first arrivals:
                      token j lands ahead of i with probability
                      1 - exp(-e (q_j/q_i - p_j/p_i)_+), a Poisson-binomial count.
* ``alpha_sorted``    the same alpha for a full vocabulary in O(V log V): the
                      term (q_j/q_i - p_j/p_i)_+ is positive exactly when
                      q_j/p_j > q_i/p_i, so with the tokens ordered by
                      rho = q/p, alpha_i = (p_i/q_i) Q_i - P_i where Q_i and P_i
                      sum q and p over the tokens of strictly larger rho.
* ``accept_iid_full`` ``accept_iid`` through ``alpha_sorted`` (depth-0 acceptance
                      of the benchmark trees at V = 128256).
* ``bound_thm41``     1 - sum_i p_i (p_i / (p_i + q_i))^K              (Thm 4.1, Eq. 5).
* ``bound_lml``       sum_i p_i K / (K + alpha_i)                      (App. B.3 rewrite).
* ``bound_no_comm``   (1 - TV) / (1 + TV) (Eq. 3): the worst-case value of a
                      communication-free coupling; the race attains at least it
                      for every pair, so it bounds ``accept_k1`` from below.
* ``pivot_cdf_h1``    P(r <= x) = sum_v p_v x^(1/p_v) for the winner's pivot (App. D.3).
* ``aaronson_mean_lb`` 1 + (pi^2/6 - 1) H(p) lower bound on E[A_t]     (Sec. 3.3, App. D.1).
"""
from __future__ import annotations

import math

import numpy as np
from scipy import integrate


def softmax(logits, T: float = 1.0):
    z = np.asarray(logits, np.float64) / T
    z = z - np.max(z)
    e = np.exp(z)
    return e / e.sum()


def accept_k1(p, q) -> float:
    p = np.asarray(p, np.float64)
    q = np.asarray(q, np.float64)
    tot = 0.0
    for i in range(p.size):
        if p[i] <= 0 or q[i] <= 0:
            continue
        den = 0.0
        for j in range(p.size):
            den += max(p[j] / p[i], q[j] / q[i])
        tot += 1.0 / den
    return tot


def alpha(p, q):
    p = np.asarray(p, np.float64)
    q = np.asarray(q, np.float64)
    a = np.zeros_like(p)
    for i in range(p.size):
        s = 0.0
        for j in range(p.size):
            s += max(q[j] / q[i] - p[j] / p[i], 0.0)
        a[i] = p[i] * s
    return a


def alpha_sorted(p, q):
    """alpha_i = p_i sum_j (q_j/q_i - p_j/p_i)_+ for tokens with p_i, q_i > 0, in
    O(V log V) (tokens with p_i = 0 get alpha 0; they carry no target mass)."""
    p = np.asarray(p, np.float64)
    q = np.asarray(q, np.float64)
    a = np.zeros_like(p)
    live = (p > 0) & (q > 0)
    pl, ql = p[live], q[live]
    rho = ql / pl
    order = np.argsort(rho, kind="stable")
    rs, ps, qs = rho[order], pl[order], ql[order]
    # suffix sums over strictly larger rho: sum over positions after the last tie of each value
    cq = np.concatenate([np.cumsum(qs[::-1])[::-1], [0.0]])
    cp = np.concatenate([np.cumsum(ps[::-1])[::-1], [0.0]])
    after = np.searchsorted(rs, rs, side="right")
    al = np.maximum(ps / qs * cq[after] - cp[after], 0.0)
    # tokens with q_j > 0 = p_j also come ahead of every live i (rho_j = inf)
    inf_q = float(q[(p <= 0) & (q > 0)].sum())
    al = al + ps / qs * inf_q
    out = np.zeros(order.size)
    out[order] = al
    a[live] = out
    # tokens with p_i > 0 = q_i can never be drafted: alpha = inf (never accepted)
    a[(p > 0) & (q <= 0)] = np.inf
    return a


def accept_iid_full(p, q, K: int) -> float:
    p = np.asarray(p, np.float64)
    a = alpha_sorted(p, q)
    frac = np.where(np.isinf(a), 1.0, a / (1.0 + np.where(np.isinf(a), 0.0, a)))
    return float(1.0 - np.sum(p * frac ** K))


def accept_iid(p, q, K: int) -> float:
    p = np.asarray(p, np.float64)
    a = alpha(p, q)
    return float(1.0 - np.sum(p * (a / (1.0 + a)) ** K))


def accept_iid_integral(p, q, K: int) -> float:
    """The IID acceptance computed by integrating the conditional Poisson tail
    (no closed-form step): sum_i int_0^inf e^{-e/p_i} P(Poisson(e a_i/p_i) <= K-1) de."""
    p = np.asarray(p, np.float64)
    a = alpha(p, q)
    tot = 0.0
    for i in range(p.size):
        lam = a[i] / p[i]

        def f(e, lam=lam, pi=p[i]):
            m = e * lam
            cdf = sum(math.exp(-m) * m ** k / math.factorial(k) for k in range(K))
            return math.exp(-e / pi) * cdf

        v, _ = integrate.quad(f, 0.0, np.inf, limit=200)
        tot += v
    return tot


def _poisson_binomial_le(probs, kmax: int) -> float:
    """P(sum of independent Bernoulli(probs) <= kmax) by the textbook DP."""
    dist = np.zeros(len(probs) + 1)
    dist[0] = 1.0
    for pr in probs:
        dist[1:] = dist[1:] * (1.0 - pr) + dist[:-1] * pr
        dist[0] *= 1.0 - pr
    return float(dist[: kmax + 1].sum())


def accept_distinct(p, q, K: int) -> float:
    p = np.asarray(p, np.float64)
    q = np.asarray(q, np.float64)
    tot = 0.0
    for i in range(p.size):
        rates = [max(q[j] / q[i] - p[j] / p[i], 0.0) for j in range(p.size) if j != i]

        def f(e, rates=rates, pi=p[i]):
            probs = [1.0 - math.exp(-e * r) for r in rates]
            return math.exp(-e / pi) * _poisson_binomial_le(probs, K - 1)

        v, _ = integrate.quad(f, 0.0, np.inf, limit=200)
        tot += v
    return tot


def bound_thm41(p, q, K: int) -> float:
    p = np.asarray(p, np.float64)
    q = np.asarray(q, np.float64)
    return float(1.0 - np.sum(p * (p / (p + q)) ** K))


def bound_lml(p, q, K: int) -> float:
    p = np.asarray(p, np.float64)
    a = alpha(p, q)
    return float(np.sum(p * K / (K + a)))


def tv(p, q) -> float:
    return 0.5 * float(np.abs(np.asarray(p, np.float64) - np.asarray(q, np.float64)).sum())


def bound_no_comm(p, q) -> float:
    d = tv(p, q)
    return (1.0 - d) / (1.0 + d)


def pivot_cdf_h1(p, x):
    p = np.asarray(p, np.float64)
    p = p[p > 0]
    x = np.asarray(x, np.float64)
    return np.sum(p[None, :] * x[:, None] ** (1.0 / p[None, :]), axis=1)


def entropy(p) -> float:
    p = np.asarray(p, np.float64)
    p = p[p > 0]
    return float(-(p * np.log(p)).sum())


def aaronson_mean_lb(p) -> float:
    return 1.0 + (math.pi ** 2 / 6.0 - 1.0) * entropy(p)


def plackett_luce_prob(q, seq) -> float:
    """Probability that the K smallest of E_i/q_i come out in the order `seq`."""
    q = np.asarray(q, np.float64)
    rem = 1.0
    pr = 1.0
    for t in seq:
        pr *= q[t] / rem
        rem -= q[t]
    return pr
