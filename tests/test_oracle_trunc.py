"""Pins of the oracle's truncation (top-k, then top-p) before the race.

The experiments sample with top-k = 50 and top-p = 1 (Sec. 6 setup), and a
truncated distribution has a support of at most k tokens (Sec. 4.2).  The
oracle applies truncation as masking (removed tokens get logit -inf, i.e.
P = 0 and E/P = +inf) and then runs the unchanged race.  These tests pin the
masking against library routines and invariants, and the truncated race
against the law of the renormalised truncated distribution.
"""
from __future__ import annotations

import numpy as np
import pytest
import torch
from scipy import stats

import oracle
from oracle import closed_forms as cf


def _ids(n, seed):
    rng = np.random.default_rng(seed)
    key = rng.integers(0, 2 ** 63, n, dtype=np.uint64) * 2 + 1
    ctx = rng.integers(0, 2 ** 63, n, dtype=np.uint64) * 2
    pos = rng.integers(0, 2 ** 31, n, dtype=np.uint32)
    return key, ctx, pos


def _tied_rows(n, V, seed):
    """bf16-rounded rows (many exact ties) with a few NaN and -inf entries."""
    rng = np.random.default_rng(seed)
    x = torch.from_numpy(rng.normal(0, 2, (n, V)).astype(np.float32)).to(torch.bfloat16).float().numpy()
    x[rng.random((n, V)) < 0.02] = -np.inf
    x[rng.random((n, V)) < 0.01] = np.nan
    return x


@pytest.mark.parametrize("k", [1, 3, 50, 200])
def test_top_k_is_the_partition_threshold(k):
    # kept = usable tokens with logit >= the k-th largest usable logit (numpy's partition)
    l = _tied_rows(40, 300, 1 + k)
    out, mg = oracle.truncate_rows(l, top_k=k)
    for r in range(l.shape[0]):
        ok = ~np.isnan(l[r]) & (l[r] > -np.inf)
        vals = l[r][ok]
        thr = np.partition(vals, vals.size - k)[vals.size - k] if vals.size >= k else -np.inf
        want = ok & (np.nan_to_num(l[r], nan=-np.inf) >= thr)
        got = out[r] > -np.inf
        assert np.array_equal(got, want)
        assert np.array_equal(out[r][got], l[r][got])
        assert got.sum() >= min(k, vals.size)
    assert np.all(np.isinf(mg))


def test_no_truncation_is_identity_up_to_nan():
    l = _tied_rows(10, 97, 5)
    for k, p in ((0, 1.0), (97, 1.0), (1000, 1.0)):
        out, _ = oracle.truncate_rows(l, top_k=k, top_p=p)
        assert np.array_equal(out, np.where(np.isnan(l), -np.inf, l))


@pytest.mark.parametrize("top_p", [0.3, 0.8, 0.95])
def test_top_p_on_distinct_logits_matches_sorted_cumsum(top_p):
    # the usual nucleus rule written with torch.sort / softmax / cumsum
    rng = np.random.default_rng(int(top_p * 100))
    n, V, T = 50, 64, 0.8
    l = rng.normal(0, 2, (n, V)).astype(np.float32)
    out, _ = oracle.truncate_rows(l, top_p=top_p, T=T)
    s, idx = torch.sort(torch.from_numpy(l).double() / T, dim=-1)
    cum = torch.softmax(s, dim=-1).cumsum(-1)
    remove = cum <= 1 - top_p
    remove[:, -1] = False
    want = ~torch.zeros_like(remove).scatter(1, idx, remove).numpy()
    assert np.array_equal(out > -np.inf, want)


@pytest.mark.parametrize("top_p", [0.2, 0.6, 0.9])
def test_top_p_keeps_the_smallest_group_prefix_above_the_mass(top_p):
    # kept mass >= top_p, and dropping the lowest kept group would fall below it;
    # tie groups are kept or dropped whole
    l = _tied_rows(60, 200, 7)
    T = 1.3
    k = 40
    topk, _ = oracle.truncate_rows(l, top_k=k)
    out, _ = oracle.truncate_rows(l, top_k=k, top_p=top_p, T=T)
    for r in range(l.shape[0]):
        base = topk[r] > -np.inf
        kept = out[r] > -np.inf
        assert np.all(base[kept])
        p = np.zeros(l.shape[1])
        p[base] = cf.softmax(l[r][base].astype(np.float64), T)
        mass = p[kept].sum()
        assert mass >= top_p - 1e-12
        lo = l[r][kept].min()
        assert not np.any(base & ~kept & (l[r] == lo))  # groups stay whole
        if np.any(l[r][kept] > lo):
            assert mass - p[kept & (l[r] == lo)].sum() < top_p + 1e-12


@pytest.mark.parametrize("top_k,top_p", [(3, 1.0), (0, 0.7), (4, 0.8)])
def test_truncated_winner_follows_the_renormalised_truncated_law(top_k, top_p):
    # exactness of the race on the truncated support (Thm A.1 with P restricted and renormalised)
    rng = np.random.default_rng(30 + top_k)
    V, n = 7, 60000
    row = rng.normal(0, 1.0, V).astype(np.float32)
    masked, _ = oracle.truncate_rows(row[None, :], top_k=top_k, top_p=top_p)
    keep = masked[0] > -np.inf
    assert 1 <= keep.sum() < V
    key, ctx, pos = _ids(n, 40 + top_k)
    win, _, _, _ = oracle.target_rows(np.tile(masked[0], (n, 1)), key, ctx, pos)
    assert np.all(keep[win])
    p = cf.softmax(row[keep].astype(np.float64))
    cnt = np.bincount(win, minlength=V)[keep]
    assert stats.chisquare(cnt, p * n).pvalue > 1e-4


def test_truncated_distinct_list_is_plackett_luce_on_the_support():
    rng = np.random.default_rng(50)
    V, K, n = 6, 2, 60000
    row = rng.normal(0, 1, V).astype(np.float32)
    masked, _ = oracle.truncate_rows(row[None, :], top_k=3)
    keep = np.flatnonzero(masked[0] > -np.inf)
    key, ctx, pos = _ids(n, 51)
    d = oracle.draft_rows(np.tile(masked[0], (n, 1)), key, ctx, pos, K, mode=oracle.DISTINCT)
    q = cf.softmax(row[keep].astype(np.float64))
    pos_of = {int(t): j for j, t in enumerate(keep)}
    pairs = [(a, b) for a in range(keep.size) for b in range(keep.size) if a != b]
    idx = {pr: t for t, pr in enumerate(pairs)}
    cnt = np.bincount([idx[(pos_of[int(a)], pos_of[int(b)])] for a, b in d["tok"]], minlength=len(pairs))
    exp = np.array([cf.plackett_luce_prob(q, pr) for pr in pairs]) * n
    assert stats.chisquare(cnt, exp).pvalue > 1e-4


def test_truncated_list_shorter_than_k_and_iid_support():
    # support of 2 tokens, K = 4: DISTINCT has 2 entries, IID labels stay in the support
    row = np.array([[0.0, 2.0, -1.0, 1.5, -3.0]], np.float32)
    masked, _ = oracle.truncate_rows(row, top_k=2)
    n = 500
    key, ctx, pos = _ids(n, 60)
    d = oracle.draft_rows(np.tile(masked[0], (n, 1)), key, ctx, pos, 4, mode=oracle.DISTINCT)
    assert np.all(np.sort(d["tok"][:, :2], axis=1) == [1, 3]) and np.all(d["tok"][:, 2:] == -1)
    assert np.all(d["ndist"] == 2)
    e = oracle.draft_rows(np.tile(masked[0], (n, 1)), key, ctx, pos, 4, mode=oracle.IID)
    assert np.all(np.isin(e["labels"], [1, 3])) and np.all(e["mult"].sum(1) == 4)
