"""Pins of the oracle's non-identical proposals (App. A, the proposition on
heterogeneous proposals): the augmented source is B independent Exp(1)
arrivals per token; one proposal reduces to the race; the target sample is
the plain race's; Y ~ P, J uniform and independent of Y, X^(b) ~ Q_b and
mutually independent; the block-matching event has the exact probability
p_i / (B + alpha_i^(b)) of the proposition's bound; identical proposals
always accept."""
from __future__ import annotations

import math

import numpy as np
import pytest
from scipy import stats

import oracle

Z = 4.5  # two-sided normal quantile for the Monte Carlo tolerances


def _ids(n, seed):
    rng = np.random.default_rng(seed)
    return (rng.integers(0, 2 ** 64, n, dtype=np.uint64), rng.integers(0, 2 ** 64, n, dtype=np.uint64),
            rng.integers(0, 2 ** 32, n, dtype=np.uint32))


def _softmax(l):
    e = np.exp(l - l.max())
    return e / e.sum()


def _alpha(p, q):
    # alpha_i^(b) = p_i sum_j (q_bj / q_bi - p_j / p_i)_+
    return np.array([[p[i] * np.maximum(q[b] / q[b, i] - p / p[i], 0.0).sum() for b in range(q.shape[0])]
                     for i in range(len(p))])


def _steps(pl, ql, n, seed, T=1.0):
    B, V = ql.shape
    key, ctx, pos = _ids(n, seed)
    P = np.broadcast_to(pl.astype(np.float32), (n, V))
    Q = np.broadcast_to(ql.astype(np.float32), (n, B, V))
    return oracle.hetero_rows(P, Q, key, ctx, pos, B, T)


def _chi2_ok(counts, probs):
    res = stats.chisquare(counts, probs * counts.sum())
    return res.pvalue > 1e-4


# ---------------------------------------------------------------- the augmented source

@pytest.mark.parametrize("B", [2, 3, 5])
def test_augmented_arrivals_are_iid_exponential(B):
    # each block's E_(i,b) is Exp(1), the blocks are independent of one another,
    # and the smallest sits in a uniform block
    n = 6000
    key, ctx, pos = _ids(n, B)
    E = np.array([[oracle.block_e(int(key[t]), int(ctx[t]), int(pos[t]), 7, b, B) for b in range(B)]
                  for t in range(n)])
    for b in range(B):
        assert stats.kstest(E[:, b], "expon").pvalue > 1e-4
    C = np.corrcoef(E.T)
    assert np.all(np.abs(C[np.triu_indices(B, 1)]) < Z / math.sqrt(n))
    # joint survival P(E_0 > s, E_1 > t) = exp(-s - t)
    for s, t in ((0.5, 0.5), (1.0, 0.3), (0.2, 2.0)):
        f = np.mean((E[:, 0] > s) & (E[:, 1] > t))
        want = math.exp(-s - t)
        assert abs(f - want) < Z * math.sqrt(want * (1 - want) / n)
    amin = E.argmin(1)
    assert _chi2_ok(np.bincount(amin, minlength=B), np.full(B, 1.0 / B))
    J = np.array([oracle.block_j(int(key[t]), int(ctx[t]), int(pos[t]), 7, B) for t in range(n)])
    assert np.array_equal(amin, J)


def test_one_block_is_the_identical_source():
    key, ctx, pos = _ids(50, 1)
    for t in range(50):
        w = oracle.word(int(key[t]), int(ctx[t]), int(pos[t]), 3)
        assert oracle.block_j(int(key[t]), int(ctx[t]), int(pos[t]), 3, 1) == 0
        assert oracle.block_e(int(key[t]), int(ctx[t]), int(pos[t]), 3, 0, 1) == oracle.exp1(w)


# ---------------------------------------------------------------- reductions

def test_one_proposal_reduces_to_the_race():
    n, V = 40, 300
    rng = np.random.default_rng(2)
    P = rng.normal(0, 2, (n, V)).astype(np.float32)
    Q = rng.normal(0, 2, (n, 1, V)).astype(np.float32)
    key, ctx, pos = _ids(n, 3)
    r = oracle.hetero_rows(P, Q, key, ctx, pos, 1)
    win, word, _, _ = oracle.target_rows(P, key, ctx, pos)
    d = oracle.draft_rows(Q[:, 0], key, ctx, pos, 1)
    assert np.array_equal(r["y"], win) and np.array_equal(r["word"], word)
    assert np.array_equal(r["x"][:, 0], d["tok"][:, 0])
    assert np.all(r["j"] == 0)
    assert np.array_equal(r["accept"], (r["x"][:, 0] == r["y"]).astype(np.int32))


@pytest.mark.parametrize("B", [2, 3, 7])
def test_target_is_the_plain_race_for_every_b(B):
    # the smallest arrival of token i over the blocks is E'_i / B, so the
    # augmented argmin's token is the identical-proposal race winner
    n, V = 60, 200
    rng = np.random.default_rng(B)
    P = rng.normal(0, 3, (n, V)).astype(np.float32)
    P[:, rng.random(V) < 0.2] = -np.inf
    Q = rng.normal(0, 3, (n, B, V)).astype(np.float32)
    key, ctx, pos = _ids(n, 10 + B)
    r = oracle.hetero_rows(P, Q, key, ctx, pos, B, 0.8)
    win, word, _, _ = oracle.target_rows(P, key, ctx, pos, 0.8)
    assert np.array_equal(r["y"], win) and np.array_equal(r["word"], word)
    for c in range(0, n, 7):
        assert r["j"][c] == oracle.block_j(int(key[c]), int(ctx[c]), int(pos[c]), int(r["y"][c]), B)
    # each proposal is its block's race alone
    blk = np.tile(np.arange(B, dtype=np.int32), n)
    x, _, _ = oracle.block_draft_rows(Q.reshape(n * B, V), np.repeat(key, B), np.repeat(ctx, B), np.repeat(pos, B),
                                      blk, B, 0.8)
    assert np.array_equal(x.reshape(n, B), r["x"])


def test_identical_proposals_always_accept():
    # Q_b = P: within block J the target's point is also the proposal's
    n, V, B = 400, 9, 4
    pl = np.random.default_rng(5).normal(0, 1, V)
    r = _steps(pl, np.tile(pl, (B, 1)), n, 6)
    assert np.all(r["accept"] == 1)
    assert np.array_equal(r["x"][np.arange(n), r["j"]], r["y"])


def test_masked_rows():
    V, B = 50, 3
    rng = np.random.default_rng(7)
    P = rng.normal(0, 1, (4, V)).astype(np.float32)
    Q = rng.normal(0, 1, (4, B, V)).astype(np.float32)
    P[0] = -np.inf                       # no usable target token
    Q[1, 2] = -np.inf                    # proposal 2 has nothing to draft
    Q[2, 0, :] = -np.inf
    Q[2, 0, 17] = 0.0                    # a single usable token
    Q[3, 1, ::2] = np.nan                # NaN logits take no part
    key, ctx, pos = _ids(4, 8)
    r = oracle.hetero_rows(P, Q, key, ctx, pos, B)
    assert r["y"][0] == -1 and r["j"][0] == -1 and r["accept"][0] == 0
    assert r["x"][1, 2] == -1
    assert r["x"][2, 0] == 17 and math.isinf(r["margin_x"][2, 0])
    assert r["x"][3, 1] % 2 == 1


# ---------------------------------------------------------------- laws (mapping theorem)

def test_laws_of_y_j_and_the_proposals():
    B, V, n = 3, 6, 60000
    rng = np.random.default_rng(9)
    pl, ql = rng.normal(0, 1, V), rng.normal(0, 1.2, (B, V))
    p, q = _softmax(pl), np.array([_softmax(x) for x in ql])
    r = _steps(pl, ql, n, 11)
    y, j, x = r["y"], r["j"], r["x"]
    assert _chi2_ok(np.bincount(y, minlength=V), p)
    # J uniform and independent of Y: the (Y, J) table against p_i / B
    assert _chi2_ok(np.bincount(y * B + j, minlength=V * B), np.repeat(p, B) / B)
    for b in range(B):
        assert _chi2_ok(np.bincount(x[:, b], minlength=V), q[b])
    # proposals mutually independent: the (X^(0), X^(1)) table against q_0 q_1
    assert _chi2_ok(np.bincount(x[:, 0] * V + x[:, 1], minlength=V * V), np.outer(q[0], q[1]).ravel())


@pytest.mark.parametrize("B,seed", [(2, 1), (3, 2), (4, 3)])
def test_block_matching_event_has_the_bound_probability(B, seed):
    # P(Y = i, J = b, X^(b) = i) = p_i / ((B-1) + sum_j max(p_j, p_i q_bj / q_bi)) = p_i / (B + alpha_i^(b))
    # (competing exponentials on V x [B]); summed over (i, b) it is the
    # proposition's bound, and the acceptance probability is at least that
    V, n = 5, 80000
    rng = np.random.default_rng(seed)
    pl, ql = rng.normal(0, 1, V), rng.normal(0, 1.5, (B, V))
    p, q = _softmax(pl), np.array([_softmax(x) for x in ql])
    a = _alpha(p, q)
    exact = p[:, None] / (B + a)
    direct = np.array([[p[i] / ((B - 1) + np.maximum(p, p[i] * q[b] / q[b, i]).sum()) for b in range(B)]
                       for i in range(V)])
    assert np.allclose(exact, direct, rtol=1e-12)
    r = _steps(pl, ql, n, 100 + seed)
    y, j, x = r["y"], r["j"], r["x"]
    hit = x[np.arange(n), j] == y
    for i in range(V):
        for b in range(B):
            f = np.sum(hit & (y == i) & (j == b))
            e = exact[i, b] * n
            assert abs(f - e) < Z * math.sqrt(e * (1 - exact[i, b])) + 1, (i, b, f, e)
    bound = exact.sum()
    acc = r["accept"].mean()
    assert acc >= bound - Z * math.sqrt(bound * (1 - bound) / n)
    assert acc >= hit.mean()
    assert np.all(r["accept"][hit] == 1)
    # conditional form: P(accept | Y = i) >= sum_b 1 / (B + alpha_i^(b))
    for i in range(V):
        sel = y == i
        c = (1.0 / (B + a[i])).sum()
        assert r["accept"][sel].mean() >= c - Z * math.sqrt(c * (1 - c) / sel.sum())


def test_block_streams_never_alias():
    # the F stream of block b uses key ^ (b+1) * 0xBB67AE8584CAA73B and the J
    # stream key ^ 0x3C6EF372FE94F82B: no block below 2^32 shares J's tweak
    # or the identity (which would reuse the first-arrival words)
    cf, cj = 0xBB67AE8584CAA73B, 0x3C6EF372FE94F82B
    b1 = cj * pow(cf, -1, 2 ** 64) % 2 ** 64
    assert b1 >= 2 ** 32
    key, ctx, pos = 123456789, 987654321, 5
    ws = {oracle.word(key, ctx, pos, i) for i in range(64)}
    wj = {oracle.word(key ^ cj, ctx, pos, i) for i in range(64)}
    wf = {oracle.word(key ^ (((b + 1) * cf) % 2 ** 64), ctx, pos, i) for b in range(4) for i in range(64)}
    assert not (ws & wj) and not (ws & wf) and not (wj & wf)


# ---------------------------------------------------------------- the multi-proposal tree

def _draw(b, d, ctx, Vs):
    # a deterministic stand-in for proposal b's race at context ctx: few tokens, so chains agree often
    h = oracle.mix64(int(ctx) ^ ((b + 1) * 0x9E3779B97F4A7C15 % 2 ** 64) ^ (d * 0x632BE59BD9B4E019 % 2 ** 64))
    return -1 if h % 13 == 0 else int(h % Vs)


@pytest.mark.parametrize("B,gamma,Vs", [(1, 3, 3), (3, 4, 2), (5, 3, 3), (8, 5, 2), (32, 2, 4)])
def test_tree_is_the_trie_of_the_proposal_chains(B, gamma, Vs):
    # brute force: each proposal's chain, then the distinct prefixes per depth
    n_seq = 6
    key, ctx, pos = _ids(n_seq, B * 10 + gamma)
    tree = oracle.hetero_tree(n_seq, B, gamma)
    N1 = 1 + B * gamma
    roots = np.arange(n_seq) * N1
    tree["node_key"][roots], tree["node_ctx"][roots], tree["node_pos"][roots] = key, ctx, pos
    rk, rc, rp = np.repeat(key, B), np.repeat(ctx, B), np.repeat(pos, B)
    owner = np.zeros(n_seq * B, np.int32)
    for d in range(gamma):
        tok = np.array([_draw(r % B, d, rc[r], Vs) if owner[r] >= 0 else 7 for r in range(n_seq * B)], np.int32)
        rk, rc, rp, owner = oracle.hetero_expand(n_seq, B, gamma, d, tok, rk, rc, rp, owner, tree)
    L = [0] + [n_seq * (1 + (d - 1) * B) for d in range(1, gamma + 1)]
    for s in range(n_seq):
        chains = []
        for b in range(B):
            c, ch = int(ctx[s]), []
            for d in range(gamma):
                x = _draw(b, d, c, Vs)
                if x < 0:
                    break
                ch.append(x)
                c = oracle.child_label(c, x)
            chains.append(ch)
        # walk the oracle's tree along every prefix and compare lists with the brute force
        for d in range(gamma):
            prefixes = sorted({tuple(ch[:d]) for ch in chains if len(ch) >= d})
            nodes_at_d = []
            for pre in prefixes:
                node, lrow = s * N1, L[0] + s
                for t, x in enumerate(pre):
                    m = list(tree["list_tok"][lrow][:tree["list_nd"][lrow]]).index(x)
                    node = tree["child_node"][lrow][m]
                    o = node - s * N1 - 1 - t * B
                    lrow = L[t + 1] + s * B + o if t + 1 < gamma else -1
                nodes_at_d.append(node)
                through = [b for b in range(B) if len(chains[b]) > d and tuple(chains[b][:d]) == pre]
                want = []
                for b in through:
                    if chains[b][d] not in want:
                        want.append(chains[b][d])
                got = list(tree["list_tok"][lrow][:tree["list_nd"][lrow]])
                assert got == want, (s, pre, got, want)
                # the node's identity is the fold of the labeler along its prefix
                lab = int(ctx[s])
                for x in pre:
                    lab = oracle.child_label(lab, x)
                assert int(tree["node_ctx"][node]) == lab and int(tree["node_pos"][node]) == int(pos[s]) + d
                assert int(tree["node_key"][node]) == int(key[s])
            assert len(set(nodes_at_d)) == len(prefixes)
        # unused node slots and list rows are empty
        used = {tuple(ch[:d]) for ch in chains for d in range(1, len(ch) + 1)}
        n_used = int(np.count_nonzero(tree["node_ctx"][s * N1 + 1:(s + 1) * N1]))
        assert n_used == len(used)
