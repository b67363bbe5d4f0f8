"""Pins of the oracle's dynamic IID draft tree (Alg. 4 with MPFR lists): the
labeler against SplitMix64's published first output, and the tree's
invariants (K draft paths per depth, one parent per node, identities)."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
from paper_2609_21858_gb300 import synth

GOLDEN = 0x9E3779B97F4A7C15
M64 = (1 << 64) - 1


def test_mix64_is_splitmix64_output():
    # SplitMix64 from state 0: first output 0xE220A8397B1DCDAF (its state after one step is the golden gamma)
    assert oracle.mix64(GOLDEN) == 0xE220A8397B1DCDAF
    s = synth.splitmix64_stream(12345, 5)
    state = 12345
    for t in range(5):
        state = (state + GOLDEN) & M64
        assert oracle.mix64(state) == int(s[t])


def test_child_label_mixes_parent_and_token():
    rng = np.random.default_rng(0)
    for _ in range(50):
        p = int(rng.integers(0, 2 ** 63)) * 2 + 1
        u = int(rng.integers(0, 200000))
        assert oracle.child_label(p, u) == oracle.mix64(p ^ (((u + 1) * GOLDEN) & M64))
    assert oracle.child_label(7, 3) != oracle.child_label(7, 4) and oracle.child_label(7, 3) != oracle.child_label(8, 3)


def build_oracle_tree(key, ctx, pos, K, gamma, V, T=1.0, seed=0):
    """The dynamic IID tree drafted by the oracle with label-keyed synthetic logits."""
    n_seq = len(key)
    N1, R1 = 1 + K * gamma, 1 + K * (gamma - 1)
    tree = dict(child_node=np.full((n_seq * R1, K), -1, np.int32), node_key=np.zeros(n_seq * N1, np.uint64),
                node_ctx=np.zeros(n_seq * N1, np.uint64), node_pos=np.zeros(n_seq * N1, np.uint32))
    roots = np.arange(n_seq) * N1
    tree["node_key"][roots], tree["node_ctx"][roots], tree["node_pos"][roots] = key, ctx, pos
    k = np.full(n_seq, K, np.int32)
    depths = []
    for d in range(gamma):
        logits = synth.label_logits(ctx, V, seed=seed)
        out = oracle.draft_rows(logits, key, ctx, pos, K, row_k=np.maximum(k, 1), mode=oracle.IID, T=T)
        depths.append(dict(key=key, ctx=ctx, pos=pos, k=k, out=out))
        key, ctx, pos, k = oracle.tree_expand(n_seq, K, gamma, d, out, key, ctx, pos, k, tree)
    return tree, depths


def test_dynamic_tree_keeps_k_paths_and_one_parent_per_node():
    K, gamma, n_seq, V = 5, 3, 120, 40
    rng = np.random.default_rng(1)
    key = rng.integers(0, 2 ** 63, n_seq, dtype=np.uint64)
    ctx = rng.integers(0, 2 ** 63, n_seq, dtype=np.uint64)
    pos = rng.integers(0, 1000, n_seq, dtype=np.uint32)
    tree, depths = build_oracle_tree(key, ctx, pos, K, gamma, V)
    N1, R1 = 1 + K * gamma, 1 + K * (gamma - 1)
    for d, st in enumerate(depths):
        w = 1 if d == 0 else K
        k = st["k"].reshape(n_seq, w)
        assert np.all(k.sum(1) == K)                      # the sequence's K draft paths
        nd = st["out"]["ndist"].reshape(n_seq, w)
        present = k > 0
        assert np.all(st["out"]["mult"].reshape(n_seq, w, K).sum(2)[present] == k[present])
        n_children = (nd * present).sum(1)
        assert np.all(n_children <= K)
        nxt_k = depths[d + 1]["k"].reshape(n_seq, K) if d + 1 < gamma else None
        D_d = 0 if d == 0 else n_seq * (1 + (d - 1) * K)
        for b in range(n_seq):
            seen = []
            for i in range(w):
                dr = D_d + b * w + i
                for m in range(K):
                    c = tree["child_node"][dr, m]
                    if present[b, i] and m < nd[b, i]:
                        assert c == b * N1 + 1 + d * K + len(seen)
                        tok = st["out"]["tok"][b * w + i, m]
                        assert tree["node_ctx"][c] == oracle.child_label(int(st["ctx"][b * w + i]), int(tok))
                        assert tree["node_pos"][c] == st["pos"][b * w + i] + 1
                        assert tree["node_key"][c] == key[b]
                        if nxt_k is not None:
                            assert nxt_k[b, len(seen)] == st["out"]["mult"][b * w + i, m]
                        seen.append(c)
                    else:
                        assert c == -1
            assert len(set(seen)) == len(seen) == n_children[b]
            if nxt_k is not None:
                assert np.all(nxt_k[b, len(seen):] == 0)
