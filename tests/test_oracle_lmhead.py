"""Pins of the oracle's LM head (logits = hidden . weight^T, the layer whose
output the race reads; App. B cost remark): exact integer arithmetic on dyadic
operands and the one-hot special case, so a transposed operand, a dropped
term or a wrong stride fails here."""
import numpy as np

import oracle


def test_dyadic_operands_give_the_exact_integer_product():
    rng = np.random.default_rng(1)
    n, V, d = 7, 13, 101
    hi = rng.integers(-3, 4, (n, d))
    wi = rng.integers(-2, 3, (V, d))
    got = oracle.lmhead_logits(hi.astype(np.float32), (wi / 64.0).astype(np.float32))
    want = (hi.astype(np.int64) @ wi.astype(np.int64).T) / 64.0  # exact integer product, exact scaling
    assert np.array_equal(got, want)
    # a non-square shape with swapped operands would not even line up: the result is [n, V]
    assert got.shape == (n, V)


def test_one_hot_hidden_state_selects_a_weight_column():
    rng = np.random.default_rng(2)
    V, d = 9, 16
    w = rng.standard_normal((V, d)).astype(np.float32)
    h = np.zeros((d, d), np.float32)
    h[np.arange(d), np.arange(d)] = 1.0
    got = oracle.lmhead_logits(h, w)
    assert np.array_equal(got, w.T.astype(np.float64))


def test_rows_are_independent_and_sums_run_over_d():
    rng = np.random.default_rng(3)
    h = rng.integers(-4, 5, (3, 50)).astype(np.float32)
    w = rng.integers(-4, 5, (6, 50)).astype(np.float32)
    full = oracle.lmhead_logits(h, w)
    for r in range(3):
        assert np.array_equal(oracle.lmhead_logits(h[r:r + 1], w)[0], full[r])
    # splitting d into two halves adds up
    a = oracle.lmhead_logits(h[:, :20], w[:, :20]) + oracle.lmhead_logits(h[:, 20:], w[:, 20:])
    assert np.array_equal(a, full)
