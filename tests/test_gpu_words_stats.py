"""The library's keyed words as random numbers: frequency and serial tests over 10^9 words of the
keyed source (the words every race, list and score is built from), on whichever build is loaded
(Philox4x32-10, or Philox4x32-7 in the child run of tests/test_gpu_philox7.py).  The method's
unbiasedness (the emitted token is distributed as P) and the detector's null law (Uniform(0,1)
pivot, Exp(1) score) assume the words of distinct counters behave as independent uniform draws
(keyed PRF, Sec. 3.1); these chi-square tests would see a bias in any byte of the word, or a
dependence between the words of neighbouring tokens, far below what 10^9 samples resolve."""
import numpy as np
import pytest
import torch
from scipy import stats

from paper_2609_21858_gb300 import pps

pytestmark = pytest.mark.gpu

N_ROWS, V = 8, 125_000_000  # 10^9 words: 8 contexts of 1.25 10^8 tokens
P_MIN = 1e-6  # a false alarm once in a million runs per test


@pytest.fixture(scope="module")
def words():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    dev = torch.device("cuda", 0)
    rng = np.random.default_rng(2024)
    key = torch.as_tensor(rng.integers(-2 ** 63, 2 ** 63 - 1, N_ROWS, dtype=np.int64), device=dev)
    ctx = torch.as_tensor(rng.integers(-2 ** 63, 2 ** 63 - 1, N_ROWS, dtype=np.int64), device=dev)
    pos = torch.as_tensor(rng.integers(0, 2 ** 31, N_ROWS, dtype=np.int64).astype(np.int32), device=dev)
    w = pps.philox_words(key, ctx, pos, V)  # int32 bit patterns of the uint32 words, [N_ROWS, V]
    yield w
    del w
    torch.cuda.empty_cache()


def _chi2_uniform(counts):
    c = counts.double().cpu().numpy()
    return stats.chisquare(c).pvalue


@pytest.mark.parametrize("shift", [24, 16, 8, 0])
def test_every_byte_of_the_words_is_uniform(words, shift):
    b = torch.bitwise_and(torch.bitwise_right_shift(words, shift), 0xFF).flatten()
    counts = torch.bincount(b, minlength=256)
    assert int(counts.sum()) == N_ROWS * V
    assert _chi2_uniform(counts) > P_MIN


def test_neighbouring_tokens_words_are_independent(words):
    # serial test: the top 4 bits of the words of tokens i and i+1 of a context (the same
    # Philox block for 3 of 4 pairs, the next block for the 4th), 256 cells
    hi = torch.bitwise_and(torch.bitwise_right_shift(words, 28), 0xF)
    pair = (hi[:, :-1] * 16 + hi[:, 1:]).flatten()
    counts = torch.bincount(pair, minlength=256)
    assert _chi2_uniform(counts) > P_MIN
    # and the same for tokens i and i+4 (the same lane of consecutive blocks)
    pair4 = (hi[:, :-4] * 16 + hi[:, 4:]).flatten()
    assert _chi2_uniform(torch.bincount(pair4, minlength=256)) > P_MIN


def test_contexts_are_independent(words):
    # the words of the same token in two contexts (different ctx, pos and key)
    hi = torch.bitwise_and(torch.bitwise_right_shift(words, 28), 0xF)
    pair = (hi[0] * 16 + hi[1]).flatten()
    assert _chi2_uniform(torch.bincount(pair, minlength=256)) > P_MIN
