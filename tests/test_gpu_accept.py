"""The product path against the paper's acceptance laws: one speculative step
(gamma = 1) at many independent contexts with the same P and Q, through
pps_draft_list and pps_verify_tree; the fraction of accepted steps must match
the exact acceptance probability of the draft list (IID: 1 - sum_i p_i
(alpha_i / (1 + alpha_i))^K, App. B; DISTINCT: the integral form; K = 1: the
single-draft Poisson matching value) within the binomial tolerance."""
import math

import numpy as np
import pytest
import torch

from oracle import closed_forms as cf
from paper_2609_21858_gb300 import pps
from parity import dev_ids

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def _accept_rate(pl, ql, K, mode, n, seed):
    V = pl.size
    rng = np.random.default_rng(seed)
    key = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    ctx = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    pos = rng.integers(0, 2 ** 31, n, dtype=np.uint32)
    k, c, p = dev_ids(key, ctx, pos)
    q = torch.as_tensor(np.tile(ql.astype(np.float32), (n, 1))).cuda()
    d = pps.draft_list(q, k, c, p, K, mode=mode)
    N1 = 1 + K
    # node slots: the root (the context the lists were drawn at) and K children
    nk, nc, npos = np.repeat(key, N1), np.repeat(ctx, N1).copy(), np.repeat(pos, N1)
    nc[np.arange(n * N1) % N1 != 0] ^= np.uint64(0x9E3779B97F4A7C15)
    p_rows = torch.as_tensor(np.tile(pl.astype(np.float32), (n * N1, 1))).cuda()
    seq_off = torch.arange(n + 1, dtype=torch.int32, device="cuda") * N1
    ndr = np.full(n * N1, -1, np.int32)
    ndr[::N1] = np.arange(n)
    child = (np.arange(n)[:, None] * N1 + 1 + np.arange(K)[None, :]).astype(np.int32)
    v = pps.verify_tree(p_rows, *dev_ids(nk, nc, npos), 1, seq_off, torch.as_tensor(ndr).cuda(), d["tok"],
                        d["ndist"], torch.as_tensor(child).cuda())
    torch.cuda.synchronize()
    return float((v["accept_len"] >= 1).float().mean().item())


@pytest.mark.parametrize("K", [1, 3, 8])
@pytest.mark.parametrize("mode", [pps.IID, pps.DISTINCT])
def test_one_step_acceptance_matches_the_closed_forms(K, mode):
    V, n = 16, 40000
    rng = np.random.default_rng(100 + K)
    pl = rng.normal(0, 1.2, V).astype(np.float32)
    ql = (pl + rng.normal(0, 1.0, V)).astype(np.float32)
    p, q = cf.softmax(pl.astype(np.float64)), cf.softmax(ql.astype(np.float64))
    if K == 1:
        want = cf.accept_k1(p, q)
    elif mode == pps.IID:
        want = cf.accept_iid(p, q, K)
    else:
        want = cf.accept_distinct(p, q, K)
    got = _accept_rate(pl, ql, K, mode, n, 7 + K + 10 * mode)
    sd = math.sqrt(want * (1 - want) / n)
    assert abs(got - want) < 4.5 * sd + 1e-9, (got, want, sd)
    # DISTINCT lists accept at least as often as IID ones, and both beat the Thm 4.1 bound
    assert want >= cf.bound_thm41(p, q, K) - 1e-12
