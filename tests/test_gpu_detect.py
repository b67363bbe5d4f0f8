"""GPU parity of the detector suite (pps_wm_detect) against the oracle: the
per-token scores of every kind, the per-segment sums, and the log p-values
(evaluated by the oracle at the GPU's own sums, so that the two questions
stay separate)."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_21858_gb300 import pps, synth
from parity import dev_ids, logp_tol_gamma

pytestmark = pytest.mark.gpu

KINDS = [(pps.SCORE_AARONSON, 0.0), (pps.SCORE_U, 0.0), (pps.SCORE_LI, 0.3), (pps.SCORE_LI, 0.5),
         (pps.SCORE_LI, 0.85), (pps.SCORE_POWER_LAW, 0.01), (pps.SCORE_POWER_LAW, 1.0)]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def _tuples(n, seed):
    rng = np.random.default_rng(seed)
    tok = rng.integers(0, 152064, n, dtype=np.int32)
    key = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    ctx = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    pos = rng.integers(0, 2 ** 32, n, dtype=np.uint32)
    return tok, key, ctx, pos


def _segments(n, seed):
    rng = np.random.default_rng(seed)
    cuts = np.sort(rng.choice(np.arange(1, n), 60, replace=False))
    seg = np.concatenate([[0], cuts[:20], cuts[20:21], cuts[20:], [n]]).astype(np.int64)  # includes an empty one
    return seg


def _check_chernoff(got, M, S):
    # the GPU minimiser is fp32: its bound is never below the true minimum and at most ~1e-6 above it
    want = oracle.chernoff_u_logp(M, S)
    if want == 0.0 or math.isinf(want):
        assert got == want
        return
    assert want - 1e-12 * max(1.0, abs(want)) <= got <= want + 1e-6 * max(1.0, abs(want))


@pytest.mark.parametrize("kind,param", KINDS)
def test_scores_sums_and_p_values_match_the_oracle(kind, param):
    n = 50000
    tok, key, ctx, pos = _tuples(n, 11 + kind)
    seg = _segments(n, 5)
    k, c, p = dev_ids(key, ctx, pos)
    sc, sums, logp = pps.wm_detect(torch.as_tensor(tok).cuda(), k, c, p, torch.as_tensor(seg).cuda(), kind, param)
    torch.cuda.synchronize()
    sc, sums, logp = sc.cpu().numpy(), sums.cpu().numpy(), logp.cpu().numpy()
    osc, osums, _ = oracle.wm_detect(tok, key, ctx, pos, seg, kind, param)
    # per-token fp32 scores against fp64: relative where large, absolute near zero
    np.testing.assert_allclose(sc, osc, rtol=2e-5, atol=2e-6 * max(1.0, np.abs(osc).max()))
    np.testing.assert_allclose(sums, osums, rtol=2e-5, atol=1e-4)
    for g in range(len(seg) - 1):
        M = int(seg[g + 1] - seg[g])
        if M == 0:
            assert logp[g] == 0.0
        elif kind == pps.SCORE_AARONSON:
            want = oracle.gamma_tail_logp(M, float(sums[g]))
            assert abs(logp[g] - want) <= logp_tol_gamma(M, float(sums[g]), want)
        elif kind == pps.SCORE_U:
            _check_chernoff(logp[g], M, float(sums[g]))
        else:
            assert math.isnan(logp[g])


def test_p_values_in_watermarked_tails_and_single_segment():
    # tokens chosen by the race (watermarked): large S_A, ln p far below zero; no seg_off = one segment
    wl = synth.make_workload("chain4x4", n_seq=8, vocab=2000, dtype=torch.float32, seed=3)
    t = wl.tree
    v = pps.verify_tree(wl.p_logits.cuda(), wl.node_key.cuda(), wl.node_ctx.cuda(), wl.node_pos.cuda(), t.gamma,
                        torch.as_tensor(t.seq_off).cuda(), torch.as_tensor(t.node_draft_row).cuda(),
                        torch.zeros(t.n_draft, t.K, dtype=torch.int32, device="cuda") - 1,
                        torch.zeros(t.n_draft, dtype=torch.int32, device="cuda"),
                        torch.as_tensor(t.child_node).cuda())
    win = v["winner"]
    _, sums, logp = pps.wm_detect(win, wl.node_key.cuda(), wl.node_ctx.cuda(), wl.node_pos.cuda())
    torch.cuda.synchronize()
    M = t.n_nodes
    S = float(sums.item())
    assert S > M  # watermarked: E[A] > 1
    want = oracle.gamma_tail_logp(M, S)
    assert abs(logp.item() - want) <= logp_tol_gamma(M, S, want)
    assert logp.item() < math.log(1e-3)


# 2^18 - 1 and 2^18: the longest segment whose Poisson series runs in fp32 and the shortest in
# fp64; 2^24 + 5: a segment where an fp32 series would have drifted by ~1e-5
@pytest.mark.parametrize("M", [1, 2, 7, 128, 1000, 4096, 20000, (1 << 18) - 1, 1 << 18, (1 << 24) + 5])
def test_gamma_and_chernoff_for_one_segment_of_m_tokens(M):
    # seg_off = NULL: one segment of all M tokens; null tokens, so S is near M (Aaronson) or M/2 (U)
    tok, key, ctx, pos = _tuples(M, M)
    k, c, p = dev_ids(key, ctx, pos)
    t = torch.as_tensor(tok).cuda()
    _, sa, la = pps.wm_detect(t, k, c, p, None, pps.SCORE_AARONSON)
    _, su, lu = pps.wm_detect(t, k, c, p, None, pps.SCORE_U)
    torch.cuda.synchronize()
    want = oracle.gamma_tail_logp(M, float(sa.item()))
    assert abs(la.item() - want) <= logp_tol_gamma(M, float(sa.item()), want)
    _check_chernoff(lu.item(), M, float(su.item()))


@pytest.mark.parametrize("kind,param", [(pps.SCORE_AARONSON, 0.0), (pps.SCORE_U, 0.0), (pps.SCORE_LI, 0.5)])
def test_one_key_per_text(kind, param):
    # the tokens of one text share the watermark key: groups of 128 tuples with one key take the
    # kernel's uniform-key path; texts of 128 and 300 tokens (boundaries inside groups too), a
    # ragged tail, and a view whose arrays are not 16-byte aligned (scalar loads)
    n = 40000 + 37
    tok, _, ctx, pos = _tuples(n, 90 + kind)
    rng = np.random.default_rng(91)
    lens = np.where(np.arange(n // 128 + 2) % 3 == 0, 300, 128)
    seg = np.concatenate([[0], np.cumsum(lens)])
    seg = seg[seg < n]
    seg = np.concatenate([seg, [n]]).astype(np.int64)
    text_key = rng.integers(0, 2 ** 64, len(seg) - 1, dtype=np.uint64)
    key = np.repeat(text_key, np.diff(seg))
    tg = torch.as_tensor(tok).cuda()
    kg, cg, pg = dev_ids(key, ctx, pos)
    for off in (0, 1):
        # off = 1: views one element in, so no array starts on a 16-byte boundary
        t, kk, cc, pp = tok[off:], key[off:], ctx[off:], pos[off:]
        sg = np.maximum(seg - off, 0)
        sg[0] = 0
        sc, sums, _ = pps.wm_detect(tg[off:], kg[off:], cg[off:], pg[off:], torch.as_tensor(sg).cuda(), kind, param)
        torch.cuda.synchronize()
        osc, osums, _ = oracle.wm_detect(t, kk, cc, pp, sg, kind, param)
        np.testing.assert_allclose(sc.cpu().numpy(), osc, rtol=2e-5, atol=2e-6 * max(1.0, np.abs(osc).max()))
        np.testing.assert_allclose(sums.cpu().numpy(), osums, rtol=2e-5, atol=1e-4)
