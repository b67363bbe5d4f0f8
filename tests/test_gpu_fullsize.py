"""Full-size parity: the named configurations launched at their full sizes, exactly as bench.py
launches them, with every output row of the compared sequences checked against the oracle.

* zipf_k8 (B=64, V=128256, K=8, gamma=5, bf16): all 2,624 target and 2,112 draft rows, in the
  DISTINCT and IID modes.
* branch16 (B=256, V=152064, static (16,3,2,1) tree, fp32, 65 GB of logits): the full launch,
  and every row of its first 32 sequences (8,224 nodes, 5,152 draft rows), in both modes.
* the K sweep (B=64, V=128256, gamma=5, bf16, K = 1..32): the full launch per K, every row of its
  first 8 sequences in both modes; the mean accept length against the oracle's (bit-exact) and the
  depth-0 acceptance against the closed form of the IID list (App. B, Thm B.2, an equality for
  multi-arrival lists and a lower bound for DISTINCT lists).
* the detector pass over 10^7 (token, key, label, position) tuples: per-token scores, segment sums
  and log p-values against the oracle's, for the Aaronson (Gamma tail) and U (Chernoff) scores.

Flips (allowed only where the oracle's key gap is below 1e-6) are counted and printed in the
session's "full-size parity report" together with the accept lengths.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import closed_forms as cf
from paper_2609_21858_gb300 import pps, synth
from parity import REPORT, compare_draft, compare_winners, dev_ids, logp_tol_gamma, run_gpu, score_rtol

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()
    oracle.set_threads(0)


def _host(x, rows):
    """fp32 host copy of rows [0, rows) of a device logits tensor (in chunks of ~1 GB)."""
    out = np.empty((rows, x.shape[1]), np.float32)
    step = max(1, (1 << 28) // x.shape[1])
    for r0 in range(0, rows, step):
        r1 = min(rows, r0 + step)
        out[r0:r1] = x[r0:r1].float().cpu().numpy()
    return out


def _oracle_first(wl, n_cmp, modes):
    """Oracle draft lists (per mode) and target winners of the first n_cmp sequences."""
    t = wl.tree
    nn, nd = n_cmp * t.nodes_per_seq, n_cmp * t.draft_per_seq
    T = float(np.float32(wl.temperature))
    q = _host(wl.q_logits, nd)
    ids_d = (synth.u64(wl.draft_key[:nd]), synth.u64(wl.draft_ctx[:nd]), synth.u32(wl.draft_pos[:nd]))
    drafts = {m: oracle.draft_rows(q, *ids_d, t.K, row_k=t.row_k[:nd], mode=m, T=T) for m in modes}
    del q
    p = _host(wl.p_logits, nn)
    win, wd, _, mg = oracle.target_rows(p, synth.u64(wl.node_key[:nn]), synth.u64(wl.node_ctx[:nn]),
                                        synth.u32(wl.node_pos[:nn]), T=T)
    return drafts, dict(winner=win, word=wd, margin=mg)


def _depth0(wl, gv, mode):
    """Root acceptance of every sequence (accept_len >= 1) against the IID closed form of its root
    pair: the mean accepted fraction, the mean closed-form probability and the binomial sd."""
    t = wl.tree
    roots = t.seq_off[:-1].astype(np.int64)
    droots = t.node_draft_row[roots].astype(np.int64)
    P = wl.p_logits[torch.as_tensor(roots, device=wl.p_logits.device)].double().cpu().numpy()
    Q = wl.q_logits[torch.as_tensor(droots, device=wl.q_logits.device)].double().cpu().numpy()
    T = float(np.float32(wl.temperature))
    pr = np.array([cf.accept_iid_full(cf.softmax(P[s], T), cf.softmax(Q[s], T), int(t.row_k[droots[s]]))
                   for s in range(t.n_seq)])
    got = float(np.mean(gv["accept_len"] >= 1))
    sd = float(math.sqrt(np.sum(pr * (1 - pr)))) / t.n_seq
    return got, float(pr.mean()), sd


def _check_config(wl, n_cmp, modes, label):
    t = wl.tree
    nn, nd = n_cmp * t.nodes_per_seq, n_cmp * t.draft_per_seq
    gpu = {}
    for m in modes:
        gd, gv, status = run_gpu(wl, m)
        assert status == 0, f"status flags {status}"
        gpu[m] = (gd, gv)
    od_all, ov = _oracle_first(wl, n_cmp, modes)
    for m in modes:
        gd, gv = gpu[m]
        od = od_all[m]
        sub = {k: (x[:nd] if x is not None and x.ndim >= 1 and x.shape[0] == t.n_draft else x) for k, x in gd.items()}
        fd = compare_draft(sub, od)
        fw = compare_winners(gv["winner"][:nn], gv["word"][:nn], ov["winner"], ov["word"], ov["margin"])
        # the GPU walk of every sequence equals the oracle's walk on the GPU's own lists and winners
        ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, gd["tok"], gd["ndist"], t.child_node, gv["winner"],
                         gv["word"])
        assert np.array_equal(gv["accept_len"], ow["accept_len"])
        assert np.array_equal(gv["n_emitted"], ow["n_emitted"])
        assert np.array_equal(gv["emitted"], ow["emitted"])
        rt = score_rtol(wl.dtype)
        np.testing.assert_allclose(gv["score"], ow["score"], rtol=rt, atol=0)
        np.testing.assert_allclose(gv["score_sum"], ow["score_sum"], rtol=rt, atol=0)
        # the oracle's own walk on its own lists and winners: equal accept lengths wherever no
        # near-tie flipped a list or a winner of that sequence
        so = t.seq_off[: n_cmp + 1]
        oo = oracle.walk(t.gamma, so, t.node_draft_row[:nn], od["tok"], od["ndist"], t.child_node[:nd],
                         ov["winner"], ov["word"])
        flipped = np.zeros(n_cmp, bool)
        d_bad = np.nonzero(np.any(sub["tok"] != od["tok"], axis=1))[0]
        n_bad = np.nonzero(gv["winner"][:nn] != ov["winner"])[0]
        flipped[d_bad // t.draft_per_seq] = True
        flipped[n_bad // t.nodes_per_seq] = True
        same = ~flipped
        assert np.array_equal(gv["accept_len"][:n_cmp][same], oo["accept_len"][same])
        assert np.array_equal(gv["emitted"][:n_cmp][same], oo["emitted"][same])
        got0, cf0, sd0 = _depth0(wl, gv, m)
        if m == pps.IID:
            # the IID closed form is exact: the realised root acceptance is a sum of Bernoullis
            assert abs(got0 - cf0) <= 5 * sd0 + 1e-9, (got0, cf0, sd0)
        else:
            # DISTINCT lists accept at least as often as IID lists
            assert got0 >= cf0 - 5 * sd0 - 1e-9, (got0, cf0, sd0)
        REPORT.append(dict(config=label, mode="IID" if m == pps.IID else "DISTINCT",
                           rows_compared=f"{nd}+{nn}", draft_flips=fd, winner_flips=fw,
                           mean_accept_gpu=round(float(gv["accept_len"][:n_cmp].mean()), 4),
                           mean_accept_oracle=round(float(oo["accept_len"].mean()), 4),
                           mean_accept_gpu_all=round(float(gv["accept_len"].mean()), 4),
                           depth0_accept=round(got0, 4), depth0_closed_form_iid=round(cf0, 4),
                           depth0_sd=round(sd0, 4)))


def test_zipf_k8_every_row_both_modes():
    wl = synth.make_workload("zipf_k8", device="cuda")
    _check_config(wl, wl.tree.n_seq, (pps.DISTINCT, pps.IID), "zipf_k8")


def test_branch16_full_launch_first_32_sequences_both_modes():
    wl = synth.make_workload("branch16", device="cuda")
    _check_config(wl, 32, (pps.DISTINCT, pps.IID), "branch16")
    del wl
    torch.cuda.empty_cache()


@pytest.mark.parametrize("K", list(range(1, 33)))
def test_k_sweep_full_launch_first_8_sequences(K):
    wl = synth.make_workload("ksweep", device="cuda", K_sweep=K)
    _check_config(wl, 8, (pps.DISTINCT, pps.IID), f"ksweep K={K}")
    del wl
    torch.cuda.empty_cache()


def test_detector_pass_1e7_tuples():
    # 10^7 tuples in segments of 128: the first half watermarked (the oracle's own race winners
    # over N(0, 3^2) logits of 64 tokens, one fresh context each), the second half uniform
    # random tokens (the null)
    n, seg_len, Vw = 10_000_000, 128, 64
    half = n // 2
    rng = np.random.default_rng(2024)
    key = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    ctx = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    pos = rng.integers(0, 2 ** 30, n, dtype=np.uint32)
    tok = rng.integers(0, 128256, n, dtype=np.int32)
    step = 1_000_000
    for r0 in range(0, half, step):
        r1 = min(half, r0 + step)
        logits = (rng.standard_normal((r1 - r0, Vw), dtype=np.float32) * 3.0).astype(np.float32)
        tok[r0:r1] = oracle.target_rows(logits, key[r0:r1], ctx[r0:r1], pos[r0:r1])[0]
    seg = np.arange(0, n + 1, seg_len, dtype=np.int64)
    k, c, p = dev_ids(key, ctx, pos)
    t = torch.as_tensor(tok).cuda()
    s = torch.as_tensor(seg).cuda()
    for kind in (pps.SCORE_AARONSON, pps.SCORE_U):
        sc, sums, logp = pps.wm_detect(t, k, c, p, s, kind)
        torch.cuda.synchronize()
        sc, sums, logp = sc.cpu().numpy(), sums.cpu().numpy(), logp.cpu().numpy()
        osc, osums, ologp = oracle.wm_detect(tok, key, ctx, pos, seg, kind)
        rt = score_rtol(torch.float32)
        if kind == pps.SCORE_AARONSON:
            np.testing.assert_allclose(sc, osc, rtol=rt, atol=0)
        else:
            # U = r itself: fp32 rounding of a value in (0, 1)
            np.testing.assert_allclose(sc, osc, rtol=rt, atol=1e-7)
        np.testing.assert_allclose(sums, osums, rtol=rt, atol=0)
        M = seg_len
        if kind == pps.SCORE_AARONSON:
            # ln p at the kernel's own sums against the oracle's ln p at the same sums, within the
            # tolerance the detector's decision requires (tests/parity.py logp_tol_gamma)
            want = np.array([oracle.gamma_tail_logp(M, float(x)) for x in sums])
            tol = np.array([logp_tol_gamma(M, float(x), w) for x, w in zip(sums, want)])
            err = np.abs(logp - want)
            assert np.all(err <= tol), (int(np.argmax(err - tol)), float(np.max(err - tol)))
            # and the decisions at 1% against the oracle's own pass
            alpha = math.log(0.01)
            dec_g, dec_o = logp <= alpha, ologp <= alpha
            n_diff = int(np.sum(dec_g != dec_o))
            assert n_diff <= 2, n_diff
            nseg = len(seg) - 1
            REPORT.append(dict(config="detector 1e7", kind="Aaronson", segments=nseg,
                               max_logp_err=float(err.max()), decisions_differing_at_1pct=n_diff,
                               tpr_at_1pct=round(float(np.mean(dec_g[: nseg // 2])), 4),
                               null_rejection=round(float(np.mean(dec_g[nseg // 2:])), 5)))
        else:
            # Chernoff bound: fp32 minimiser, never below the oracle's bound at the same sum, at
            # most ~1e-6 above it
            want = np.array([oracle.chernoff_u_logp(M, float(x)) for x in sums])
            fin = np.isfinite(want) & (want != 0.0)
            assert np.all(logp[~fin] == want[~fin])
            w, g = want[fin], logp[fin]
            assert np.all(g >= w - 1e-12 * np.maximum(1.0, np.abs(w)))
            assert np.all(g <= w + 1e-6 * np.maximum(1.0, np.abs(w)))
