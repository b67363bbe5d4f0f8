"""Shared GPU-vs-oracle comparison for the parity tests.

Rules (the tolerance the path is held to):
* token indices, accept lengths, multiplicities and Philox words: bit-exact;
  a differing index is allowed only where the oracle's gap between the keys
  involved is below 1e-6 (a near-tie), and every such flip is counted;
* watermark scores: within 1e-5 relative for fp32 logits, 1e-3 for bf16.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2609_21858_gb300 import pps, synth

FLIP_MARGIN = 1e-6
# one dict per full-size comparison (flip counts, accept lengths); printed at the end of the session
REPORT: list = []
TOP_P_MARGIN = 1e-12  # top-p decisions closer than this to 1 - top_p may differ (exp and summation rounding)


def dev_ids(key, ctx, pos, device="cuda"):
    return (torch.as_tensor(np.asarray(key).view(np.int64)).to(device),
            torch.as_tensor(np.asarray(ctx).view(np.int64)).to(device),
            torch.as_tensor(np.asarray(pos).view(np.int32)).to(device))


def score_rtol(dtype) -> float:
    return 1e-5 if dtype == torch.float32 else 1e-3


# Detector p-values.  A segment is declared watermarked when ln p <= ln alpha.  The per-token scores
# may err by SCORE_REL = 1e-5 relative (the fp32 tolerance above), which moves a segment's sum S by
# up to 1e-5 S and its ln p by 1e-5 S |d ln p / dS|.  Evaluating ln p at the kernel's own S must add
# no more than a tenth of that, and in any case no more than LOGP_FLOOR = 2e-6 (a relative change of
# 2e-6 in p, which no decision at a significance level resolves).
SCORE_REL = 1e-5
LOGP_FLOOR = 2e-6


def logp_tol_gamma(M: int, S: float, lnq: float) -> float:
    """Tolerance on ln p of the Aaronson sum S of M tokens (p = Q(M, S), the regularised upper
    incomplete gamma; d ln Q / dS = -S^(M-1) e^-S / (Gamma(M) Q))."""
    import math
    if M <= 0 or not (S > 0) or not math.isfinite(lnq):
        return LOGP_FLOOR
    dlog = math.exp(min(700.0, (M - 1) * math.log(S) - S - math.lgamma(M) - lnq))
    return LOGP_FLOOR + 0.1 * SCORE_REL * S * dlog


def compare_draft(g, o, rows=None, loose=None):
    """g: GPU dict (numpy), o: oracle dict, loose: rows whose truncation decision was a
    near-tie (may differ).  Returns number of allowed flips."""
    tok_g, tok_o = g["tok"], o["tok"]
    bad = np.nonzero(np.any(tok_g != tok_o, axis=1))[0]
    flips = 0
    for r in bad:
        assert o["min_gap"][r] < FLIP_MARGIN or (loose is not None and loose[r]), (
            f"draft row {r if rows is None else rows[r]}: gpu {tok_g[r]} oracle {tok_o[r]} gap {o['min_gap'][r]}")
        flips += 1
    ok = np.setdiff1d(np.arange(tok_g.shape[0]), bad)
    assert np.array_equal(g["mult"][ok], o["mult"][ok]), "multiplicities differ"
    assert np.array_equal(g["ndist"][ok], o["ndist"][ok]), "distinct counts differ"
    if "samples" in g and g["samples"] is not None:
        assert np.array_equal(g["samples"][ok], o["labels"][ok]), "ordered samples differ"
    if "key" in g and g["key"] is not None:
        valid = tok_o[ok] >= 0
        np.testing.assert_allclose(g["key"][ok][valid], o["key"][ok][valid], rtol=0, atol=5e-5)
    return flips


def compare_winners(win_g, word_g, win_o, word_o, margin_o, loose=None):
    bad = np.nonzero(win_g != win_o)[0]
    for r in bad:
        assert margin_o[r] < FLIP_MARGIN or (loose is not None and loose[r]), (
            f"node {r}: gpu {win_g[r]} oracle {win_o[r]} margin {margin_o[r]}")
    ok = np.setdiff1d(np.arange(win_g.shape[0]), bad)
    assert np.array_equal(word_g[ok], word_o[ok]), "winner words differ"
    return len(bad)


def run_gpu(wl, mode=pps.DISTINCT, device="cuda", top_k=0, top_p=1.0):
    t = wl.tree
    g = lambda x: torch.as_tensor(np.asarray(x)).to(device).contiguous()
    q, p = wl.q_logits.to(device), wl.p_logits.to(device)
    status = torch.zeros(1, dtype=torch.int32, device=device)
    d = pps.draft_list(q, wl.draft_key.to(device), wl.draft_ctx.to(device), wl.draft_pos.to(device), t.K,
                       row_k=g(t.row_k), mode=mode, temperature=wl.temperature, status=status, top_k=top_k,
                       top_p=top_p)
    v = pps.verify_tree(p, wl.node_key.to(device), wl.node_ctx.to(device), wl.node_pos.to(device), t.gamma,
                        g(t.seq_off), g(t.node_draft_row), d["tok"], d["ndist"], g(t.child_node),
                        temperature=wl.temperature, status=status, top_k=top_k, top_p=top_p)
    torch.cuda.synchronize()
    cpu = lambda dd: {k: (x.cpu().numpy() if x is not None else None) for k, x in dd.items()}
    d, v = cpu(d), cpu(v)
    v["word"] = v["word"].view(np.uint32)
    return d, v, int(status.item())


def f32(x) -> float:
    """x as the fp32 value the C-ABI receives"""
    return float(np.float32(x))


def run_oracle(wl, mode=pps.DISTINCT, top_k=0, top_p=1.0):
    """Oracle lists and winners; with top_k > 0 the logits are truncated first (oracle.truncate_rows).
    Also returns, per draft row and per node, whether a top-p decision was a near-tie."""
    t = wl.tree
    T = f32(wl.temperature)
    q = wl.q_logits.float().cpu().numpy()
    p = wl.p_logits.float().cpu().numpy()
    loose_q = np.zeros(q.shape[0], bool)
    loose_p = np.zeros(p.shape[0], bool)
    if top_k > 0:
        q, mq = oracle.truncate_rows(q, top_k, f32(top_p), T)
        p, mp = oracle.truncate_rows(p, top_k, f32(top_p), T)
        loose_q, loose_p = mq < TOP_P_MARGIN, mp < TOP_P_MARGIN
    d = oracle.draft_rows(q, synth.u64(wl.draft_key), synth.u64(wl.draft_ctx), synth.u32(wl.draft_pos), t.K,
                          row_k=t.row_k, mode=mode, T=T)
    win, wd, ky, mg = oracle.target_rows(p, synth.u64(wl.node_key), synth.u64(wl.node_ctx), synth.u32(wl.node_pos),
                                         T=T)
    d["loose"] = loose_q
    return d, dict(winner=win, word=wd, key=ky, margin=mg, loose=loose_p)


def check_workload(wl, mode=pps.DISTINCT, top_k=0, top_p=1.0):
    """Full comparison of one workload; returns (draft flips, winner flips)."""
    t = wl.tree
    gd, gv, status = run_gpu(wl, mode, top_k=top_k, top_p=top_p)
    od, ov = run_oracle(wl, mode, top_k=top_k, top_p=top_p)
    assert status == 0, f"status flags {status}"
    fd = compare_draft(gd, od, loose=od["loose"])
    fw = compare_winners(gv["winner"], gv["word"], ov["winner"], ov["word"], ov["margin"], loose=ov["loose"])
    # the walk: the oracle walk on the GPU's own lists and winners must match exactly
    ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, gd["tok"], gd["ndist"], t.child_node, gv["winner"],
                     gv["word"])
    assert np.array_equal(gv["accept_len"], ow["accept_len"])
    assert np.array_equal(gv["n_emitted"], ow["n_emitted"])
    assert np.array_equal(gv["emitted"], ow["emitted"])
    rt = score_rtol(wl.dtype)
    np.testing.assert_allclose(gv["score"], ow["score"], rtol=rt, atol=0)
    np.testing.assert_allclose(gv["score_sum"], ow["score_sum"], rtol=rt, atol=0)
    if fd == 0 and fw == 0:
        # no near-ties: the oracle's own walk on its own lists is the same
        ow2 = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, od["tok"], od["ndist"], t.child_node, ov["winner"],
                          ov["word"])
        assert np.array_equal(gv["accept_len"], ow2["accept_len"])
        assert np.array_equal(gv["emitted"], ow2["emitted"])
    return fd, fw
