"""bench.py's parity accounting (the `parity` and `philox7.parity` blocks of the bench line): fed
the oracle's own lists, winners and accept lengths it reports no flip and no mismatch; a wrong
winner where the oracle's key gap is wide is a mismatch, and a wrong list where the gap is below
1e-6 (planted in the oracle's record, on the CPU) is a flip.  Host logic only."""
import numpy as np
import torch

import bench
import oracle
from paper_2609_21858_gb300 import synth


def _step():
    wl = synth.make_workload("chain4x4", device="cpu", n_seq=3, vocab=500, seed=7)
    t = wl.tree
    keep = {}
    run, nd, nn, _ = bench.oracle_sample(wl, t.n_draft, t.n_nodes, keep=keep)
    assert (nd, nn) == (t.n_draft, t.n_nodes)
    run()
    od = keep["draft"]
    win, wd, _, _ = keep["target"]
    ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, od["tok"], od["ndist"], t.child_node, win, wd)
    dout = {"tok": torch.as_tensor(np.array(od["tok"]))}
    vout = {"winner": torch.as_tensor(np.array(win)), "accept_len": torch.as_tensor(np.array(ow["accept_len"]))}
    return wl, keep, dout, vout


def test_oracle_outputs_give_no_flip_and_no_mismatch():
    wl, keep, dout, vout = _step()
    r = bench.step_parity(wl, keep, dout, vout)
    assert r["draft_flips"] == 0 and r["winner_flips"] == 0 and r["mismatches"] == 0
    assert r["accept_len_equal_to_oracle"]
    assert r["mean_accept_len"]["gpu"] == r["mean_accept_len"]["oracle"]


def test_a_wrong_winner_is_a_mismatch_and_a_close_wrong_list_is_a_flip():
    wl, keep, dout, vout = _step()
    _, _, _, mg = keep["target"]
    i = int(np.argmax(mg))  # the widest gap: a changed winner there is an error
    w2 = vout["winner"].clone()
    w2[i] = (int(w2[i]) + 1) % wl.vocab
    r = bench.step_parity(wl, keep, dout, dict(vout, winner=w2))
    assert r["mismatches"] == 1 and r["winner_flips"] == 0
    # a draft row whose oracle gap is (planted) below 1e-6: two tokens swapped there is a flip
    j = 0
    keep["draft"]["min_gap"][j] = 0.0
    t2 = dout["tok"].clone()
    t2[j, [0, 1]] = t2[j, [1, 0]]
    r = bench.step_parity(wl, keep, dict(dout, tok=t2), vout)
    assert r["draft_flips"] == 1 and r["mismatches"] == 0
