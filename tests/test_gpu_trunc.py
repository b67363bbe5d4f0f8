"""GPU parity of the truncated race (top-k, then top-p, before the race)
against the oracle's masking followed by its untruncated race, through the
C ABI (pps_draft_list_trunc / pps_verify_tree_trunc)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_21858_gb300 import pps, synth
from parity import check_workload, compare_draft, compare_winners, f32, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


@pytest.mark.parametrize("top_k,top_p", [(50, 1.0), (1, 1.0), (5, 0.9), (64, 0.5), (20, 0.97)])
@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_chain4x4_truncated(top_k, top_p, mode):
    wl = synth.make_workload("chain4x4", n_seq=8)
    check_workload(wl, mode, top_k=top_k, top_p=top_p)


@pytest.mark.parametrize("top_k,top_p", [(50, 1.0), (8, 0.8)])
def test_zipf_k8_truncated_reduced(top_k, top_p):
    wl = synth.make_workload("zipf_k8", n_seq=3)
    check_workload(wl, pps.DISTINCT, top_k=top_k, top_p=top_p)
    check_workload(wl, pps.IID, top_k=top_k, top_p=top_p)


def test_fp32_tiny_and_branch16_truncated():
    check_workload(synth.make_workload("tiny"), pps.DISTINCT, top_k=50, top_p=0.9)
    check_workload(synth.make_workload("branch16", n_seq=1), pps.DISTINCT, top_k=50, top_p=1.0)


@pytest.mark.parametrize("V,dtype", [(3, torch.bfloat16), (13, torch.float32), (70, torch.bfloat16),
                                     (1003, torch.bfloat16), (4099, torch.float32)])
def test_ragged_vocab_truncated(V, dtype):
    K = min(4, V)
    wl = synth.make_workload("chain4x4", n_seq=5, vocab=V, branching=(K, 1), dtype=dtype, seed=11 + V)
    check_workload(wl, pps.DISTINCT, top_k=min(50, V), top_p=0.9)
    check_workload(wl, pps.IID, top_k=10, top_p=1.0)


def test_unaligned_rows_truncated():
    base = synth.make_workload("chain4x4", n_seq=3, vocab=2001, seed=21)
    for attr in ("p_logits", "q_logits"):
        x = getattr(base, attr)
        wide = torch.zeros(x.shape[0], x.shape[1] + 3, dtype=x.dtype)
        wide[:, 1:1 + x.shape[1]] = x
        setattr(base, attr, wide.cuda()[:, 1:1 + x.shape[1]])
    check_workload(base, pps.DISTINCT, top_k=50, top_p=0.95)


def test_temperature_truncated():
    wl = synth.make_workload("chain4x4", n_seq=3, vocab=5000, seed=41)
    wl.temperature = 0.6
    check_workload(wl, pps.DISTINCT, top_k=30, top_p=0.8)
    wl.temperature = 1.7
    check_workload(wl, pps.IID, top_k=30, top_p=0.8)


def test_masked_nan_and_short_rows_truncated():
    wl = synth.make_workload("chain4x4", n_seq=4, vocab=3000, dtype=torch.float32, seed=31)
    p, q = wl.p_logits, wl.q_logits
    rng = np.random.default_rng(0)
    for x in (p, q):
        x[torch.as_tensor(rng.random(x.shape) < 0.3)] = float("-inf")
        x[torch.as_tensor(rng.random(x.shape) < 0.01)] = float("nan")
    p[3, :] = float("-inf")       # no usable token: winner -1
    q[2, :-3] = float("-inf")     # 3 usable tokens < top_k
    p[7, :-20] = float("nan")     # 20 usable tokens
    for tk, tp in ((50, 1.0), (10, 0.7)):
        gd, gv, status = run_gpu(wl, top_k=tk, top_p=tp)
        od, ov = run_oracle(wl, top_k=tk, top_p=tp)
        assert status == 0
        compare_draft(gd, od, loose=od["loose"])
        compare_winners(gv["winner"], gv["word"], ov["winner"], ov["word"], ov["margin"], loose=ov["loose"])
        assert gv["winner"][3] == -1


def _tie_rows(wl, n_ties, top_k):
    """Rows whose top_k-th logit ties with n_ties tokens (more than the 64-entry list holds)."""
    rng = np.random.default_rng(n_ties)
    for x in (wl.p_logits, wl.q_logits):
        V = x.shape[1]
        for r in range(0, x.shape[0], 2):
            cols = torch.as_tensor(rng.choice(V, n_ties + top_k // 2, replace=False), device=x.device)
            x[r, cols[: top_k // 2]] = 8.0 + torch.arange(top_k // 2, device=x.device, dtype=x.dtype) * 0.25
            x[r, cols[top_k // 2:]] = 6.0   # the tie group at the top_k-th place


@pytest.mark.parametrize("top_p", [1.0, 0.999999, 0.6])
def test_top_k_tie_group_larger_than_the_list(top_p):
    # the tie group of l_(k) overflows the 64-entry lists: the row is finished by a
    # second pass (kept tie group: exact race over logit >= l_(k); dropped: the list)
    wl = synth.make_workload("chain4x4", n_seq=4, vocab=32000, seed=61)
    _tie_rows(wl, 300, 40)
    gd, gv, status = run_gpu(wl, top_k=40, top_p=top_p)
    od, ov = run_oracle(wl, top_k=40, top_p=top_p)
    assert status == 0
    compare_draft(gd, od, loose=od["loose"])
    compare_winners(gv["winner"], gv["word"], ov["winner"], ov["word"], ov["margin"], loose=ov["loose"])


def test_constant_rows_keep_everything():
    wl = synth.make_workload("chain4x4", n_seq=2, vocab=5000, seed=71)
    wl.p_logits[1, :] = 1.5
    wl.q_logits[0, :] = -2.0
    check_workload(wl, pps.DISTINCT, top_k=3, top_p=1.0)


def test_full_size_zipf_k8_truncated_sampled_rows():
    wl = synth.make_workload("zipf_k8", device="cuda")
    t = wl.tree
    gd, gv, status = run_gpu(wl, top_k=50, top_p=1.0)
    assert status == 0
    rng = np.random.default_rng(8)
    dr = np.sort(rng.choice(t.n_draft, 48, replace=False))
    nr = np.sort(rng.choice(t.n_nodes, 48, replace=False))
    dsel, nsel = torch.as_tensor(dr, device="cuda"), torch.as_tensor(nr, device="cuda")
    qm, _ = oracle.truncate_rows(wl.q_logits[dsel].float().cpu().numpy(), 50, 1.0, 1.0)
    pm, _ = oracle.truncate_rows(wl.p_logits[nsel].float().cpu().numpy(), 50, 1.0, 1.0)
    od = oracle.draft_rows(qm, synth.u64(wl.draft_key[dsel]), synth.u64(wl.draft_ctx[dsel]),
                           synth.u32(wl.draft_pos[dsel]), t.K, row_k=t.row_k[dr])
    sub = {k: (x[dr] if x is not None and x.ndim >= 1 and x.shape[0] == t.n_draft else x) for k, x in gd.items()}
    compare_draft(sub, od, rows=dr)
    win, wd, _, mg = oracle.target_rows(pm, synth.u64(wl.node_key[nsel]), synth.u64(wl.node_ctx[nsel]),
                                        synth.u32(wl.node_pos[nsel]))
    compare_winners(gv["winner"][nr], gv["word"][nr], win, wd, mg)
    ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, gd["tok"], gd["ndist"], t.child_node, gv["winner"],
                     gv["word"])
    assert np.array_equal(gv["accept_len"], ow["accept_len"]) and np.array_equal(gv["emitted"], ow["emitted"])
