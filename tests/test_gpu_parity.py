"""GPU parity: libpps (through its C ABI) against the CPU oracle on the same
seeded inputs.  Sizes span several CTAs, rows split across CTAs and ragged
tails; tests/test_gpu_fullsize.py runs the named configurations at full size."""
import math
import os

import numpy as np
import pytest
import torch
from scipy import stats

import oracle
from oracle import closed_forms as cf
from paper_2609_21858_gb300 import pps, synth
from parity import check_workload, compare_draft, compare_winners, dev_ids, run_gpu, run_oracle, score_rtol

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def _rand_ids(n, seed):
    rng = np.random.default_rng(seed)
    return (rng.integers(0, 2 ** 64, n, dtype=np.uint64), rng.integers(0, 2 ** 64, n, dtype=np.uint64),
            rng.integers(0, 2 ** 32, n, dtype=np.uint32))


# ------------------------------------------------------------------ keyed source

@pytest.mark.parametrize("arrival", [1, 2, 7])
def test_philox_words_bit_exact(arrival):
    key, ctx, pos = _rand_ids(5, arrival)
    V = 1003
    g = pps.philox_words(*dev_ids(key, ctx, pos), V, arrival).cpu().numpy().view(np.uint32)
    o = oracle.words(key, ctx, pos, V, arrival)
    assert np.array_equal(g, o)


def test_philox_matches_curand():
    if pps.philox_rounds() != 10:
        pytest.skip("cuRAND's Philox generator has 10 rounds")
    import ctypes
    lib = ctypes.CDLL(os.path.join(ROOT, "tests", "native", "_build", "libcurandprobe.so"))
    rng = np.random.default_rng(3)
    n = 64
    ctr = rng.integers(0, 2 ** 32, (n, 4), dtype=np.uint64).astype(np.uint32)
    ctr[:, 1] &= 0x3FFFFFFF  # cuRAND's 64-bit offset holds 4 * (ctr0 | ctr1 << 32)
    key = rng.integers(0, 2 ** 32, (n, 2), dtype=np.uint64).astype(np.uint32)
    dc = torch.as_tensor(ctr.view(np.int32)).cuda()
    dk = torch.as_tensor(key.view(np.int32)).cuda()
    out = torch.zeros(n, 4, dtype=torch.int32, device="cuda")
    rc = lib.curand_philox_blocks(ctypes.c_void_p(dc.data_ptr()), ctypes.c_void_p(dk.data_ptr()),
                                  ctypes.c_void_p(out.data_ptr()), n, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0
    got = out.cpu().numpy().view(np.uint32)
    for t in range(n):
        assert list(got[t]) == list(oracle.philox4x32_10(ctr[t], key[t]))
    # and libpps's words at the same counters
    for t in range(8):
        kk = int(key[t, 0]) | (int(key[t, 1]) << 32)
        cx = int(ctr[t, 2]) | (int(ctr[t, 3]) << 32)
        base = int(ctr[t, 0]) << 2
        if base + 4 > 2 ** 31:
            continue
        w = pps.philox_words(*dev_ids([kk], [cx], [int(ctr[t, 1])]), base + 4).cpu().numpy().view(np.uint32)[0]
        assert list(w[base:base + 4]) == list(got[t])


def test_key_transform_error_all_words():
    # the streaming filter's error bound assumes |x32 - x| <= 3e-6 for every word
    err = pps.selftest_key_error(0, 1 << 32)
    assert err <= 3.0e-6, err


# ------------------------------------------------------------------ workloads

@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_tiny_config_full_size(mode):
    wl = synth.make_workload("tiny")
    fd, fw = check_workload(wl, mode)
    assert fd + fw <= 1


@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_chain4x4_config_full_size(mode):
    wl = synth.make_workload("chain4x4")
    check_workload(wl, mode)


@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_zipf_k8_config_reduced(mode):
    wl = synth.make_workload("zipf_k8", n_seq=3)
    check_workload(wl, mode)


def test_branch16_config_reduced():
    wl = synth.make_workload("branch16", n_seq=1)
    check_workload(wl, pps.DISTINCT)
    check_workload(wl, pps.IID)


@pytest.mark.parametrize("K", [1, 2, 5, 8, 16, 31, 32])
def test_k_sweep_reduced(K):
    wl = synth.make_workload("ksweep", K_sweep=K, n_seq=1, vocab=20000)
    check_workload(wl, pps.DISTINCT)
    check_workload(wl, pps.IID)


# ------------------------------------------------------------------ edge cases

@pytest.mark.parametrize("V,dtype", [(1, torch.float32), (2, torch.bfloat16), (7, torch.bfloat16),
                                     (13, torch.float32), (1003, torch.bfloat16), (4099, torch.float32)])
def test_ragged_vocab(V, dtype):
    K = min(4, V)
    br = (K, 1) if V > 1 else (1,)
    wl = synth.make_workload("chain4x4", n_seq=5, vocab=V, branching=br, dtype=dtype, seed=11 + V)
    check_workload(wl, pps.DISTINCT)
    check_workload(wl, pps.IID)


def test_list_as_long_as_vocab():
    wl = synth.make_workload("tiny", n_seq=6, vocab=12, branching=(12,), seed=5)
    check_workload(wl, pps.DISTINCT)
    check_workload(wl, pps.IID)


def test_unaligned_rows_take_scalar_path():
    base = synth.make_workload("chain4x4", n_seq=3, vocab=2001, seed=21)
    for attr in ("p_logits", "q_logits"):
        x = getattr(base, attr)
        wide = torch.zeros(x.shape[0], x.shape[1] + 3, dtype=x.dtype)
        wide[:, 1:1 + x.shape[1]] = x
        setattr(base, attr, wide.cuda()[:, 1:1 + x.shape[1]])  # row stride V+3, start offset 1 element
    check_workload(base, pps.DISTINCT)


def test_masked_and_infinite_logits():
    wl = synth.make_workload("chain4x4", n_seq=4, vocab=3000, dtype=torch.float32, seed=31)
    p, q = wl.p_logits, wl.q_logits
    rng = np.random.default_rng(0)
    for x in (p, q):
        m = torch.as_tensor(rng.random(x.shape) < 0.3)
        x[m] = float("-inf")
        x[torch.as_tensor(rng.random(x.shape) < 0.01)] = float("nan")
    p[3, :] = float("-inf")       # a node with no usable token: winner -1
    p[5, 17] = float("inf")       # +inf logits win, lowest index first
    p[5, 2000] = float("inf")
    q[2, :-3] = float("-inf")     # fewer usable tokens than the list length
    q[6, 100] = float("inf")
    gd, gv, status = run_gpu(wl)
    od, ov = run_oracle(wl)
    assert status == 0
    compare_draft(gd, od)
    compare_winners(gv["winner"], gv["word"], ov["winner"], ov["word"], ov["margin"])
    assert gv["winner"][3] == -1 and gv["winner"][5] == 17
    assert list(gd["tok"][2][: 3]) == list(od["tok"][2][:3])
    t = wl.tree
    ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, gd["tok"], gd["ndist"], t.child_node, gv["winner"],
                     gv["word"])
    assert np.array_equal(gv["emitted"], ow["emitted"]) and np.array_equal(gv["n_emitted"], ow["n_emitted"])


def test_temperature():
    wl = synth.make_workload("chain4x4", n_seq=3, vocab=5000, seed=41)
    wl.temperature = 0.6
    check_workload(wl, pps.DISTINCT)
    wl.temperature = 1.7
    check_workload(wl, pps.IID)


def test_many_short_rows():
    wl = synth.make_workload("tiny", n_seq=3000, vocab=40, branching=(3, 1), seed=51)
    check_workload(wl, pps.DISTINCT)


def test_near_ties_are_resolved_exactly():
    # fp32 logits built so that pairs of tokens have race keys within ~1e-7 of each other: the fp32
    # stage cannot order them, the fp64 stage must
    n, V = 40, 600
    key, ctx, pos = _rand_ids(n, 61)
    rng = np.random.default_rng(62)
    logits = rng.normal(0, 1.0, (n, V)).astype(np.float32)
    for r in range(n):
        w = oracle.words(key[r:r + 1], ctx[r:r + 1], pos[r:r + 1], V)[0]
        x = np.array([math.log(oracle.exp1(int(v))) for v in w])
        s = x - logits[r]
        order = np.argsort(s)
        a, b = order[0], order[1 + r % 3]
        # make b's key equal a's up to float rounding of the logit
        logits[r, b] = np.float32(x[b] - s[a] + (1e-7 if r % 2 else -1e-7))
    L = torch.as_tensor(logits).cuda()
    ids = dev_ids(key, ctx, pos)
    win_o, wd_o, _, mg_o = oracle.target_rows(logits, key, ctx, pos)
    d_o = oracle.draft_rows(logits, key, ctx, pos, 4, mode=oracle.DISTINCT)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = pps.draft_list(L, *ids, 4, status=status)
    torch.cuda.synchronize()
    got = d["tok"].cpu().numpy()
    exact = 0
    for r in range(n):
        if d_o["min_gap"][r] > 1e-12:
            assert list(got[r]) == list(d_o["tok"][r]), (r, got[r], d_o["tok"][r], d_o["min_gap"][r])
            exact += 1
    assert exact >= n - 2 and int(status.item()) == 0


def test_iid_multi_arrival_near_ties_are_resolved_exactly():
    # fp32 logits built so that a token's second arrival ties another token's first arrival
    # within ~1e-7: the fp32 IID epilogue must see the tie and hand the row to the fp64 stage
    n, V, K = 60, 600, 4
    key, ctx, pos = _rand_ids(n, 71)
    rng = np.random.default_rng(72)
    logits = rng.normal(0, 1.0, (n, V)).astype(np.float32)
    for r in range(n):
        w1 = oracle.words(key[r:r + 1], ctx[r:r + 1], pos[r:r + 1], V)[0]
        w2 = oracle.words(key[r:r + 1], ctx[r:r + 1], pos[r:r + 1], V, 2)[0]
        x = np.array([math.log(oracle.exp1(int(v))) for v in w1])
        s = x - logits[r]
        order = np.argsort(s)
        a, b = order[0], order[1 + r % 3]
        g2 = math.log(oracle.exp1(int(w1[b])) + oracle.exp1(int(w2[b])))
        logits[r, b] = np.float32(g2 - s[a] + (1e-7 if r % 2 else -1e-7))
    L = torch.as_tensor(logits).cuda()
    ids = dev_ids(key, ctx, pos)
    d_o = oracle.draft_rows(logits, key, ctx, pos, K, mode=oracle.IID)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = pps.draft_list(L, *ids, K, mode=pps.IID, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for name, want in (("samples", d_o["labels"]), ("mult", d_o["mult"]), ("tok", d_o["tok"])):
        got = d[name].cpu().numpy()
        for r in range(n):
            if d_o["min_gap"][r] > 1e-12:
                assert list(got[r]) == list(want[r]), (name, r, got[r], want[r])


@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_k32_full_vocab_lists_complete(mode):
    # k = 32 fills the 32-entry list: the left-out-key drop bound must prove every row complete
    wl = synth.make_workload("ksweep", K_sweep=32, n_seq=2)
    gd, gv, status = run_gpu(wl, mode)
    assert status == 0
    t = wl.tree
    roots = np.nonzero(t.row_k == 32)[0]
    sel = torch.as_tensor(roots)
    od = oracle.draft_rows(wl.q_logits[sel].float().numpy(), synth.u64(wl.draft_key[sel]),
                           synth.u64(wl.draft_ctx[sel]), synth.u32(wl.draft_pos[sel]), 32, mode=mode)
    sub = {k: (x[roots] if x is not None and x.ndim >= 1 and x.shape[0] == t.n_draft else x) for k, x in gd.items()}
    compare_draft(sub, od, rows=roots)


def test_crowded_k32_boundary_is_rescanned_exactly():
    # the 32nd and 33rd race keys tie within ~1e-7: the list cannot prove itself complete and the
    # row is finished by the exact second pass
    n, V, K = 24, 600, 32
    key, ctx, pos = _rand_ids(n, 81)
    rng = np.random.default_rng(82)
    logits = rng.normal(0, 1.0, (n, V)).astype(np.float32)
    for r in range(n):
        w = oracle.words(key[r:r + 1], ctx[r:r + 1], pos[r:r + 1], V)[0]
        x = np.array([math.log(oracle.exp1(int(v))) for v in w])
        s = x - logits[r]
        order = np.argsort(s)
        a, b = order[31], order[32 + r % 3]
        logits[r, b] = np.float32(x[b] - s[a] + (1e-7 if r % 2 else -1e-7))
    L = torch.as_tensor(logits).cuda()
    ids = dev_ids(key, ctx, pos)
    d_o = oracle.draft_rows(logits, key, ctx, pos, K, mode=oracle.DISTINCT)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = pps.draft_list(L, *ids, K, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    got = d["tok"].cpu().numpy()
    for r in range(n):
        if d_o["min_gap"][r] > 1e-12:
            assert list(got[r]) == list(d_o["tok"][r]), (r, got[r], d_o["tok"][r])


def test_workspace_reuse_is_deterministic():
    wl = synth.make_workload("chain4x4", n_seq=4, vocab=9000, seed=71)
    a = run_gpu(wl)
    b = run_gpu(wl)
    for k in a[0]:
        if a[0][k] is not None:
            assert np.array_equal(a[0][k], b[0][k])
    for k in ("winner", "word", "accept_len", "emitted"):
        assert np.array_equal(a[1][k], b[1][k])


# ------------------------------------------------------------------ detector

def test_wm_score_matches_oracle_with_segments():
    n = 100003
    key, ctx, pos = _rand_ids(n, 81)
    rng = np.random.default_rng(82)
    tok = rng.integers(0, 150000, n).astype(np.int32)
    cuts = np.sort(rng.choice(np.arange(1, n), 700, replace=False))
    seg = np.concatenate([[0], cuts, [cuts[-1]], [n]]).astype(np.int64)  # includes an empty segment
    so, ss = oracle.wm_score(tok, key, ctx, pos, seg_off=seg)
    sg, sums = pps.wm_score(torch.as_tensor(tok).cuda(), *dev_ids(key, ctx, pos), seg_off=torch.as_tensor(seg).cuda())
    torch.cuda.synchronize()
    np.testing.assert_allclose(sg.cpu().numpy(), so, rtol=1e-5, atol=0)
    np.testing.assert_allclose(sums.cpu().numpy(), ss, rtol=1e-5, atol=1e-9)
    _, tot = pps.wm_score(torch.as_tensor(tok).cuda(), *dev_ids(key, ctx, pos), want_scores=False)
    assert tot.item() == pytest.approx(so.sum(), rel=1e-6)
    assert stats.kstest(sg.cpu().numpy(), "expon").pvalue > 1e-4  # keys independent of the tokens: null law


def test_wm_score_of_emitted_tokens_matches_walk():
    wl = synth.make_workload("zipf_k8", n_seq=2, vocab=30000, seed=91)
    gd, gv, _ = run_gpu(wl)
    t = wl.tree
    # regenerate the emitted tokens' scores from their nodes' ids
    toks, ks, cs, ps, ref = [], [], [], [], []
    key, ctx, pos = synth.u64(wl.node_key), synth.u64(wl.node_ctx), synth.u32(wl.node_pos)
    for s in range(t.n_seq):
        c = t.seq_off[s]
        for m in range(gv["n_emitted"][s]):
            toks.append(gv["emitted"][s][m]); ks.append(key[c]); cs.append(ctx[c]); ps.append(pos[c])
            ref.append(gv["score"][s][m])
            if m + 1 < gv["n_emitted"][s]:
                dr = t.node_draft_row[c]
                k = list(gd["tok"][dr][:gd["ndist"][dr]]).index(gv["emitted"][s][m])
                c = t.child_node[dr][k]
    sg, _ = pps.wm_score(torch.as_tensor(np.array(toks, np.int32)).cuda(), *dev_ids(ks, cs, ps))
    np.testing.assert_allclose(sg.cpu().numpy(), np.array(ref), rtol=1e-5)


# ------------------------------------------------------------------ invariance

def test_drafter_invariance_on_gpu():
    wl = synth.make_workload("chain4x4", n_seq=6, vocab=4000, seed=101)
    _, v1, _ = run_gpu(wl)
    wl.q_logits = (wl.q_logits.float() + torch.randn(wl.q_logits.shape) * 3.0).to(wl.dtype)
    _, v2, _ = run_gpu(wl)
    assert np.array_equal(v1["winner"], v2["winner"]) and np.array_equal(v1["word"], v2["word"])
