"""GPU parity of the LM head with the race fused into it (pps_lmhead_*).

* pps_lmhead_logits (tcgen05 GEMM, bf16 operands, fp32 accumulation) against
  the oracle's fp64 product: exactly, on dyadic operands whose partial sums
  are all representable (any summation order gives the exact value); within
  the worst-case accumulation bound 2 d 2^-23 sum_j |h_j w_j| otherwise.
* pps_lmhead_draft_list / pps_lmhead_verify_tree against the unfused path
  (pps_lmhead_logits, then pps_draft_list / pps_verify_tree on its fp32
  logits): bit for bit, since both race the same accumulator values exactly.
* The fused path against the oracle's race on the oracle's logits, on dyadic
  operands (identical logits), with the flip rule of tests/parity.py.
* The benchmark's LM-head workload at full size (V = 128256, d = 4096 target
  and 2048 draft, 2624 + 2112 rows): fused against unfused on every row.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_21858_gb300 import pps, synth
from parity import FLIP_MARGIN, compare_draft, compare_winners

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def _dyadic(n, V, d, seed):
    """hidden in {-1, 0, 1}, weight in {-2..2}/64: every partial sum is a multiple of 1/64 below
    2^7 in magnitude, exact in fp32 whatever the order of the additions."""
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    h = torch.randint(-1, 2, (n, d), generator=g, device="cuda").to(torch.bfloat16)
    w = (torch.randint(-2, 3, (V, d), generator=g, device="cuda").float() / 64.0).to(torch.bfloat16)
    return h, w


def _ids(n, seed):
    rng = np.random.default_rng(seed)
    key = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    ctx = rng.integers(0, 2 ** 64, n, dtype=np.uint64)
    pos = rng.integers(0, 2 ** 32, n, dtype=np.uint32)
    t = lambda a, dt: torch.as_tensor(a.view(dt)).cuda()
    return (key, ctx, pos), (t(key, np.int64), t(ctx, np.int64), t(pos, np.int32))


# ------------------------------------------------------------------ the GEMM

@pytest.mark.parametrize("n,V,d", [(300, 1000, 520), (128, 256, 64), (1, 17, 8), (129, 513, 72), (260, 2048, 1024)])
def test_logits_exact_on_dyadic_operands(n, V, d):
    h, w = _dyadic(n, V, d, n + V + d)
    got = pps.lmhead_logits(h, w)
    torch.cuda.synchronize()
    want = oracle.lmhead_logits(h.float().cpu().numpy(), w.float().cpu().numpy())
    assert np.array_equal(got.cpu().numpy().astype(np.float64), want)


def test_logits_within_the_accumulation_bound():
    n, V, d = 257, 3000, 1040
    g = torch.Generator(device="cuda")
    g.manual_seed(7)
    h = torch.randn(n, d, generator=g, device="cuda").to(torch.bfloat16)
    w = (torch.randn(V, d, generator=g, device="cuda") / d ** 0.5 * 2.0).to(torch.bfloat16)
    got = pps.lmhead_logits(h, w).double().cpu().numpy()
    want = oracle.lmhead_logits(h.float().cpu().numpy(), w.float().cpu().numpy())
    # bf16 x bf16 products are exact in fp32; d - 1 additions, each off by at most 2^-23 relative
    # (truncating adders included), bound the error by 2 d 2^-23 sum_j |h_j w_j|
    mag = (h.float().abs() @ w.float().abs().T).double().cpu().numpy()
    assert np.all(np.abs(got - want) <= 2.0 * d * 2.0 ** -23 * mag)
    # and a sanity check against torch's fp32 product
    ref = (h.float() @ w.float().T).double().cpu().numpy()
    assert np.all(np.abs(got - ref) <= 4.0 * d * 2.0 ** -23 * mag)


def test_logits_into_a_strided_output_and_strided_operands():
    n, V, d = 140, 700, 200
    h0, w0 = _dyadic(n, V, d, 3)
    h = torch.zeros(n, d + 56, dtype=torch.bfloat16, device="cuda")[:, :d]
    h.copy_(h0)
    w = torch.zeros(V, d + 8, dtype=torch.bfloat16, device="cuda")[:, :d]
    w.copy_(w0)
    out = torch.full((n, V + 12), 7.0, device="cuda")
    pps.lmhead_logits(h, w, out=out)
    torch.cuda.synchronize()
    want = oracle.lmhead_logits(h0.float().cpu().numpy(), w0.float().cpu().numpy())
    assert np.array_equal(out[:, :V].cpu().numpy().astype(np.float64), want)
    assert torch.all(out[:, V:] == 7.0)  # nothing written past the vocabulary


# ------------------------------------------------------------------ the fused race

def _normal(n, V, d, seed, scale=2.5):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    h = torch.randn(n, d, generator=g, device="cuda").to(torch.bfloat16)
    w = (torch.randn(V, d, generator=g, device="cuda") * (scale / d ** 0.5)).to(torch.bfloat16)
    return h, w


def _assert_same(a: dict, b: dict, names):
    for k in names:
        if a.get(k) is None and b.get(k) is None:
            continue
        assert torch.equal(a[k], b[k]), k


DRAFT = ("tok", "key", "mult", "ndist", "samples")
VERIFY = ("winner", "word", "accept_len", "n_emitted", "emitted", "score", "score_sum")


@pytest.mark.parametrize("K,mode", [(1, pps.DISTINCT), (4, pps.DISTINCT), (8, pps.DISTINCT), (4, pps.IID),
                                    (8, pps.IID)])
def test_fused_draft_lists_equal_the_unfused_path(K, mode):
    n, V, d = 300, 5000, 520
    h, w = _normal(n, V, d, 11 + K)
    _, (key, ctx, pos) = _ids(n, 12 + K)
    g = torch.Generator(device="cuda")
    g.manual_seed(K)
    row_k = torch.randint(1, K + 1, (n,), generator=g, device="cuda", dtype=torch.int32)
    for T in (1.0, 0.7):
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        fused = pps.lmhead_draft_list(h, w, key, ctx, pos, K, row_k=row_k, mode=mode, temperature=T, status=st)
        logits = pps.lmhead_logits(h, w)
        st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
        ref = pps.draft_list(logits, key, ctx, pos, K, row_k=row_k, mode=mode, temperature=T, status=st2)
        torch.cuda.synchronize()
        assert int(st.item()) == 0 and int(st2.item()) == 0
        _assert_same(fused, ref, DRAFT)


def _tree_case(n_seq, branching, V, d, seed):
    t = synth.make_tree(branching, n_seq)
    hq, wq = _normal(t.n_draft, V, d, seed)
    hp, wp = _normal(t.n_nodes, V, d, seed + 1)
    _, (nk, nc, npos) = _ids(t.n_nodes, seed + 2)
    dn = torch.as_tensor(t.draft_node, device="cuda", dtype=torch.long)
    gi = lambda x: torch.as_tensor(np.asarray(x)).cuda().contiguous()
    return t, hq, wq, hp, wp, (nk, nc, npos), (nk[dn], nc[dn], npos[dn]), gi


@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_fused_verify_tree_equals_the_unfused_path(mode):
    t, hq, wq, hp, wp, nid, did, gi = _tree_case(40, (4, 2, 1), 3000, 264, 21)
    d = pps.lmhead_draft_list(hq, wq, *did, t.K, row_k=gi(t.row_k), mode=mode)
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    fused = pps.lmhead_verify_tree(hp, wp, *nid, t.gamma, gi(t.seq_off), gi(t.node_draft_row), d["tok"], d["ndist"],
                                   gi(t.child_node), status=st)
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    ref = pps.verify_tree(pps.lmhead_logits(hp, wp), *nid, t.gamma, gi(t.seq_off), gi(t.node_draft_row), d["tok"],
                          d["ndist"], gi(t.child_node), status=st2)
    torch.cuda.synchronize()
    assert int(st.item()) == 0 and int(st2.item()) == 0
    _assert_same(fused, ref, VERIFY)
    assert int(fused["accept_len"].sum().item()) > 0


def test_fused_race_matches_the_oracle_on_dyadic_operands():
    # dyadic operands: the GPU's logits are the oracle's exactly, so the fused race must give the
    # oracle's lists and winners (flips only at near-ties below 1e-6) and the oracle's walk
    t = synth.make_tree((3, 1), 50)
    V, d = 1500, 200
    hq, wq = _dyadic(t.n_draft, V, d, 31)
    hp, wp = _dyadic(t.n_nodes, V, d, 32)
    (nk_np, nc_np, np_np), (nk, nc, npos) = _ids(t.n_nodes, 33)
    dn = np.asarray(t.draft_node, np.int64)
    dnt = torch.as_tensor(dn, device="cuda")
    gi = lambda x: torch.as_tensor(np.asarray(x)).cuda().contiguous()
    for mode in (pps.DISTINCT, pps.IID):
        g = pps.lmhead_draft_list(hq, wq, nk[dnt], nc[dnt], npos[dnt], t.K, row_k=gi(t.row_k), mode=mode)
        v = pps.lmhead_verify_tree(hp, wp, nk, nc, npos, t.gamma, gi(t.seq_off), gi(t.node_draft_row), g["tok"],
                                   g["ndist"], gi(t.child_node))
        torch.cuda.synchronize()
        lq = oracle.lmhead_logits(hq.float().cpu().numpy(), wq.float().cpu().numpy()).astype(np.float32)
        lp = oracle.lmhead_logits(hp.float().cpu().numpy(), wp.float().cpu().numpy()).astype(np.float32)
        od = oracle.draft_rows(lq, nk_np[dn], nc_np[dn], np_np[dn], t.K, row_k=t.row_k, mode=mode)
        win, wd, _, mg = oracle.target_rows(lp, nk_np, nc_np, np_np)
        gd = {k: (x.cpu().numpy() if x is not None else None) for k, x in g.items()}
        compare_draft(gd, od)
        compare_winners(v["winner"].cpu().numpy(), v["word"].cpu().numpy().view(np.uint32), win, wd, mg)
        ow = oracle.walk(t.gamma, t.seq_off, t.node_draft_row, gd["tok"], gd["ndist"], t.child_node,
                         v["winner"].cpu().numpy(), v["word"].cpu().numpy().view(np.uint32))
        assert np.array_equal(v["accept_len"].cpu().numpy(), ow["accept_len"])
        assert np.array_equal(v["emitted"].cpu().numpy(), ow["emitted"])
        np.testing.assert_allclose(v["score_sum"].cpu().numpy(), ow["score_sum"], rtol=1e-5)


def test_full_size_lmhead_workload_every_row():
    # the benchmark's LM-head workload: the K = 8 chain tree of 64 sequences, V = 128256, target
    # d = 4096 (2624 node rows), draft d = 2048 (2112 draft rows); fused against unfused everywhere
    wl = synth.lmhead_workload(device="cuda")
    t = wl.tree
    gi = lambda x: torch.as_tensor(np.asarray(x)).cuda().contiguous()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    d = pps.lmhead_draft_list(wl.hq, wl.wq, wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K, row_k=gi(t.row_k),
                              status=st)
    ref_d = pps.draft_list(pps.lmhead_logits(wl.hq, wl.wq), wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K,
                           row_k=gi(t.row_k), status=st)
    args = (t.gamma, gi(t.seq_off), gi(t.node_draft_row), d["tok"], d["ndist"], gi(t.child_node))
    v = pps.lmhead_verify_tree(wl.hp, wl.wp, wl.node_key, wl.node_ctx, wl.node_pos, *args, status=st)
    ref_v = pps.verify_tree(pps.lmhead_logits(wl.hp, wl.wp), wl.node_key, wl.node_ctx, wl.node_pos, *args, status=st)
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    _assert_same(d, ref_d, DRAFT)
    _assert_same(v, ref_v, VERIFY)
    assert 0.5 < float(v["accept_len"].float().mean().item()) <= t.gamma
