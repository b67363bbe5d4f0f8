"""GPU parity of non-identical proposals (the augmented race on V x [B]):
proposal rows (pps_draft_hetero) against the oracle's block races, the
winner's block (pps_hetero_block), the multi-proposal tree (pps_hetero_expand
+ pps_verify_tree) against the oracle depth by depth, and the one-step
acceptance of the product path against the proposition's exact block-matching
probability."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2609_21858_gb300 import pps, synth, tree
from parity import FLIP_MARGIN, TOP_P_MARGIN, compare_winners, dev_ids, f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def u64(t):
    return t.cpu().numpy().view(np.uint64)


def _ids(n, seed):
    rng = np.random.default_rng(seed)
    return (rng.integers(0, 2 ** 64, n, dtype=np.uint64), rng.integers(0, 2 ** 64, n, dtype=np.uint64),
            rng.integers(0, 2 ** 31, n, dtype=np.uint32))


def _check_rows(q, key, ctx, pos, blk, B, T=1.0):
    """Run pps_draft_hetero on q (CUDA) and compare with the oracle; returns the flips."""
    k, c, p = dev_ids(key, ctx, pos)
    bt = torch.as_tensor(blk, dtype=torch.int32).cuda()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    okey = torch.empty(q.shape[0], dtype=torch.float32, device="cuda")
    x = pps.draft_hetero(q, k, c, p, bt, B, temperature=T, status=status, out_key=okey)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    gx, gk = x.cpu().numpy(), okey.cpu().numpy()
    ox, ok, om = oracle.block_draft_rows(q.float().cpu().numpy(), key, ctx, pos, blk, B, T)
    bad = np.nonzero(gx != ox)[0]
    for r in bad:
        assert om[r] < FLIP_MARGIN, f"row {r}: gpu {gx[r]} oracle {ox[r]} margin {om[r]}"
    good = np.setdiff1d(np.nonzero(ox >= 0)[0], bad)
    np.testing.assert_allclose(gk[good], ok[good], rtol=0, atol=5e-5)
    return len(bad)


@pytest.mark.parametrize("B,V,dtype", [(2, 500, torch.float32), (3, 4099, torch.bfloat16),
                                       (8, 32000, torch.bfloat16), (32, 1003, torch.float32),
                                       (1, 2000, torch.bfloat16), (5, 70, torch.bfloat16)])
def test_proposal_rows_match_the_oracle(B, V, dtype):
    n = 96
    rng = np.random.default_rng(B * 1000 + V)
    q = torch.as_tensor(rng.normal(0, 3, (n, V)).astype(np.float32)).to(dtype).cuda()
    key, ctx, pos = _ids(n, V)
    blk = rng.integers(0, B, n).astype(np.int32)
    _check_rows(q, key, ctx, pos, blk, B)


def test_proposal_rows_zipf_logits_and_temperature():
    n, V, B = 64, 20000, 4
    ctx = synth.splitmix64_stream(5, n)
    q = torch.as_tensor(synth.label_logits(ctx, V, seed=3)).to(torch.bfloat16).cuda()
    key, _, pos = _ids(n, 6)
    blk = np.arange(n, dtype=np.int32) % B
    for T in (0.6, 1.0, 1.8):
        _check_rows(q, key, ctx, pos, blk, B, T)


def test_proposal_rows_masked_nan_short_and_unaligned():
    n, V, B = 40, 3001, 6
    rng = np.random.default_rng(9)
    x = rng.normal(0, 2, (n, V)).astype(np.float32)
    x[rng.random(x.shape) < 0.3] = -np.inf
    x[rng.random(x.shape) < 0.01] = np.nan
    x[3, :] = -np.inf          # nothing usable: -1
    x[5, :] = -np.inf
    x[5, 1234] = 0.5           # one usable token
    x[7, :-2] = np.nan         # two usable tokens
    key, ctx, pos = _ids(n, 10)
    blk = rng.integers(0, B, n).astype(np.int32)
    _check_rows(torch.as_tensor(x).cuda(), key, ctx, pos, blk, B)
    # unaligned rows take the scalar path
    wide = torch.zeros(n, V + 3, dtype=torch.bfloat16)
    wide[:, 1:1 + V] = torch.as_tensor(x).to(torch.bfloat16)
    _check_rows(wide.cuda()[:, 1:1 + V], key, ctx, pos, blk, B)


def test_full_size_proposal_rows_sampled():
    # the bench's proposal rows: 8 proposals x 64 sequences, V = 128256, bf16; 48 rows checked
    n, V, B = 512, 128256, 8
    g = torch.Generator(device="cuda")
    g.manual_seed(4)
    q = synth._zipf(g, n, V, 1.0, True, "cuda").to(torch.bfloat16)
    key, ctx, pos = _ids(n, 12)
    blk = np.arange(n, dtype=np.int32) % B
    k, c, p = dev_ids(key, ctx, pos)
    x = pps.draft_hetero(q, k, c, p, torch.as_tensor(blk).cuda(), B)
    torch.cuda.synchronize()
    rows = np.sort(np.random.default_rng(1).choice(n, 48, replace=False))
    ox, _, om = oracle.block_draft_rows(q[torch.as_tensor(rows, device="cuda")].float().cpu().numpy(), key[rows],
                                        ctx[rows], pos[rows], blk[rows], B)
    gx = x.cpu().numpy()[rows]
    for i in np.nonzero(gx != ox)[0]:
        assert om[i] < FLIP_MARGIN


def test_block_key_logarithm_error_is_within_its_bound():
    # the fp32 block key's bound (kBlkErr) assumes lg2.approx errs by at most 2^-17
    # over the key's whole input range; checked over every fp32 input there
    assert pps.selftest_lg2_error(2.0 ** -40, 2.0 ** 7) <= 2.0 ** -17


def test_winner_blocks_match_the_oracle():
    n = 5000
    rng = np.random.default_rng(2)
    key, ctx, pos = _ids(n, 3)
    tok = rng.integers(-1, 128256, n).astype(np.int32)
    k, c, p = dev_ids(key, ctx, pos)
    for B in (1, 2, 7, 32):
        j = pps.hetero_block(torch.as_tensor(tok).cuda(), k, c, p, B).cpu().numpy()
        want = np.array([oracle.block_j(int(key[t]), int(ctx[t]), int(pos[t]), int(tok[t]), B) if tok[t] >= 0
                         else -1 for t in range(n)])
        assert np.array_equal(j, want)


@pytest.mark.parametrize("B,gamma,V,dtype", [(4, 3, 500, torch.float32), (8, 5, 4000, torch.bfloat16),
                                             (1, 2, 300, torch.float32), (3, 4, 50, torch.bfloat16)])
def test_hetero_tree_matches_the_oracle(B, gamma, V, dtype):
    n_seq = 24
    rng = np.random.default_rng(B * 100 + gamma)
    key = torch.as_tensor(rng.integers(0, 2 ** 63, n_seq, dtype=np.int64)).cuda()
    ctx = torch.as_tensor(rng.integers(0, 2 ** 63, n_seq, dtype=np.int64)).cuda()
    pos = torch.as_tensor(rng.integers(0, 5000, n_seq, dtype=np.int32)).cuda()
    seen = []

    def draft_logits(d, k_, c_, p_, b_):
        # proposal b's "model": label logits with its own seed; few tokens at V = 50 so chains meet
        cc, bb = u64(c_), b_.cpu().numpy()
        lg = np.empty((cc.size, V), np.float32)
        for b in range(B):
            sel = bb == b
            lg[sel] = synth.label_logits(cc[sel], V, seed=100 + b, noise=1.0 + 0.3 * b)
        seen.append((u64(k_), cc, p_.cpu().numpy().view(np.uint32), bb, lg))
        return torch.as_tensor(lg).to(dtype).cuda()

    t = tree.build_hetero(key, ctx, pos, B, gamma, draft_logits)
    torch.cuda.synchronize()
    N1 = 1 + B * gamma
    otree = oracle.hetero_tree(n_seq, B, gamma)
    roots = np.arange(n_seq) * N1
    otree["node_key"][roots], otree["node_ctx"][roots], otree["node_pos"][roots] = (
        u64(key), u64(ctx), pos.cpu().numpy().view(np.uint32))
    okey, octx, opos = (np.repeat(u64(key), B), np.repeat(u64(ctx), B),
                        np.repeat(pos.cpu().numpy().view(np.uint32), B))
    oown = np.zeros(n_seq * B, np.int32)
    for d in range(gamma):
        gk, gc, gp, gb, lg = seen[d]
        s = t.rows(d)
        assert np.array_equal(gk, okey) and np.array_equal(gc, octx) and np.array_equal(gp, opos)
        assert np.array_equal(t.row_owner[s].cpu().numpy(), oown)
        lgo = torch.as_tensor(lg).to(dtype).float().numpy()
        ox, _, om = oracle.block_draft_rows(lgo, okey, octx, opos, gb, B)
        gx = t.draft_tok[s].cpu().numpy()
        alive = oown >= 0
        for r in np.nonzero(alive & (gx != ox))[0]:
            assert om[r] < FLIP_MARGIN, (d, r, gx[r], ox[r], om[r])
        okey, octx, opos, oown = oracle.hetero_expand(n_seq, B, gamma, d, gx, okey, octx, opos, oown, otree)
    for name, g in (("list_tok", t.list_tok), ("list_nd", t.list_nd), ("child_node", t.child_node)):
        assert np.array_equal(g.cpu().numpy(), otree[name]), name
    for name in ("node_key", "node_ctx"):
        assert np.array_equal(u64(getattr(t, name)), otree[name]), name
    assert np.array_equal(t.node_pos.cpu().numpy().view(np.uint32), otree["node_pos"])
    # target race over every node slot (the plain race), then the walk over the node lists
    plg = synth.label_logits(u64(t.node_ctx), V, seed=11)
    p = torch.as_tensor(plg).to(dtype).cuda()
    v = t.verify(p)
    torch.cuda.synchronize()
    win, wd, _, mg = oracle.target_rows(torch.as_tensor(plg).to(dtype).float().numpy(), u64(t.node_key),
                                        u64(t.node_ctx), t.node_pos.cpu().numpy().view(np.uint32))
    gw, gword = v["winner"].cpu().numpy(), v["word"].cpu().numpy().view(np.uint32)
    compare_winners(gw, gword, win, wd, mg)
    ow = oracle.walk(gamma, t.seq_off.cpu().numpy(), t.node_draft_row.cpu().numpy(), t.list_tok.cpu().numpy(),
                     t.list_nd.cpu().numpy(), t.child_node.cpu().numpy(), gw, gword)
    assert np.array_equal(v["accept_len"].cpu().numpy(), ow["accept_len"])
    assert np.array_equal(v["emitted"].cpu().numpy(), ow["emitted"])


def test_one_step_acceptance_is_the_propositions_coupling():
    # gamma = 1, the same P and Q_b at every sequence: the block-matching event
    # {X^(J) = Y} has probability sum_(i,b) p_i / (B + alpha_i^(b)) (the
    # proposition's bound) and acceptance is at least that
    n_seq, B, V = 40000, 3, 6
    rng = np.random.default_rng(21)
    pl, ql = rng.normal(0, 1, V), rng.normal(0, 1.4, (B, V))
    p = np.exp(pl - pl.max())
    p /= p.sum()
    q = np.exp(ql - ql.max(1, keepdims=True))
    q /= q.sum(1, keepdims=True)
    alpha = np.array([[p[i] * np.maximum(q[b] / q[b, i] - p / p[i], 0).sum() for b in range(B)] for i in range(V)])
    bound = (p[:, None] / (B + alpha)).sum()
    key, ctx, pos = dev_ids(*_ids(n_seq, 22))
    qt = torch.as_tensor(np.tile(ql.astype(np.float32), (n_seq, 1))).cuda()
    t = tree.build_hetero(key, ctx, pos, B, 1, lambda *_: qt)
    pt = torch.as_tensor(np.broadcast_to(pl.astype(np.float32), (t.n_nodes, V)).copy()).cuda()
    v = t.verify(pt)
    y = v["winner"][t.roots]
    j = pps.hetero_block(y.contiguous(), key, ctx, pos, B)
    x = t.draft_tok[t.rows(0)].view(n_seq, B)
    hit = (x.gather(1, j.long().view(-1, 1)).view(-1) == y).float().mean().item()
    acc = v["accept_len"].float().mean().item()
    sd = math.sqrt(bound * (1 - bound) / n_seq)
    assert abs(hit - bound) < 4.5 * sd, (hit, bound)
    assert acc >= hit
    assert acc >= bound - 4.5 * sd


# ---------------------------------------------------------------- truncated proposal rows

def _check_trunc_rows(q, key, ctx, pos, blk, B, top_k, top_p, T=1.0):
    k, c, p = dev_ids(key, ctx, pos)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    x = pps.draft_hetero(q, k, c, p, torch.as_tensor(blk, dtype=torch.int32).cuda(), B, temperature=T,
                         status=status, top_k=top_k, top_p=top_p)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    # the oracle gets top_p and T as the fp32 values the C ABI receives
    qm, loose = oracle.truncate_rows(q.float().cpu().numpy(), top_k, f32(top_p), f32(T))
    ox, _, om = oracle.block_draft_rows(qm, key, ctx, pos, blk, B, f32(T))
    gx = x.cpu().numpy()
    for r in np.nonzero(gx != ox)[0]:
        assert om[r] < FLIP_MARGIN or loose[r] < TOP_P_MARGIN, (r, gx[r], ox[r], om[r], loose[r])


@pytest.mark.parametrize("top_k,top_p", [(50, 1.0), (5, 0.9), (64, 0.5), (1, 1.0)])
@pytest.mark.parametrize("B,V,dtype", [(3, 4099, torch.bfloat16), (8, 1003, torch.float32),
                                       (32, 20000, torch.bfloat16)])
def test_truncated_proposal_rows_match_the_oracle(top_k, top_p, B, V, dtype):
    n = 64
    ctx = synth.splitmix64_stream(B + V, n)
    q = torch.as_tensor(synth.label_logits(ctx, V, seed=B)).to(dtype).cuda()
    key, _, pos = _ids(n, V + 1)
    blk = (np.arange(n) % B).astype(np.int32)
    _check_trunc_rows(q, key, ctx, pos, blk, B, top_k, top_p)


def test_truncated_proposal_rows_tie_overflow_and_masks():
    # a top-k tie group larger than the 64-entry list (the exact second pass, with block keys)
    n, V, B = 24, 32000, 4
    rng = np.random.default_rng(31)
    x = rng.normal(0, 1, (n, V)).astype(np.float32)
    for r in range(0, n, 2):
        cols = rng.choice(V, 320, replace=False)
        x[r, cols[:20]] = 8.0 + 0.25 * np.arange(20)
        x[r, cols[20:]] = 6.0
    x[1, :] = -np.inf
    x[3, :-5] = np.nan
    q = torch.as_tensor(x).to(torch.bfloat16).cuda()
    key, ctx, pos = _ids(n, 32)
    blk = rng.integers(0, B, n).astype(np.int32)
    for tk, tp in ((40, 1.0), (40, 0.6), (10, 0.999999)):
        _check_trunc_rows(q, key, ctx, pos, blk, B, tk, tp)


def test_truncated_hetero_tree_matches_the_oracle():
    n_seq, B, gamma, V, top_k = 16, 4, 3, 3000, 20
    rng = np.random.default_rng(40)
    key = torch.as_tensor(rng.integers(0, 2 ** 63, n_seq, dtype=np.int64)).cuda()
    ctx = torch.as_tensor(rng.integers(0, 2 ** 63, n_seq, dtype=np.int64)).cuda()
    pos = torch.as_tensor(rng.integers(0, 5000, n_seq, dtype=np.int32)).cuda()
    seen = []

    def draft_logits(d, k_, c_, p_, b_):
        cc, bb = u64(c_), b_.cpu().numpy()
        lg = np.empty((cc.size, V), np.float32)
        for b in range(B):
            lg[bb == b] = synth.label_logits(cc[bb == b], V, seed=200 + b)
        seen.append((u64(k_), cc, p_.cpu().numpy().view(np.uint32), bb, lg))
        return torch.as_tensor(lg).cuda()

    t = tree.build_hetero(key, ctx, pos, B, gamma, draft_logits, top_k=top_k, top_p=0.95)
    torch.cuda.synchronize()
    for d in range(gamma):
        gk, gc, gp, gb, lg = seen[d]
        s = t.rows(d)
        own = t.row_owner[s].cpu().numpy()
        qm, loose = oracle.truncate_rows(lg, top_k, f32(0.95), 1.0)
        ox, _, om = oracle.block_draft_rows(qm, gk, gc, gp, gb, B)
        gx = t.draft_tok[s].cpu().numpy()
        for r in np.nonzero((own >= 0) & (gx != ox))[0]:
            assert om[r] < FLIP_MARGIN or loose[r] < TOP_P_MARGIN
    plg = synth.label_logits(u64(t.node_ctx), V, seed=13)
    v = t.verify(torch.as_tensor(plg).cuda(), top_k=top_k, top_p=0.95)
    torch.cuda.synchronize()
    pm, ploose = oracle.truncate_rows(plg, top_k, f32(0.95), 1.0)
    win, wd, _, mg = oracle.target_rows(pm, u64(t.node_key), u64(t.node_ctx), t.node_pos.cpu().numpy().view(np.uint32))
    gw, gword = v["winner"].cpu().numpy(), v["word"].cpu().numpy().view(np.uint32)
    compare_winners(gw, gword, win, wd, mg, loose=ploose < TOP_P_MARGIN)
    ow = oracle.walk(gamma, t.seq_off.cpu().numpy(), t.node_draft_row.cpu().numpy(), t.list_tok.cpu().numpy(),
                     t.list_nd.cpu().numpy(), t.child_node.cpu().numpy(), gw, gword)
    assert np.array_equal(v["accept_len"].cpu().numpy(), ow["accept_len"])
