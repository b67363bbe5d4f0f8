"""GPU parity of the dynamic IID draft tree: at every depth the GPU's IID
lists against the oracle's on the same contexts and logits, the GPU's
expansion against the oracle's expansion of the GPU lists (bit-exact), then
the target race over every node and the walk."""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_21858_gb300 import pps, synth, tree
from parity import compare_draft, compare_winners

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def u64(t):
    return t.cpu().numpy().view(np.uint64)


@pytest.mark.parametrize("K,gamma,V,dtype", [(4, 3, 500, torch.float32), (8, 5, 4000, torch.bfloat16),
                                             (1, 2, 300, torch.float32), (16, 2, 2000, torch.bfloat16)])
def test_dynamic_tree_matches_the_oracle(K, gamma, V, dtype):
    n_seq = 24
    rng = np.random.default_rng(K * 100 + gamma)
    key = torch.as_tensor(rng.integers(0, 2 ** 63, n_seq, dtype=np.int64)).cuda()
    ctx = torch.as_tensor(rng.integers(0, 2 ** 63, n_seq, dtype=np.int64)).cuda()
    pos = torch.as_tensor(rng.integers(0, 5000, n_seq, dtype=np.int32)).cuda()
    seen = []

    def draft_logits(d, k_, c_, p_):
        lg = synth.label_logits(u64(c_), V, seed=7)
        seen.append((u64(k_), u64(c_), p_.cpu().numpy().view(np.uint32), lg))
        return torch.as_tensor(lg).to(dtype).cuda()

    t = tree.build(key, ctx, pos, K, gamma, draft_logits)
    torch.cuda.synchronize()
    N1 = 1 + K * gamma
    # oracle, depth by depth, expanding the GPU's own lists
    otree = dict(child_node=np.full((t.n_draft, K), -1, np.int32), node_key=np.zeros(n_seq * N1, np.uint64),
                 node_ctx=np.zeros(n_seq * N1, np.uint64), node_pos=np.zeros(n_seq * N1, np.uint32))
    roots = np.arange(n_seq) * N1
    otree["node_key"][roots], otree["node_ctx"][roots], otree["node_pos"][roots] = (
        u64(key), u64(ctx), pos.cpu().numpy().view(np.uint32))
    k = np.full(n_seq, K, np.int32)
    okey, octx, opos = u64(key), u64(ctx), pos.cpu().numpy().view(np.uint32)
    for d in range(gamma):
        gk, gc, gp, lg = seen[d]
        assert np.array_equal(gk, okey) and np.array_equal(gc, octx) and np.array_equal(gp, opos)
        lgo = torch.as_tensor(lg).to(dtype).float().numpy()
        od = oracle.draft_rows(lgo, okey, octx, opos, K, row_k=np.maximum(k, 1), mode=oracle.IID)
        rows = t.rows(d)
        gd = dict(tok=t.draft_tok[rows].cpu().numpy(), mult=t.draft_mult[rows].cpu().numpy(),
                  ndist=t.draft_ndist[rows].cpu().numpy(), samples=None, key=None)
        assert np.array_equal(t.row_k[rows].cpu().numpy(), k)
        present = k > 0
        sub = lambda x: x[present]
        compare_draft({kk: (sub(v) if v is not None else None) for kk, v in gd.items()},
                      {kk: sub(v) for kk, v in od.items()})
        okey, octx, opos, k = oracle.tree_expand(n_seq, K, gamma, d, gd, okey, octx, opos, k, otree)
    assert np.array_equal(t.child_node.cpu().numpy(), otree["child_node"])
    for name in ("node_key", "node_ctx"):
        assert np.array_equal(u64(getattr(t, name)), otree[name]), name
    assert np.array_equal(t.node_pos.cpu().numpy().view(np.uint32), otree["node_pos"])
    # target race over every node slot, then the walk
    plg = synth.label_logits(u64(t.node_ctx), V, seed=11)
    p = torch.as_tensor(plg).to(dtype).cuda()
    v = t.verify(p)
    torch.cuda.synchronize()
    win, wd, _, mg = oracle.target_rows(torch.as_tensor(plg).to(dtype).float().numpy(), u64(t.node_key),
                                        u64(t.node_ctx), t.node_pos.cpu().numpy().view(np.uint32))
    gw, gword = v["winner"].cpu().numpy(), v["word"].cpu().numpy().view(np.uint32)
    compare_winners(gw, gword, win, wd, mg)
    ow = oracle.walk(gamma, t.seq_off.cpu().numpy(), t.node_draft_row.cpu().numpy(), t.draft_tok.cpu().numpy(),
                     t.draft_ndist.cpu().numpy(), t.child_node.cpu().numpy(), gw, gword)
    assert np.array_equal(v["accept_len"].cpu().numpy(), ow["accept_len"])
    assert np.array_equal(v["emitted"].cpu().numpy(), ow["emitted"])
    # the root keeps K paths: every sequence emitted at least its root's winner
    assert np.all(v["n_emitted"].cpu().numpy() >= 1)
