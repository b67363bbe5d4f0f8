"""The path shards by sequence with no data exchange: world_size-2 gloo ranks
on CPU each evaluate their contiguous share of the sequences (oracle draft
lists, target races and walks on their rows only) and the gathered result
equals the single-process one.  Also checks bench.py's max-over-ranks timing."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _evaluate(wl, seqs):
    """Oracle decode block for the sequences `seqs` of workload `wl`, using only their rows."""
    import oracle
    from paper_2609_21858_gb300 import synth
    t = wl.tree
    out = {}
    for s in seqs:
        n0, n1 = t.seq_off[s], t.seq_off[s + 1]
        nodes = np.arange(n0, n1)
        drows = np.array([t.node_draft_row[c] for c in nodes if t.node_draft_row[c] >= 0])
        d = oracle.draft_rows(wl.q_logits[drows].float().numpy(), synth.u64(wl.draft_key)[drows],
                              synth.u64(wl.draft_ctx)[drows], synth.u32(wl.draft_pos)[drows], t.K,
                              row_k=t.row_k[drows])
        win, wd, _, _ = oracle.target_rows(wl.p_logits[nodes].float().numpy(), synth.u64(wl.node_key)[nodes],
                                           synth.u64(wl.node_ctx)[nodes], synth.u32(wl.node_pos)[nodes])
        # local renumbering of this sequence's tree
        ndr = np.where(t.node_draft_row[nodes] >= 0, t.node_draft_row[nodes] - drows.min(), -1)
        cn = np.where(t.child_node[drows] >= 0, t.child_node[drows] - n0, -1)
        w = oracle.walk(t.gamma, [0, n1 - n0], ndr, d["tok"], d["ndist"], cn, win, wd)
        out[int(s)] = (list(w["emitted"][0]), int(w["accept_len"][0]), float(w["score_sum"][0]), list(d["tok"].ravel()))
    return out


def _rank_main(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import sys
    sys.path.insert(0, ROOT)
    from paper_2609_21858_gb300 import synth
    import bench
    wl = synth.make_workload("chain4x4", n_seq=6, vocab=300, seed=17)
    n = wl.tree.n_seq
    mine = range(rank * n // world, (rank + 1) * n // world)
    part = _evaluate(wl, mine)
    parts = [None] * world
    dist.all_gather_object(parts, part)
    t = bench.max_over_ranks(float(rank + 1), world)
    if rank == 0:
        merged = {}
        for p in parts:
            merged.update(p)
        q.put((merged, t))
    dist.barrier()
    dist.destroy_process_group()


def test_sequence_sharding_needs_no_exchange():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    merged, tmax = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    from paper_2609_21858_gb300 import synth
    wl = synth.make_workload("chain4x4", n_seq=6, vocab=300, seed=17)
    single = _evaluate(wl, range(wl.tree.n_seq))
    assert merged.keys() == single.keys()
    for s in single:
        assert merged[s][0] == single[s][0] and merged[s][1] == single[s][1] and merged[s][3] == single[s][3]
        assert merged[s][2] == pytest.approx(single[s][2], rel=1e-15)
    assert tmax == 2.0
