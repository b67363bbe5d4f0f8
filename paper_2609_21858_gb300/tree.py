"""The dynamic IID draft tree (Alg. 4 with MPFR lists, Eq. 4) on the GPU.

Each context c of depth d draws nu(c) i.i.d. samples (pps_draft_list in IID
mode); every distinct label u becomes a child c||u that draws nu(c||u) = its
multiplicity, so a sequence keeps K draft paths at every depth.  The drafter
is the caller's: `draft_logits(depth, key, ctx, pos)` returns the logits of a
depth's rows (a model forward on those contexts).  The tree lives in the
fixed-capacity layout of pps_tree_expand (include/pps.h), so its node and
draft-row numbering, seq_off and node_draft_row never change; the target
model then scores every node slot and pps_verify_tree walks the tree.

This module only allocates and sequences library calls; all arithmetic runs
in libpps.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

from . import pps


@dataclass
class IIDTree:
    n_seq: int
    K: int
    gamma: int
    node_key: torch.Tensor        # [n_seq*N1] identities of every node slot
    node_ctx: torch.Tensor
    node_pos: torch.Tensor
    seq_off: torch.Tensor         # [n_seq+1]
    node_draft_row: torch.Tensor  # [n_seq*N1]
    draft_tok: torch.Tensor       # [n_seq*R1, K] per draft row, in the layout's row order
    draft_mult: torch.Tensor
    draft_ndist: torch.Tensor     # [n_seq*R1]
    child_node: torch.Tensor      # [n_seq*R1, K]
    draft_k: torch.Tensor         # [n_seq*R1] nu of every draft row (0 = absent node)

    @property
    def nodes_per_seq(self) -> int:
        return 1 + self.K * self.gamma

    @property
    def rows_per_seq(self) -> int:
        return 1 + self.K * (self.gamma - 1)


def layout(n_seq: int, K: int, gamma: int, device):
    """seq_off and node_draft_row of the fixed-capacity layout, and the draft-row slots of each depth."""
    N1, R1 = 1 + K * gamma, 1 + K * (gamma - 1)
    seq_off = torch.arange(n_seq + 1, dtype=torch.int32, device=device) * N1
    ndr = np.full(N1, -1, np.int64)
    ndr[:R1] = np.arange(R1)  # node offset o < R1 (depth < gamma) owns draft row offset o
    ndr = np.concatenate([np.where(ndr >= 0, ndr + b * R1, -1) for b in range(n_seq)])
    depth_rows = []
    for d in range(gamma):
        off, w = (0, 1) if d == 0 else (1 + (d - 1) * K, K)
        depth_rows.append(torch.as_tensor((np.arange(n_seq)[:, None] * R1 + off + np.arange(w)[None, :]).ravel(),
                                          device=device))
    return seq_off, torch.as_tensor(ndr.astype(np.int32), device=device), depth_rows


def build(root_key, root_ctx, root_pos, K: int, gamma: int, draft_logits, temperature: float = 1.0,
          top_k: int = 0, top_p: float = 1.0, stream=None) -> IIDTree:
    """Draft a dynamic IID tree of depth gamma for every root context (tensors of n_seq)."""
    dev = root_key.device
    n_seq = root_key.numel()
    N1, R1 = 1 + K * gamma, 1 + K * (gamma - 1)
    seq_off, ndr, depth_rows = layout(n_seq, K, gamma, dev)
    i64 = dict(dtype=torch.int64, device=dev)
    t = IIDTree(n_seq, K, gamma,
                node_key=torch.zeros(n_seq * N1, **i64), node_ctx=torch.zeros(n_seq * N1, **i64),
                node_pos=torch.zeros(n_seq * N1, dtype=torch.int32, device=dev), seq_off=seq_off,
                node_draft_row=ndr,
                draft_tok=torch.full((n_seq * R1, K), -1, dtype=torch.int32, device=dev),
                draft_mult=torch.zeros((n_seq * R1, K), dtype=torch.int32, device=dev),
                draft_ndist=torch.zeros(n_seq * R1, dtype=torch.int32, device=dev),
                child_node=torch.full((n_seq * R1, K), -1, dtype=torch.int32, device=dev),
                draft_k=torch.zeros(n_seq * R1, dtype=torch.int32, device=dev))
    roots = seq_off[:-1].long()
    t.node_key[roots], t.node_ctx[roots], t.node_pos[roots] = root_key, root_ctx, root_pos
    key, ctx, pos = root_key.contiguous(), root_ctx.contiguous(), root_pos.contiguous()
    k = torch.full((n_seq,), K, dtype=torch.int32, device=dev)
    for d in range(gamma):
        logits = draft_logits(d, key, ctx, pos)
        out = pps.draft_list(logits, key, ctx, pos, K, row_k=k, mode=pps.IID, temperature=temperature,
                             top_k=top_k, top_p=top_p, stream=stream)
        rows = depth_rows[d]
        t.draft_tok[rows], t.draft_mult[rows], t.draft_ndist[rows], t.draft_k[rows] = (
            out["tok"], out["mult"], out["ndist"], k)
        # children of this depth (the leaves too: the target model scores them)
        nxt = dict(key=torch.empty(n_seq * K, **i64), ctx=torch.empty(n_seq * K, **i64),
                   pos=torch.empty(n_seq * K, dtype=torch.int32, device=dev),
                   k=torch.empty(n_seq * K, dtype=torch.int32, device=dev))
        pps.tree_expand(K, gamma, d, out, key, ctx, pos, k, nxt, t.child_node,
                        dict(key=t.node_key, ctx=t.node_ctx, pos=t.node_pos), stream=stream)
        key, ctx, pos, k = nxt["key"], nxt["ctx"], nxt["pos"], nxt["k"]
    return t
