"""The dynamic IID draft tree (Alg. 4 with MPFR lists, Eq. 4) on the GPU.

Each context c of depth d draws nu(c) i.i.d. samples (pps_draft_list in IID
mode); every distinct label u becomes a child c||u that draws nu(c||u) = its
multiplicity, so a sequence keeps K draft paths at every depth.  The drafter
is the caller's: `draft_logits(depth, key, ctx, pos)` returns the logits of a
depth's rows (a model forward on those contexts).  The tree lives in the
fixed-capacity layout of pps_tree_expand (include/pps.h): nodes
sequence-major (so seq_off and node_draft_row never change), draft rows
depth-major (so each depth's lists are written in place by one call).  The
target model then scores every node slot and pps_verify_tree walks the tree.

This module only allocates and sequences library calls; all arithmetic runs
in libpps.
"""
from __future__ import annotations

import numpy as np
import torch

from . import pps


class TreeBuilder:
    """Buffers for the dynamic IID trees of n_seq sequences (reused by every `run`)."""

    def __init__(self, n_seq: int, K: int, gamma: int, device="cuda"):
        self.n_seq, self.K, self.gamma = n_seq, K, gamma
        dev = torch.device(device)
        N1 = 1 + K * gamma
        self.n_nodes = n_seq * N1
        self.n_draft = n_seq * (1 + K * (gamma - 1))
        self.depth_start = [0] + [n_seq * (1 + (d - 1) * K) for d in range(1, gamma + 1)]
        self.width = [1] + [K] * gamma
        i32, i64 = dict(dtype=torch.int32, device=dev), dict(dtype=torch.int64, device=dev)
        self.seq_off = torch.arange(n_seq + 1, **i32) * N1
        ndr = np.full((n_seq, N1), -1, np.int64)
        for d in range(gamma):
            off = 0 if d == 0 else 1 + (d - 1) * K
            w = self.width[d]
            ndr[:, off:off + w] = self.depth_start[d] + np.arange(n_seq)[:, None] * w + np.arange(w)[None, :]
        self.node_draft_row = torch.as_tensor(ndr.ravel().astype(np.int32), device=dev)
        self.node_key = torch.zeros(self.n_nodes, **i64)
        self.node_ctx = torch.zeros(self.n_nodes, **i64)
        self.node_pos = torch.zeros(self.n_nodes, **i32)
        self.draft_tok = torch.full((self.n_draft, K), -1, **i32)
        self.draft_mult = torch.zeros((self.n_draft, K), **i32)
        self.draft_ndist = torch.zeros(self.n_draft, **i32)
        self.child_node = torch.full((self.n_draft, K), -1, **i32)
        # identities and nu of every depth's rows, depth-major like the draft rows
        self.row_key = torch.zeros(self.depth_start[gamma] + n_seq * K, **i64)
        self.row_ctx = torch.zeros_like(self.row_key)
        self.row_pos = torch.zeros(self.row_key.numel(), **i32)
        self.row_k = torch.zeros(self.row_key.numel(), **i32)
        self.roots = self.seq_off[:-1].long()
        self.ws = pps.workspace(n_seq * K, 0, dev)

    def rows(self, d: int) -> slice:
        return slice(self.depth_start[d], self.depth_start[d] + self.n_seq * self.width[d])

    def run(self, root_key, root_ctx, root_pos, draft_logits, temperature: float = 1.0, top_k: int = 0,
            top_p: float = 1.0, stream=None):
        """Draft the trees: per depth one pps_draft_list (IID) and one pps_tree_expand."""
        K = self.K
        s0 = self.rows(0)
        self.row_key[s0], self.row_ctx[s0], self.row_pos[s0] = root_key, root_ctx, root_pos
        self.row_k[s0] = K
        self.node_key[self.roots], self.node_ctx[self.roots], self.node_pos[self.roots] = root_key, root_ctx, root_pos
        for d in range(self.gamma):
            s, sn = self.rows(d), self.rows(d + 1)
            key, ctx, pos, k = self.row_key[s], self.row_ctx[s], self.row_pos[s], self.row_k[s]
            out = dict(tok=self.draft_tok[s], key=None, mult=self.draft_mult[s], ndist=self.draft_ndist[s],
                       samples=None)
            pps.draft_list(draft_logits(d, key, ctx, pos), key, ctx, pos, K, row_k=k, mode=pps.IID,
                           temperature=temperature, ws=self.ws, out=out, top_k=top_k, top_p=top_p, stream=stream)
            nxt = dict(key=self.row_key[sn], ctx=self.row_ctx[sn], pos=self.row_pos[sn], k=self.row_k[sn])
            pps.tree_expand(K, self.gamma, d, out, key, ctx, pos, k, nxt, self.child_node,
                            dict(key=self.node_key, ctx=self.node_ctx, pos=self.node_pos), stream=stream)
        return self

    def verify(self, p_logits, temperature: float = 1.0, top_k: int = 0, top_p: float = 1.0, ws=None, out=None,
               status=None, stream=None):
        """The target race over every node slot and the walk (pps_verify_tree)."""
        return pps.verify_tree(p_logits, self.node_key, self.node_ctx, self.node_pos, self.gamma, self.seq_off,
                               self.node_draft_row, self.draft_tok, self.draft_ndist, self.child_node,
                               temperature=temperature, ws=ws, out=out, status=status, stream=stream, top_k=top_k,
                               top_p=top_p)


def build(root_key, root_ctx, root_pos, K: int, gamma: int, draft_logits, **kw) -> TreeBuilder:
    """Draft dynamic IID trees for the root contexts (n_seq tensors) with fresh buffers."""
    return TreeBuilder(root_key.numel(), K, gamma, root_key.device).run(root_key, root_ctx, root_pos, draft_logits,
                                                                        **kw)


class HeteroTreeBuilder:
    """Draft trees of B non-identical proposals (App. A, heterogeneous
    proposals, applied at every node): proposal b drafts a chain of gamma
    tokens with its own model, one pps_draft_hetero row per proposal and depth;
    chains that agree share nodes (pps_hetero_expand), so node c's draft list
    is the set of distinct tokens its proposals drew.  The target race at
    every node is the plain race (the augmented race's token), and
    pps_verify_tree walks the tree with K = B.  The drafter is the caller's:
    `draft_logits(depth, key, ctx, pos, block)` returns the logits of a
    depth's n_seq * B proposal rows (row s * B + b from proposal b's model)."""

    def __init__(self, n_seq: int, B: int, gamma: int, device="cuda"):
        self.n_seq, self.B, self.gamma = n_seq, B, gamma
        dev = torch.device(device)
        N1 = 1 + B * gamma
        self.n_nodes = n_seq * N1
        self.n_lists = n_seq * (1 + B * (gamma - 1))
        list_start = [0] + [n_seq * (1 + (d - 1) * B) for d in range(1, gamma + 1)]
        width = [1] + [B] * gamma
        i32, i64 = dict(dtype=torch.int32, device=dev), dict(dtype=torch.int64, device=dev)
        self.seq_off = torch.arange(n_seq + 1, **i32) * N1
        ndr = np.full((n_seq, N1), -1, np.int64)
        for d in range(gamma):
            off = 0 if d == 0 else 1 + (d - 1) * B
            w = width[d]
            ndr[:, off:off + w] = list_start[d] + np.arange(n_seq)[:, None] * w + np.arange(w)[None, :]
        self.node_draft_row = torch.as_tensor(ndr.ravel().astype(np.int32), device=dev)
        self.node_key = torch.zeros(self.n_nodes, **i64)
        self.node_ctx = torch.zeros(self.n_nodes, **i64)
        self.node_pos = torch.zeros(self.n_nodes, **i32)
        self.list_tok = torch.full((self.n_lists, B), -1, **i32)
        self.list_nd = torch.zeros(self.n_lists, **i32)
        self.child_node = torch.full((self.n_lists, B), -1, **i32)
        # proposal rows, depth-major: depth d's row (s, b) = d * n_seq * B + s * B + b
        nr = gamma * n_seq * B
        self.row_key = torch.zeros(nr, **i64)
        self.row_ctx = torch.zeros(nr, **i64)
        self.row_pos = torch.zeros(nr, **i32)
        self.row_owner = torch.zeros(nr, **i32)
        self.row_block = torch.arange(B, **i32).repeat(n_seq * gamma)
        self.draft_tok = torch.full((nr,), -1, **i32)
        self.roots = self.seq_off[:-1].long()
        self.ws = pps.workspace(n_seq * B, 0, dev)

    def rows(self, d: int) -> slice:
        n = self.n_seq * self.B
        return slice(d * n, (d + 1) * n)

    def run(self, root_key, root_ctx, root_pos, draft_logits, temperature: float = 1.0, top_k: int = 0,
            top_p: float = 1.0, stream=None):
        """Draft the trees: per depth one pps_draft_hetero and one pps_hetero_expand."""
        B = self.B
        s0 = self.rows(0)
        self.row_key[s0] = root_key.repeat_interleave(B)
        self.row_ctx[s0] = root_ctx.repeat_interleave(B)
        self.row_pos[s0] = root_pos.repeat_interleave(B)
        self.row_owner[s0] = 0
        self.node_key[self.roots], self.node_ctx[self.roots], self.node_pos[self.roots] = root_key, root_ctx, root_pos
        lists = dict(tok=self.list_tok, ndist=self.list_nd, child=self.child_node)
        nodes = dict(key=self.node_key, ctx=self.node_ctx, pos=self.node_pos)
        for d in range(self.gamma):
            s = self.rows(d)
            key, ctx, pos, blk = self.row_key[s], self.row_ctx[s], self.row_pos[s], self.row_block[s]
            pps.draft_hetero(draft_logits(d, key, ctx, pos, blk), key, ctx, pos, blk, B, temperature=temperature,
                             ws=self.ws, out_tok=self.draft_tok[s], stream=stream, top_k=top_k, top_p=top_p)
            nxt = None
            if d + 1 < self.gamma:
                sn = self.rows(d + 1)
                nxt = dict(key=self.row_key[sn], ctx=self.row_ctx[sn], pos=self.row_pos[sn], owner=self.row_owner[sn])
            pps.hetero_expand(B, self.gamma, d, self.draft_tok[s], key, ctx, pos, self.row_owner[s], nxt, lists,
                              nodes, stream=stream)
        return self

    def verify(self, p_logits, temperature: float = 1.0, top_k: int = 0, top_p: float = 1.0, ws=None, out=None,
               status=None, stream=None):
        """The target race over every node slot and the walk (pps_verify_tree, K = B)."""
        return pps.verify_tree(p_logits, self.node_key, self.node_ctx, self.node_pos, self.gamma, self.seq_off,
                               self.node_draft_row, self.list_tok, self.list_nd, self.child_node,
                               temperature=temperature, ws=ws, out=out, status=status, stream=stream, top_k=top_k,
                               top_p=top_p)


def build_hetero(root_key, root_ctx, root_pos, B: int, gamma: int, draft_logits, **kw) -> HeteroTreeBuilder:
    """Draft the trees of B proposals for the root contexts (n_seq tensors) with fresh buffers."""
    return HeteroTreeBuilder(root_key.numel(), B, gamma, root_key.device).run(root_key, root_ctx, root_pos,
                                                                              draft_logits, **kw)
