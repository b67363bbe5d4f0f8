"""Seeded synthetic workloads shaped like the paper's LLM decoding runs.

This module holds no arithmetic of the sampling method: it only draws
logits, keys, context labels and the static draft-tree topology.  Both the
CUDA path and the CPU oracle consume what it produces.

The paper evaluates Qwen2.5 / Llama-3.1 / Vicuna target-drafter pairs on
CNN/DailyMail and ELI5 (Sec. 5, App. C).  Neither the models nor the datasets
are available, so every workload is synthetic: vocabulary sizes match those
model families (32000, 128256, 152064), logits follow rank-Zipf or
peaked/flat mixtures that mimic next-token logits, and the draft logits are the
target logits plus Gaussian noise, so that draft and target disagree the way a
small drafter does.

Tree topology.  A tree is given by its branching per depth, e.g. ``(8, 1, 1,
1, 1)`` = the root keeps a list of 8 distinct drafts and every child extends
its chain with its top-1 draft ("K chains of depth gamma"), ``(16, 3, 2, 1)``
= static branching.  Nodes are numbered breadth-first inside a sequence and
sequences are contiguous.  Internal nodes (depth < gamma) own one draft row
each, in node order; list slot k of a node's draft row leads to its k-th
child.  Context labels: every node gets an independent 64-bit label and
position = base position + depth; every sequence gets a 64-bit watermark key.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

_MASK64 = (1 << 64) - 1


def splitmix64_stream(seed: int, n: int) -> np.ndarray:
    """n 64-bit values of the SplitMix64 stream started at `seed`."""
    out = np.empty(n, np.uint64)
    s = seed & _MASK64
    for t in range(n):
        s = (s + 0x9E3779B97F4A7C15) & _MASK64
        z = s
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
        out[t] = z ^ (z >> 31)
    return out


@dataclass
class Tree:
    """Static draft-tree topology for `n_seq` identical sequences."""
    branching: tuple
    n_seq: int
    nodes_per_seq: int = 0
    draft_per_seq: int = 0
    seq_off: np.ndarray = field(default=None)          # [n_seq+1] int32
    node_depth: np.ndarray = field(default=None)       # [n_nodes] int32
    node_draft_row: np.ndarray = field(default=None)   # [n_nodes] int32, -1 for leaves
    draft_node: np.ndarray = field(default=None)       # [n_draft] int32
    row_k: np.ndarray = field(default=None)            # [n_draft] int32 list length per draft row
    child_node: np.ndarray = field(default=None)       # [n_draft, K] int32, -1 where no child

    @property
    def gamma(self) -> int:
        return len(self.branching)

    @property
    def n_nodes(self) -> int:
        return self.nodes_per_seq * self.n_seq

    @property
    def n_draft(self) -> int:
        return self.draft_per_seq * self.n_seq

    @property
    def K(self) -> int:
        return int(max(self.branching))


def make_tree(branching, n_seq: int) -> Tree:
    branching = tuple(int(b) for b in branching)
    K = max(branching)
    # one sequence, breadth first
    depth = [0]
    children = [[]]
    frontier = [0]
    for d, b in enumerate(branching):
        nxt = []
        for c in frontier:
            for _ in range(b):
                depth.append(d + 1)
                children.append([])
                children[c].append(len(depth) - 1)
                nxt.append(len(depth) - 1)
        frontier = nxt
    nps = len(depth)
    internal = [c for c in range(nps) if depth[c] < len(branching)]
    dps = len(internal)
    t = Tree(branching=branching, n_seq=n_seq, nodes_per_seq=nps, draft_per_seq=dps)
    t.seq_off = (np.arange(n_seq + 1, dtype=np.int64) * nps).astype(np.int32)
    t.node_depth = np.tile(np.asarray(depth, np.int32), n_seq)
    ndr = np.full(nps, -1, np.int64)
    for r, c in enumerate(internal):
        ndr[c] = r
    t.node_draft_row = np.concatenate([np.where(ndr >= 0, ndr + b * dps, -1) for b in range(n_seq)]).astype(np.int32)
    t.draft_node = np.concatenate([np.asarray(internal, np.int64) + b * nps for b in range(n_seq)]).astype(np.int32)
    t.row_k = np.tile(np.asarray([branching[depth[c]] for c in internal], np.int32), n_seq)
    cn = np.full((dps, K), -1, np.int64)
    for r, c in enumerate(internal):
        for k, ch in enumerate(children[c]):
            cn[r, k] = ch
    t.child_node = np.concatenate([np.where(cn >= 0, cn + b * nps, -1) for b in range(n_seq)]).astype(np.int32)
    return t


@dataclass
class Workload:
    name: str
    vocab: int
    dtype: torch.dtype
    tree: Tree
    temperature: float
    p_logits: torch.Tensor      # [n_nodes, V] target logits, one row per node
    q_logits: torch.Tensor      # [n_draft, V] draft logits, one row per internal node
    node_key: torch.Tensor      # [n_nodes] int64 (bit pattern of the u64 key)
    node_ctx: torch.Tensor      # [n_nodes] int64 (bit pattern of the u64 label)
    node_pos: torch.Tensor      # [n_nodes] int32 (u32 position)
    draft_key: torch.Tensor     # [n_draft] ids of the draft rows (= their nodes' ids)
    draft_ctx: torch.Tensor
    draft_pos: torch.Tensor
    recipe: str = ""

    @property
    def K(self) -> int:
        return self.tree.K

    def row_bytes(self) -> int:
        return self.vocab * torch.tensor([], dtype=self.dtype).element_size()


# --- logit families ---------------------------------------------------------

def _zipf(gen, rows, V, exponent, permute, device):
    rank = torch.arange(1, V + 1, device=device, dtype=torch.float32)
    base = -exponent * torch.log(rank)
    out = torch.empty(rows, V, device=device, dtype=torch.float32)
    chunk = max(1, (1 << 26) // V)
    for r0 in range(0, rows, chunk):
        r1 = min(rows, r0 + chunk)
        noise = torch.randn(r1 - r0, V, generator=gen, device=device)
        if permute:
            perm = torch.argsort(torch.rand(r1 - r0, V, generator=gen, device=device), dim=1)
            out[r0:r1] = base[perm] + noise
        else:
            out[r0:r1] = base[None, :] + noise
    return out


def _entropy_of_scale(V, sigma, gen, device):
    z = torch.randn(V, generator=gen, device=device, dtype=torch.float64) * sigma
    p = torch.softmax(z, 0)
    return float(-(p * torch.log(p.clamp_min(1e-300))).sum())


def flat_sigma(V: int, target_entropy: float, device="cpu", seed: int = 12345) -> float:
    """Gaussian logit scale whose softmax entropy is ~target_entropy (bisection)."""
    lo, hi = 0.0, 20.0
    for _ in range(60):
        mid = 0.5 * (lo + hi)
        g = torch.Generator(device=device)
        g.manual_seed(seed)
        if _entropy_of_scale(V, mid, g, device) > target_entropy:
            lo = mid
        else:
            hi = mid
    return 0.5 * (lo + hi)


def _peaked_flat(gen, rows, V, sigma_flat, device):
    out = torch.randn(rows, V, generator=gen, device=device, dtype=torch.float32)
    peaked = torch.arange(rows, device=device) % 2 == 0
    out[~peaked] *= sigma_flat
    pk = out[peaked]
    if pk.numel():
        top = torch.argmax(pk, dim=1)
        rest = pk.clone()
        rest.scatter_(1, top[:, None], float("-inf"))
        lse_rest = torch.logsumexp(rest, dim=1)
        pk.scatter_(1, top[:, None], (math.log(9.0) + lse_rest)[:, None])
        out[peaked] = pk
    return out


# --- configurations ---------------------------------------------------------

CONFIGS = {
    # name: (seed, n_seq, V, branching, dtype, family, draft noise sd)
    "tiny": (0, 64, 1000, (2,), torch.float32, "gauss3", 1.0),
    "chain4x4": (1, 8, 32000, (4, 1, 1, 1), torch.bfloat16, "zipf1.1", 0.7),
    "zipf_k8": (2, 64, 128256, (8, 1, 1, 1, 1), torch.bfloat16, "zipf1.0perm", 1.0),
    "branch16": (3, 256, 152064, (16, 3, 2, 1), torch.float32, "peakedflat", 1.5),
}


def kchain(K: int, gamma: int = 5):
    return (K,) + (1,) * (gamma - 1)


def make_workload(name: str, device="cpu", n_seq: int | None = None, vocab: int | None = None,
                  branching=None, dtype=None, seed: int | None = None, K_sweep: int | None = None) -> Workload:
    """Build a named workload.  `n_seq`, `vocab`, `branching`, `dtype`, `seed`
    override the named configuration (smaller cases for parity tests).
    ``name == "ksweep"`` is the K sweep (Zipf 1.0, V=128256, gamma=5, K=K_sweep)."""
    if name == "ksweep":
        base = (4, 64, 128256, kchain(K_sweep or 1), torch.bfloat16, "zipf1.0perm", 1.0)
    else:
        base = CONFIGS[name]
    s0, ns0, V0, br0, dt0, fam, noise = base
    seed = s0 if seed is None else seed
    n_seq = ns0 if n_seq is None else n_seq
    V = V0 if vocab is None else vocab
    br = br0 if branching is None else tuple(branching)
    dt = dt0 if dtype is None else dtype
    tree = make_tree(br, n_seq)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    R = tree.n_nodes
    if fam == "gauss3":
        p = torch.randn(R, V, generator=gen, device=device) * 3.0
        recipe = "target logits iid N(0,3^2)"
    elif fam == "zipf1.1":
        p = _zipf(gen, R, V, 1.1, False, device)
        recipe = "target logits -1.1 ln(rank) + N(0,1), rank = token index + 1"
    elif fam == "zipf1.0perm":
        p = _zipf(gen, R, V, 1.0, True, device)
        recipe = "target logits -ln(rank) + N(0,1), ranks randomly permuted per row"
    elif fam == "peakedflat":
        sig = flat_sigma(V, 6.0, device="cpu")
        p = _peaked_flat(gen, R, V, sig, device)
        recipe = f"alternating peaked rows (top-1 prob 0.9 over N(0,1)) and flat rows N(0,{sig:.4f}^2) (entropy ~6 nats)"
    else:
        raise ValueError(fam)
    dn = torch.as_tensor(tree.draft_node, device=device, dtype=torch.long)
    q = p[dn] + torch.randn(tree.n_draft, V, generator=gen, device=device) * noise
    recipe += f"; draft logits = target logits of the same node + N(0,{noise}^2)"
    p = p.to(dt)
    q = q.to(dt)
    # ids: keys per sequence, labels per node, positions = base + depth
    ids = splitmix64_stream(seed * 0x100000001 + 77, n_seq + tree.n_nodes + n_seq)
    keys = ids[:n_seq]
    ctx = ids[n_seq:n_seq + tree.n_nodes]
    base_pos = (ids[n_seq + tree.n_nodes:] % np.uint64(4096)).astype(np.int64) + 16
    seq_of_node = np.repeat(np.arange(n_seq), tree.nodes_per_seq)
    node_key = keys[seq_of_node]
    node_pos = (base_pos[seq_of_node] + tree.node_depth).astype(np.uint32)
    t_key = torch.from_numpy(node_key.view(np.int64).copy()).to(device)
    t_ctx = torch.from_numpy(ctx.view(np.int64).copy()).to(device)
    t_pos = torch.from_numpy(node_pos.view(np.int32).copy()).to(device)
    return Workload(name=name, vocab=V, dtype=dt, tree=tree, temperature=1.0, p_logits=p, q_logits=q,
                    node_key=t_key, node_ctx=t_ctx, node_pos=t_pos,
                    draft_key=t_key[dn], draft_ctx=t_ctx[dn], draft_pos=t_pos[dn], recipe=recipe)


def u64(t: torch.Tensor) -> np.ndarray:
    """View an int64 id tensor as numpy uint64."""
    return t.detach().cpu().numpy().view(np.uint64)


def u32(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy().view(np.uint32)


def _mix64_np(z: np.ndarray) -> np.ndarray:
    z = z.astype(np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


def label_logits(labels, V: int, seed: int = 0, zipf: float = 1.0, noise: float = 1.5) -> np.ndarray:
    """A synthetic "model": logits of a context as a fixed function of its 64-bit label,
    -zipf * ln(rank) + noise * N(0,1), the ranks and the noise drawn from SplitMix64 of
    (label, token, seed).  Deterministic, so both sides of a test see the same logits for
    the same context, wherever it sits in a tree."""
    lab = np.asarray(labels, dtype=np.uint64).reshape(-1, 1)
    col = np.arange(V, dtype=np.uint64).reshape(1, -1)
    with np.errstate(over="ignore"):
        base = lab ^ (col * np.uint64(0x9E3779B97F4A7C15)) ^ np.uint64(seed & _MASK64)
    h1 = _mix64_np(base)
    h2 = _mix64_np(h1 ^ np.uint64(0xD1B54A32D192ED03))
    u1 = ((h1 >> np.uint64(11)).astype(np.float64) + 0.5) / 2.0 ** 53
    u2 = ((h2 >> np.uint64(11)).astype(np.float64) + 0.5) / 2.0 ** 53
    g = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * np.pi * u2)
    # a per-context permutation of ranks: order of an independent hash
    perm = np.argsort(_mix64_np(h2 ^ np.uint64(0x5851F42D4C957F2D)), axis=1, kind="stable")
    rank = np.empty_like(perm)
    np.put_along_axis(rank, perm, np.arange(1, V + 1).reshape(1, -1).repeat(lab.shape[0], 0), axis=1)
    return (-zipf * np.log(rank) + noise * g).astype(np.float32)


# --- LM-head operands (the fused race takes hidden states and weights, not logits) ----------

@dataclass
class LmHeadWorkload:
    tree: Tree
    vocab: int
    hp: torch.Tensor        # [n_nodes, d_target] bf16 hidden states of the target model, one per node
    wp: torch.Tensor        # [V, d_target] bf16 target LM-head matrix
    hq: torch.Tensor        # [n_draft, d_draft] bf16 hidden states of the draft model, one per draft row
    wq: torch.Tensor        # [V, d_draft] bf16 draft LM-head matrix
    node_key: torch.Tensor
    node_ctx: torch.Tensor
    node_pos: torch.Tensor
    draft_key: torch.Tensor
    draft_ctx: torch.Tensor
    draft_pos: torch.Tensor
    temperature: float = 1.0
    recipe: str = ""


def lmhead_workload(n_seq: int = 64, branching=(8, 1, 1, 1, 1), vocab: int = 128256, d_target: int = 4096,
                    d_draft: int = 2048, seed: int = 5, device="cpu") -> LmHeadWorkload:
    """Operands whose products are Zipf-shaped logits, like the zipf_k8 workload but produced by
    an LM head: column 0 of every hidden state is 1 and column 0 of weight row i is -ln(rank_i)
    (one random permutation of the ranks: the model's token frequencies); the other columns are
    N(0, 1) (hidden) and N(0, 1/(d-1)) (weights), so target logits are -ln(rank) + N(0, 1).  The
    draft model reads the first d_draft columns of the same hidden states with its weight columns
    1..d_draft-1 equal to the target's, scaled to unit variance: draft logits = -ln(rank) + a noise
    correlated ~sqrt((d_draft-1)/(d_target-1)) with the target's."""
    assert 2 <= d_draft <= d_target
    tree = make_tree(tuple(branching), n_seq)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    V = vocab
    rank = torch.argsort(torch.rand(V, generator=gen, device=device)).float() + 1.0
    wp = torch.randn(V, d_target, generator=gen, device=device) / math.sqrt(d_target - 1)
    wp[:, 0] = -torch.log(rank)
    wq = wp[:, :d_draft] * math.sqrt((d_target - 1) / (d_draft - 1))
    wq[:, 0] = wp[:, 0]
    hp = torch.randn(tree.n_nodes, d_target, generator=gen, device=device)
    hp[:, 0] = 1.0
    dn = torch.as_tensor(tree.draft_node, device=device, dtype=torch.long)
    hq = hp[dn, :d_draft]
    ids = splitmix64_stream(seed * 0x100000001 + 99, n_seq + tree.n_nodes + n_seq)
    keys = ids[:n_seq]
    ctx = ids[n_seq:n_seq + tree.n_nodes]
    base_pos = (ids[n_seq + tree.n_nodes:] % np.uint64(4096)).astype(np.int64) + 16
    seq_of_node = np.repeat(np.arange(n_seq), tree.nodes_per_seq)
    t_key = torch.from_numpy(keys[seq_of_node].view(np.int64).copy()).to(device)
    t_ctx = torch.from_numpy(ctx.view(np.int64).copy()).to(device)
    t_pos = torch.from_numpy((base_pos[seq_of_node] + tree.node_depth).astype(np.uint32).view(np.int32).copy()).to(device)
    return LmHeadWorkload(tree=tree, vocab=V, hp=hp.to(torch.bfloat16), wp=wp.to(torch.bfloat16),
                          hq=hq.to(torch.bfloat16), wq=wq.to(torch.bfloat16), node_key=t_key, node_ctx=t_ctx,
                          node_pos=t_pos, draft_key=t_key[dn], draft_ctx=t_ctx[dn], draft_pos=t_pos[dn],
                          recipe=f"LM head: V={V}, d={d_target} (target) / {d_draft} (draft), hidden column 0 = 1, "
                                 f"weight column 0 = -ln(rank), other entries Gaussian")
