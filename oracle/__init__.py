"""CPU oracle for the keyed Poisson-race multi-draft speculative sampler.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (``paper_2609_21858_gb300``) never imports it and
shares no code with it.

The arithmetic lives in ``pps_oracle.c`` (plain C, fp64); this module only
compiles it with gcc and marshals numpy arrays through ctypes.  The closed
forms used to pin it (acceptance probabilities, the watermark pivot law) are
in ``oracle.closed_forms``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pps_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

DISTINCT = 0
IID = 1


def build(force: bool = False) -> str:
    """Compile the oracle shared library with gcc (-O2, OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _P(t):
    return ctypes.POINTER(t)


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            u32p, u64p, i32p, i64p, f32p, f64p = (_P(ctypes.c_uint32), _P(ctypes.c_uint64), _P(ctypes.c_int32),
                                                  _P(ctypes.c_int64), _P(ctypes.c_float), _P(ctypes.c_double))
            i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
            L.orc_philox4x32_10.argtypes = [u32p, u32p, u32p]
            L.orc_philox4x32_10.restype = None
            L.orc_philox4x32.argtypes = [u32p, u32p, i32, u32p]
            L.orc_philox4x32.restype = None
            L.orc_set_philox_rounds.argtypes = [i32]
            L.orc_set_philox_rounds.restype = i32
            L.orc_word.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32, i64, i32]
            L.orc_word.restype = ctypes.c_uint32
            L.orc_uniform.argtypes = [ctypes.c_uint32]
            L.orc_uniform.restype = f64
            L.orc_exp1.argtypes = [ctypes.c_uint32]
            L.orc_exp1.restype = f64
            L.orc_score_word.argtypes = [ctypes.c_uint32]
            L.orc_score_word.restype = f64
            L.orc_race_key.argtypes = [ctypes.c_uint32, f64, f64]
            L.orc_race_key.restype = f64
            L.orc_target_rows.argtypes = [f32p, i64, i64, i64, f64, u64p, u64p, u32p, i32p, u32p, f64p, f64p]
            L.orc_target_rows.restype = None
            L.orc_draft_rows.argtypes = [f32p, i64, i64, i64, f64, u64p, u64p, u32p, i32, i32p, i32,
                                         i32p, f64p, i32p, i32p, i32p, f64p]
            L.orc_draft_rows.restype = None
            L.orc_walk.argtypes = [i32, i32, i32p, i32p, i32p, i32p, i32, i32p, i32p, u32p,
                                   i32p, i32p, i32p, f64p, f64p]
            L.orc_walk.restype = None
            L.orc_wm_score.argtypes = [i64, i32p, u64p, u64p, u32p, f64p, i32, i64p, f64p]
            L.orc_wm_score.restype = None
            L.orc_words.argtypes = [i64, i64, u64p, u64p, u32p, i32, u32p]
            L.orc_words.restype = None
            L.orc_score_kind.argtypes = [ctypes.c_uint32, i32, f64]
            L.orc_score_kind.restype = f64
            L.orc_gamma_tail_logp.argtypes = [i64, f64]
            L.orc_gamma_tail_logp.restype = f64
            L.orc_chernoff_u_logp.argtypes = [i64, f64]
            L.orc_chernoff_u_logp.restype = f64
            L.orc_wm_detect.argtypes = [i64, i32p, u64p, u64p, u32p, i32, f64, i32, i64p, f64p, f64p, f64p]
            L.orc_wm_detect.restype = None
            L.orc_mix64.argtypes = [ctypes.c_uint64]
            L.orc_mix64.restype = ctypes.c_uint64
            L.orc_child_label.argtypes = [ctypes.c_uint64, i32]
            L.orc_child_label.restype = ctypes.c_uint64
            L.orc_tree_expand.argtypes = [i32, i32, i32, i32, i32p, i32p, i32p, u64p, u64p, u32p, i32p,
                                          u64p, u64p, u32p, i32p, i32p, u64p, u64p, u32p]
            L.orc_tree_expand.restype = None
            L.orc_hetero_expand.argtypes = [i32, i32, i32, i32, i32p, u64p, u64p, u32p, i32p, u64p, u64p, u32p,
                                            i32p, i32p, i32p, i32p, u64p, u64p, u32p]
            L.orc_hetero_expand.restype = None
            L.orc_block_j.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32, i64, i32]
            L.orc_block_j.restype = i32
            L.orc_block_e.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32, i64, i32, i32]
            L.orc_block_e.restype = f64
            L.orc_block_draft_rows.argtypes = [f32p, i64, i64, i64, f64, u64p, u64p, u32p, i32p, i32, i32p, f64p,
                                               f64p]
            L.orc_block_draft_rows.restype = None
            L.orc_hetero_rows.argtypes = [f32p, f32p, i64, i32, i64, f64, u64p, u64p, u32p, i32p, i32p, i32p,
                                          u32p, i32p, f64p, f64p]
            L.orc_hetero_rows.restype = None
            L.orc_truncate_rows.argtypes = [f32p, i64, i64, i64, f64, i32, f64, f32p, f64p]
            L.orc_truncate_rows.restype = None
            L.orc_lmhead_logits.argtypes = [f32p, f32p, i64, i64, i64, f64p]
            L.orc_lmhead_logits.restype = None
            L.orc_set_threads.argtypes = [ctypes.c_int]
            L.orc_set_threads.restype = ctypes.c_int
            _lib = L
    return _lib


def _ptr(a, t):
    return a.ctypes.data_as(_P(t)) if a is not None else None


def _c(a, dtype):
    return np.ascontiguousarray(np.asarray(a, dtype=dtype))


def set_threads(n: int = 0) -> int:
    """Set (n > 0) and return the number of OpenMP threads the oracle uses."""
    return int(lib().orc_set_threads(int(n)))


def philox4x32_10(ctr, key):
    c = _c(ctr, np.uint32)
    k = _c(key, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().orc_philox4x32_10(_ptr(c, ctypes.c_uint32), _ptr(k, ctypes.c_uint32), _ptr(out, ctypes.c_uint32))
    return out


def philox4x32(ctr, key, rounds: int):
    c = _c(ctr, np.uint32)
    k = _c(key, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().orc_philox4x32(_ptr(c, ctypes.c_uint32), _ptr(k, ctypes.c_uint32), int(rounds), _ptr(out, ctypes.c_uint32))
    return out


def set_philox_rounds(rounds: int = 0) -> int:
    """Set (rounds > 0) and return the Philox round count of the keyed source (10 by default;
    7 for the library built with PPS_PHILOX_ROUNDS=7).  Process-wide."""
    return int(lib().orc_set_philox_rounds(int(rounds)))


def word(key: int, ctx: int, pos: int, token: int, arrival: int = 1) -> int:
    return int(lib().orc_word(key, ctx, pos, token, arrival))


def uniform(w: int) -> float:
    return float(lib().orc_uniform(w))


def exp1(w: int) -> float:
    return float(lib().orc_exp1(w))


def score_word(w: int) -> float:
    return float(lib().orc_score_word(w))


def race_key(w: int, logit: float, T: float = 1.0) -> float:
    return float(lib().orc_race_key(w, logit, T))


def words(key, ctx, pos, vocab: int, arrival: int = 1):
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    n = key.shape[0]
    out = np.zeros((n, vocab), np.uint32)
    lib().orc_words(n, vocab, _ptr(key, ctypes.c_uint64), _ptr(ctx, ctypes.c_uint64), _ptr(pos, ctypes.c_uint32),
                    arrival, _ptr(out, ctypes.c_uint32))
    return out


def target_rows(logits, key, ctx, pos, T: float = 1.0):
    """Per row: (winner, word, key, margin) of the target race argmin_i E_i/P(i)."""
    l = _c(logits, np.float32)
    n, V = l.shape
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    win = np.zeros(n, np.int32)
    wd = np.zeros(n, np.uint32)
    ky = np.zeros(n, np.float64)
    mg = np.zeros(n, np.float64)
    lib().orc_target_rows(_ptr(l, ctypes.c_float), n, V, V, float(T), _ptr(key, ctypes.c_uint64),
                          _ptr(ctx, ctypes.c_uint64), _ptr(pos, ctypes.c_uint32), _ptr(win, ctypes.c_int32),
                          _ptr(wd, ctypes.c_uint32), _ptr(ky, ctypes.c_double), _ptr(mg, ctypes.c_double))
    return win, wd, ky, mg


def draft_rows(logits, key, ctx, pos, K: int, row_k=None, mode: int = DISTINCT, T: float = 1.0):
    """Per row: dict(tok, key, mult, ndist, labels, min_gap) of the draft list."""
    l = _c(logits, np.float32)
    n, V = l.shape
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    rk = _c(row_k, np.int32) if row_k is not None else None
    tok = np.zeros((n, K), np.int32)
    ky = np.zeros((n, K), np.float64)
    mult = np.zeros((n, K), np.int32)
    nd = np.zeros(n, np.int32)
    lab = np.zeros((n, K), np.int32)
    gap = np.zeros(n, np.float64)
    lib().orc_draft_rows(_ptr(l, ctypes.c_float), n, V, V, float(T), _ptr(key, ctypes.c_uint64),
                         _ptr(ctx, ctypes.c_uint64), _ptr(pos, ctypes.c_uint32), int(K), _ptr(rk, ctypes.c_int32),
                         int(mode), _ptr(tok, ctypes.c_int32), _ptr(ky, ctypes.c_double), _ptr(mult, ctypes.c_int32),
                         _ptr(nd, ctypes.c_int32), _ptr(lab, ctypes.c_int32), _ptr(gap, ctypes.c_double))
    return dict(tok=tok, key=ky, mult=mult, ndist=nd, labels=lab, min_gap=gap)


def walk(gamma: int, seq_off, node_draft_row, draft_tok, draft_ndist, child_node, winner, word_):
    seq_off = _c(seq_off, np.int32)
    ndr = _c(node_draft_row, np.int32)
    dt = _c(draft_tok, np.int32)
    K = dt.shape[1] if dt.ndim == 2 else 1
    dn = _c(draft_ndist, np.int32)
    cn = _c(child_node, np.int32)
    win = _c(winner, np.int32)
    wd = _c(word_, np.uint32)
    n_seq = seq_off.shape[0] - 1
    W = gamma + 1
    acc = np.zeros(n_seq, np.int32)
    ne = np.zeros(n_seq, np.int32)
    em = np.zeros((n_seq, W), np.int32)
    sc = np.zeros((n_seq, W), np.float64)
    ss = np.zeros(n_seq, np.float64)
    lib().orc_walk(n_seq, gamma, _ptr(seq_off, ctypes.c_int32), _ptr(ndr, ctypes.c_int32), _ptr(dt, ctypes.c_int32),
                   _ptr(dn, ctypes.c_int32), K, _ptr(cn, ctypes.c_int32), _ptr(win, ctypes.c_int32),
                   _ptr(wd, ctypes.c_uint32), _ptr(acc, ctypes.c_int32), _ptr(ne, ctypes.c_int32),
                   _ptr(em, ctypes.c_int32), _ptr(sc, ctypes.c_double), _ptr(ss, ctypes.c_double))
    return dict(accept_len=acc, n_emitted=ne, emitted=em, score=sc, score_sum=ss)


def wm_score(tokens, key, ctx, pos, seg_off=None):
    t = _c(tokens, np.int32)
    n = t.shape[0]
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    sc = np.zeros(n, np.float64)
    so = _c(seg_off, np.int64) if seg_off is not None else None
    n_seg = (so.shape[0] - 1) if so is not None else 1
    sums = np.zeros(n_seg, np.float64)
    lib().orc_wm_score(n, _ptr(t, ctypes.c_int32), _ptr(key, ctypes.c_uint64), _ptr(ctx, ctypes.c_uint64),
                       _ptr(pos, ctypes.c_uint32), _ptr(sc, ctypes.c_double), n_seg, _ptr(so, ctypes.c_int64),
                       _ptr(sums, ctypes.c_double))
    return sc, sums


def truncate_rows(logits, top_k: int = 0, top_p: float = 1.0, T: float = 1.0):
    """Top-k then top-p truncation as masking: (logits with removed tokens set to -inf, margin)."""
    l = _c(logits, np.float32)
    n, V = l.shape
    out = np.zeros((n, V), np.float32)
    mg = np.zeros(n, np.float64)
    lib().orc_truncate_rows(_ptr(l, ctypes.c_float), n, V, V, float(T), int(top_k), float(top_p),
                            _ptr(out, ctypes.c_float), _ptr(mg, ctypes.c_double))
    return out, mg


AARONSON, U_SCORE, LI, PL = 0, 1, 2, 3


def score_kind(w: int, kind: int, param: float = 0.0) -> float:
    return float(lib().orc_score_kind(w, int(kind), float(param)))


def gamma_tail_logp(M: int, S: float) -> float:
    """ln P(Gamma(M,1) >= S)"""
    return float(lib().orc_gamma_tail_logp(int(M), float(S)))


def chernoff_u_logp(M: int, S: float) -> float:
    """Chernoff bound on ln P(sum of M iid U(0,1) >= S)"""
    return float(lib().orc_chernoff_u_logp(int(M), float(S)))


def wm_detect(tokens, key, ctx, pos, seg_off, kind: int = AARONSON, param: float = 0.0):
    """Per token scores, per segment sums and log p-values of the detector pass."""
    t = _c(tokens, np.int32)
    n = t.shape[0]
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    so = _c(seg_off, np.int64)
    n_seg = so.shape[0] - 1
    sc = np.zeros(n, np.float64)
    sums = np.zeros(n_seg, np.float64)
    logp = np.zeros(n_seg, np.float64)
    lib().orc_wm_detect(n, _ptr(t, ctypes.c_int32), _ptr(key, ctypes.c_uint64), _ptr(ctx, ctypes.c_uint64),
                        _ptr(pos, ctypes.c_uint32), int(kind), float(param), n_seg, _ptr(so, ctypes.c_int64),
                        _ptr(sc, ctypes.c_double), _ptr(sums, ctypes.c_double), _ptr(logp, ctypes.c_double))
    return sc, sums, logp


def mix64(z: int) -> int:
    return int(lib().orc_mix64(z))


def child_label(parent: int, token: int) -> int:
    return int(lib().orc_child_label(parent, int(token)))


def tree_expand(n_seq, K, gamma, depth, d, key, ctx, pos, row_k, tree):
    """One depth of the dynamic IID tree; `d` = draft_rows(IID) output of this depth's rows,
    `tree` = dict(child_node [draft rows, K] (depth-major rows), node_key/ctx/pos [n_seq*N1]),
    updated in place.
    Returns (next_key, next_ctx, next_pos, next_k) of depth+1's rows."""
    n = n_seq * K
    nk, nc = np.zeros(n, np.uint64), np.zeros(n, np.uint64)
    npos, nkk = np.zeros(n, np.uint32), np.zeros(n, np.int32)
    tok, mult, nd = _c(d["tok"], np.int32), _c(d["mult"], np.int32), _c(d["ndist"], np.int32)
    key, ctx, pos, rk = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32), _c(row_k, np.int32)
    lib().orc_tree_expand(n_seq, K, gamma, depth, _ptr(tok, ctypes.c_int32), _ptr(mult, ctypes.c_int32),
                          _ptr(nd, ctypes.c_int32), _ptr(key, ctypes.c_uint64), _ptr(ctx, ctypes.c_uint64),
                          _ptr(pos, ctypes.c_uint32), _ptr(rk, ctypes.c_int32), _ptr(nk, ctypes.c_uint64),
                          _ptr(nc, ctypes.c_uint64), _ptr(npos, ctypes.c_uint32), _ptr(nkk, ctypes.c_int32),
                          _ptr(tree["child_node"], ctypes.c_int32), _ptr(tree["node_key"], ctypes.c_uint64),
                          _ptr(tree["node_ctx"], ctypes.c_uint64), _ptr(tree["node_pos"], ctypes.c_uint32))
    return nk, nc, npos, nkk


def block_j(key: int, ctx: int, pos: int, i: int, B: int) -> int:
    """Block J_i of token i's smallest augmented arrival."""
    return int(lib().orc_block_j(key, ctx, pos, int(i), int(B)))


def block_e(key: int, ctx: int, pos: int, i: int, b: int, B: int) -> float:
    """First arrival E_(i,b) of augmented point (i, b)."""
    return float(lib().orc_block_e(key, ctx, pos, int(i), int(b), int(B)))


def block_draft_rows(q_logits, key, ctx, pos, block, B: int, T: float = 1.0):
    """Proposal races per row: (x, key, margin)."""
    q = _c(q_logits, np.float32)
    n, V = q.shape
    key, ctx, pos, block = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32), _c(block, np.int32)
    x = np.zeros(n, np.int32)
    k, m = np.zeros(n, np.float64), np.zeros(n, np.float64)
    lib().orc_block_draft_rows(_ptr(q, ctypes.c_float), n, V, V, float(T), _ptr(key, ctypes.c_uint64),
                               _ptr(ctx, ctypes.c_uint64), _ptr(pos, ctypes.c_uint32), _ptr(block, ctypes.c_int32),
                               int(B), _ptr(x, ctypes.c_int32), _ptr(k, ctypes.c_double), _ptr(m, ctypes.c_double))
    return x, k, m


def hetero_rows(p_logits, q_logits, key, ctx, pos, B: int, T: float = 1.0):
    """One step with B non-identical proposals per context:
    dict(x [n, B], y, j, word, accept, margin_y, margin_x [n, B])."""
    p = _c(p_logits, np.float32)
    n, V = p.shape
    q = _c(q_logits, np.float32).reshape(n * B, V)
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    x = np.zeros(n * B, np.int32)
    y, j, acc = np.zeros(n, np.int32), np.zeros(n, np.int32), np.zeros(n, np.int32)
    word = np.zeros(n, np.uint32)
    my, mx = np.zeros(n, np.float64), np.zeros(n * B, np.float64)
    lib().orc_hetero_rows(_ptr(p, ctypes.c_float), _ptr(q, ctypes.c_float), n, int(B), V, float(T),
                          _ptr(key, ctypes.c_uint64), _ptr(ctx, ctypes.c_uint64), _ptr(pos, ctypes.c_uint32),
                          _ptr(x, ctypes.c_int32), _ptr(y, ctypes.c_int32), _ptr(j, ctypes.c_int32),
                          _ptr(word, ctypes.c_uint32), _ptr(acc, ctypes.c_int32), _ptr(my, ctypes.c_double),
                          _ptr(mx, ctypes.c_double))
    return dict(x=x.reshape(n, B), y=y, j=j, word=word, accept=acc, margin_y=my, margin_x=mx.reshape(n, B))


def hetero_expand(n_seq, B, gamma, depth, tok, key, ctx, pos, owner, tree):
    """One depth of the tree of B proposals; `tok` = the proposals' draws at this depth's
    rows, `tree` = dict(list_tok, child_node [n_lists, B], list_nd [n_lists],
    node_key/ctx/pos [n_seq*N1]), updated in place.
    Returns (next_key, next_ctx, next_pos, next_owner) of depth+1's rows."""
    n = n_seq * B
    nk, nc = np.zeros(n, np.uint64), np.zeros(n, np.uint64)
    npos, no = np.zeros(n, np.uint32), np.zeros(n, np.int32)
    tok, owner = _c(tok, np.int32), _c(owner, np.int32)
    key, ctx, pos = _c(key, np.uint64), _c(ctx, np.uint64), _c(pos, np.uint32)
    lib().orc_hetero_expand(n_seq, int(B), int(gamma), int(depth), _ptr(tok, ctypes.c_int32),
                            _ptr(key, ctypes.c_uint64), _ptr(ctx, ctypes.c_uint64), _ptr(pos, ctypes.c_uint32),
                            _ptr(owner, ctypes.c_int32), _ptr(nk, ctypes.c_uint64), _ptr(nc, ctypes.c_uint64),
                            _ptr(npos, ctypes.c_uint32), _ptr(no, ctypes.c_int32),
                            _ptr(tree["list_tok"], ctypes.c_int32), _ptr(tree["list_nd"], ctypes.c_int32),
                            _ptr(tree["child_node"], ctypes.c_int32), _ptr(tree["node_key"], ctypes.c_uint64),
                            _ptr(tree["node_ctx"], ctypes.c_uint64), _ptr(tree["node_pos"], ctypes.c_uint32))
    return nk, nc, npos, no


def hetero_tree(n_seq, B, gamma):
    """Empty oracle tree arrays of the multi-proposal layout."""
    N1 = 1 + B * gamma
    nl = n_seq * (1 + B * (gamma - 1))
    return dict(list_tok=np.full((nl, B), -1, np.int32), child_node=np.full((nl, B), -1, np.int32),
                list_nd=np.zeros(nl, np.int32), node_key=np.zeros(n_seq * N1, np.uint64),
                node_ctx=np.zeros(n_seq * N1, np.uint64), node_pos=np.zeros(n_seq * N1, np.uint32))


def lmhead_logits(hidden, weight):
    """logits = hidden . weight^T in fp64 (hidden [n, d], weight [V, d], fp32 images of bf16)."""
    h = _c(hidden, np.float32)
    w = _c(weight, np.float32)
    n, d = h.shape
    V = w.shape[0]
    assert w.shape[1] == d
    out = np.zeros((n, V), np.float64)
    lib().orc_lmhead_logits(_ptr(h, ctypes.c_float), _ptr(w, ctypes.c_float), n, V, d, _ptr(out, ctypes.c_double))
    return out
