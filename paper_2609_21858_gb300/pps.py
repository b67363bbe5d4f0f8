"""ctypes binding of libpps (include/pps.h): same entry-point names, argument
marshalling only.  Torch supplies device memory and the current stream; every
step of the computation runs in the library's CUDA kernels.  There is no CPU
fallback: a missing or unloadable libpps.so raises immediately.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))


def library_path(rounds: int = 10) -> str:
    """The build of libpps whose keyed source is Philox4x32 with `rounds` rounds: 10
    (libpps.so, the default) or 7 (libpps_r7.so)."""
    if rounds not in (7, 10):
        raise ValueError("libpps is built for Philox4x32-10 and Philox4x32-7 only")
    return os.path.join(_HERE, "_lib", "libpps.so" if rounds == 10 else "libpps_r7.so")


# PPS_PHILOX_ROUNDS=7 in the environment selects the Philox4x32-7 build at import
LIB_PATH = library_path(int(os.environ.get("PPS_PHILOX_ROUNDS", "10")))

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_WORKSPACE, ERR_CUDA, ERR_SIZE = 0, 1, 2, 3, 4, 5
NOALLOC_MAX_ROWS = 4096  # PPS_NOALLOC_MAX_ROWS of include/pps.h (tests/test_abi.py checks the two agree)
F32, BF16 = 0, 1
DISTINCT, IID = 0, 1
FLAG_GUARD, FLAG_LOGIT_RANGE, FLAG_TREE, FLAG_TIMEOUT = 1, 2, 4, 8
MAX_K = 32
MAX_TOP_K = 64
MAX_BLOCKS = 32
LMHEAD_MAX_K = 8

_lock = threading.Lock()
_lib = None


class RowIds(ctypes.Structure):
    _fields_ = [("key", ctypes.c_void_p), ("ctx_hash", ctypes.c_void_p), ("pos", ctypes.c_void_p)]


class PPSError(RuntimeError):
    def __init__(self, fn, code):
        super().__init__(f"{fn} failed: {code} ({status_string(code)})")
        self.code = code


def use_library(rounds: int = 10):
    """Switch the binding to the build for Philox4x32-`rounds` (the next call loads it).
    Device memory (workspaces, outputs) carries over; results follow the new keyed source."""
    global _lib, LIB_PATH
    with _lock:
        LIB_PATH = library_path(rounds)
        _lib = None


def philox_rounds() -> int:
    """Rounds of the keyed source of the loaded library (pps_philox_rounds)."""
    return int(lib().pps_philox_rounds())


def lib():
    """Load libpps.so (raises if it was not built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"libpps.so not found at {LIB_PATH}; build it with "
                                   "`python -c 'import __graft_entry__ as g; g.build()'`")
            L = ctypes.CDLL(LIB_PATH)
            vp, i64, i32, f32, u64, sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float,
                                          ctypes.c_uint64, ctypes.c_size_t)
            L.pps_version.restype = ctypes.c_char_p
            L.pps_philox_rounds.argtypes = []
            L.pps_philox_rounds.restype = ctypes.c_int
            L.pps_status_string.argtypes = [ctypes.c_int]
            L.pps_status_string.restype = ctypes.c_char_p
            L.pps_workspace_size.argtypes = [i64, i64, i32, i32]
            L.pps_workspace_size.restype = sz
            L.pps_workspace_clear.argtypes = [vp, sz, vp]
            L.pps_workspace_clear.restype = ctypes.c_int
            L.pps_draft_list.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, i32, vp, ctypes.c_int,
                                         vp, vp, vp, vp, vp, vp, vp, sz, vp]
            L.pps_draft_list.restype = ctypes.c_int
            L.pps_verify_tree.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, i32, i32, vp, vp, i64, vp,
                                          vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
            L.pps_verify_tree.restype = ctypes.c_int
            L.pps_draft_list_trunc.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, i32, f32, i32, vp,
                                               ctypes.c_int, vp, vp, vp, vp, vp, vp, vp, sz, vp]
            L.pps_draft_list_trunc.restype = ctypes.c_int
            L.pps_verify_tree_trunc.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, i32, f32, i32, i32, vp,
                                                vp, i64, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
            L.pps_verify_tree_trunc.restype = ctypes.c_int
            L.pps_draft_list_noalloc.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, i32, vp, ctypes.c_int,
                                                 vp, vp, vp, vp, vp, vp, vp]
            L.pps_draft_list_noalloc.restype = ctypes.c_int
            L.pps_wm_score.argtypes = [vp, RowIds, i64, i32, vp, vp, vp, vp]
            L.pps_tree_expand.argtypes = [i32, i32, i32, i32, vp, vp, vp, RowIds, vp, vp, vp, vp, vp, vp, vp, vp,
                                          vp, vp]
            L.pps_tree_expand.restype = ctypes.c_int
            L.pps_wm_detect.argtypes = [vp, RowIds, i64, i32, vp, ctypes.c_int, ctypes.c_double, vp, vp, vp, vp]
            L.pps_wm_detect.restype = ctypes.c_int
            L.pps_wm_score.restype = ctypes.c_int
            L.pps_draft_hetero.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, vp, i32, vp, vp, vp, vp,
                                           sz, vp]
            L.pps_draft_hetero.restype = ctypes.c_int
            L.pps_draft_hetero_trunc.argtypes = [vp, ctypes.c_int, i64, i64, i64, RowIds, f32, i32, f32, vp, i32, vp,
                                                 vp, vp, vp, sz, vp]
            L.pps_draft_hetero_trunc.restype = ctypes.c_int
            L.pps_hetero_expand.argtypes = [i32, i32, i32, i32, vp, RowIds, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                            vp, vp]
            L.pps_hetero_expand.restype = ctypes.c_int
            L.pps_hetero_block.argtypes = [vp, RowIds, i64, i32, vp, vp]
            L.pps_hetero_block.restype = ctypes.c_int
            L.pps_lmhead_workspace_size.argtypes = [i64, i32]
            L.pps_lmhead_workspace_size.restype = sz
            L.pps_lmhead_logits.argtypes = [vp, i64, vp, i64, i64, i64, i64, vp, i64, vp]
            L.pps_lmhead_logits.restype = ctypes.c_int
            L.pps_lmhead_draft_list.argtypes = [vp, i64, vp, i64, i64, i64, i64, RowIds, f32, i32, vp, ctypes.c_int,
                                                vp, vp, vp, vp, vp, vp, vp, sz, vp]
            L.pps_lmhead_draft_list.restype = ctypes.c_int
            L.pps_lmhead_verify_tree.argtypes = [vp, i64, vp, i64, i64, i64, i64, RowIds, f32, i32, i32, vp, vp, i64,
                                                 vp, vp, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]
            L.pps_lmhead_verify_tree.restype = ctypes.c_int
            L.pps_philox_words.argtypes = [RowIds, i64, i64, i32, vp, vp]
            L.pps_philox_words.restype = ctypes.c_int
            L.pps_selftest_philox_rate.argtypes = [u64, vp, i32, vp]
            L.pps_selftest_philox_rate.restype = ctypes.c_int
            L.pps_selftest_lg2_error.argtypes = [f32, f32, vp, vp]
            L.pps_selftest_lg2_error.restype = ctypes.c_int
            L.pps_selftest_key_error.argtypes = [u64, u64, vp, vp]
            L.pps_selftest_key_error.restype = ctypes.c_int
            _lib = L
    return _lib


def version() -> str:
    return lib().pps_version().decode()


def status_string(code: int) -> str:
    return lib().pps_status_string(int(code)).decode()


def _check(fn, code):
    if code != OK:
        raise PPSError(fn, code)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream, dev=None):
    """The stream's handle; with no stream, the current stream of `dev` (the tensors' device)."""
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    elif dev is not None and stream.device != dev:
        raise ValueError(f"stream is on {stream.device}, the tensors on {dev}")
    return ctypes.c_void_p(stream.cuda_stream)


def _need(name, t, dev, dtype, numel=0, contiguous=True):
    """Raise unless tensor `t` (skipped when None) is on `dev` with `dtype` and holds at least
    `numel` elements: the library writes and reads through plain pointers, so a short or
    misplaced buffer must be refused here, before anything is launched."""
    if t is None:
        return
    if not isinstance(t, torch.Tensor) or not t.is_cuda or t.device != dev:
        raise TypeError(f"{name} must be a CUDA tensor on {dev}")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if contiguous and not t.is_contiguous():
        raise TypeError(f"{name} must be contiguous")
    if t.numel() < numel:
        raise ValueError(f"{name} holds {t.numel()} elements; the call needs {numel}")


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"logits must be bfloat16 or float32, got {t.dtype}")


def _ids(key, ctx, pos, n=0, dev=None):
    """Row ids (bit patterns of the unsigned key, context label and position), n of each."""
    for name, t, dt in (("key", key, torch.int64), ("ctx", ctx, torch.int64), ("pos", pos, torch.int32)):
        if not t.is_cuda or t.dtype != dt or not t.is_contiguous():
            raise TypeError(f"{name} must be a contiguous CUDA {dt} tensor (bit pattern of the unsigned id)")
        _need(name, t, dev if dev is not None else t.device, dt, n)
    return RowIds(key.data_ptr(), ctx.data_ptr(), pos.data_ptr())


def _need_out(out: dict, spec, dev):
    for name, dt, numel in spec:
        _need(name, out.get(name), dev, dt, numel)


def _rows(logits):
    if not logits.is_cuda or logits.dim() != 2 or logits.stride(1) != 1:
        raise TypeError("logits must be a 2-D CUDA tensor with unit stride along the vocabulary")
    return logits.shape[0], logits.shape[1], logits.stride(0)


def workspace_size(n_rows: int, vocab: int = 0, K: int = 1, n_seq: int = 0) -> int:
    return int(lib().pps_workspace_size(n_rows, vocab, K, n_seq))


def workspace(n_rows: int, n_seq: int = 0, device=None) -> torch.Tensor:
    """A zeroed workspace (reusable across calls of the same or smaller size)."""
    nb = workspace_size(n_rows, 0, 1, n_seq)
    return torch.zeros(nb, dtype=torch.uint8, device=device or "cuda")


def workspace_clear(ws: torch.Tensor, stream=None):
    _need("ws", ws, ws.device, torch.uint8)
    with torch.cuda.device(ws.device):
        _check("pps_workspace_clear", lib().pps_workspace_clear(_ptr(ws), ws.numel(), _stream(stream, ws.device)))


def _need_draft(out, n, K, row_k, status, dev):
    _need_out(out, [("tok", torch.int32, n * K), ("key", torch.float32, n * K), ("mult", torch.int32, n * K),
                    ("ndist", torch.int32, n), ("samples", torch.int32, n * K)], dev)
    for name in ("tok", "mult", "ndist"):
        if out.get(name) is None:
            raise TypeError(f"out[{name!r}] is required")
    _need("row_k", row_k, dev, torch.int32, n)
    _need("status", status, dev, torch.int32, 1)


def draft_list(q_logits, key, ctx, pos, K: int, row_k=None, mode: int = DISTINCT, temperature: float = 1.0,
               ws=None, status=None, out=None, keys: bool = True, samples: bool = True, stream=None,
               top_k: int = 0, top_p: float = 1.0):
    """pps_draft_list (pps_draft_list_trunc when top_k > 0).  Returns dict(tok, key, mult, ndist, samples)."""
    n, V, stride = _rows(q_logits)
    dev = q_logits.device
    if out is None:
        out = dict(tok=torch.empty(n, K, dtype=torch.int32, device=dev),
                   key=torch.empty(n, K, dtype=torch.float32, device=dev) if keys else None,
                   mult=torch.empty(n, K, dtype=torch.int32, device=dev),
                   ndist=torch.empty(n, dtype=torch.int32, device=dev),
                   samples=torch.empty(n, K, dtype=torch.int32, device=dev) if samples else None)
    if ws is None:
        ws = workspace(n, 0, dev)
    _need_draft(out, n, K, row_k, status, dev)
    _need("ws", ws, dev, torch.uint8)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        if top_k > 0:
            code = lib().pps_draft_list_trunc(_ptr(q_logits), _dtype_code(q_logits), n, V, stride, ids,
                                              float(temperature), int(top_k), float(top_p), int(K), _ptr(row_k),
                                              int(mode), _ptr(out["tok"]), _ptr(out.get("key")), _ptr(out["mult"]),
                                              _ptr(out["ndist"]), _ptr(out.get("samples")), _ptr(status), _ptr(ws),
                                              ws.numel(), _stream(stream, dev))
            _check("pps_draft_list_trunc", code)
            return out
        code = lib().pps_draft_list(_ptr(q_logits), _dtype_code(q_logits), n, V, stride, ids, float(temperature),
                                    int(K), _ptr(row_k), int(mode), _ptr(out["tok"]), _ptr(out.get("key")),
                                    _ptr(out["mult"]), _ptr(out["ndist"]), _ptr(out.get("samples")), _ptr(status),
                                    _ptr(ws), ws.numel(), _stream(stream, dev))
    _check("pps_draft_list", code)
    return out


def draft_list_noalloc(q_logits, key, ctx, pos, K: int, row_k=None, mode: int = DISTINCT, temperature: float = 1.0,
                       status=None, out=None, keys: bool = True, samples: bool = True, stream=None):
    """pps_draft_list_noalloc: pps_draft_list without a workspace, for callers
    that cannot allocate device memory per call (the library's built-in
    scratch serves up to NOALLOC_MAX_ROWS rows; calls must not overlap on the GPU)."""
    n, V, stride = _rows(q_logits)
    dev = q_logits.device
    if out is None:
        out = dict(tok=torch.empty(n, K, dtype=torch.int32, device=dev),
                   key=torch.empty(n, K, dtype=torch.float32, device=dev) if keys else None,
                   mult=torch.empty(n, K, dtype=torch.int32, device=dev),
                   ndist=torch.empty(n, dtype=torch.int32, device=dev),
                   samples=torch.empty(n, K, dtype=torch.int32, device=dev) if samples else None)
    _need_draft(out, n, K, row_k, status, dev)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        code = lib().pps_draft_list_noalloc(_ptr(q_logits), _dtype_code(q_logits), n, V, stride, ids,
                                            float(temperature), int(K), _ptr(row_k), int(mode), _ptr(out["tok"]),
                                            _ptr(out.get("key")), _ptr(out["mult"]), _ptr(out["ndist"]),
                                            _ptr(out.get("samples")), _ptr(status), _stream(stream, dev))
    _check("pps_draft_list_noalloc", code)
    return out


def verify_tree(p_logits, key, ctx, pos, gamma: int, seq_off, node_draft_row, draft_tok, draft_ndist, child_node,
                temperature: float = 1.0, ws=None, status=None, out=None, stream=None, top_k: int = 0,
                top_p: float = 1.0):
    """pps_verify_tree (pps_verify_tree_trunc when top_k > 0).
    Returns dict(winner, word, accept_len, n_emitted, emitted, score, score_sum)."""
    n, V, stride = _rows(p_logits)
    dev = p_logits.device
    n_seq = seq_off.numel() - 1
    K = draft_tok.shape[1]
    W = gamma + 1
    if out is None:
        out = dict(winner=torch.empty(n, dtype=torch.int32, device=dev),
                   word=torch.empty(n, dtype=torch.int32, device=dev),
                   accept_len=torch.empty(n_seq, dtype=torch.int32, device=dev),
                   n_emitted=torch.empty(n_seq, dtype=torch.int32, device=dev),
                   emitted=torch.empty(n_seq, W, dtype=torch.int32, device=dev),
                   score=torch.empty(n_seq, W, dtype=torch.float32, device=dev),
                   score_sum=torch.empty(n_seq, dtype=torch.float64, device=dev))
    if ws is None:
        ws = workspace(n, n_seq, dev)
    n_draft = draft_tok.shape[0]
    for name, t, numel in (("seq_off", seq_off, n_seq + 1), ("node_draft_row", node_draft_row, n),
                           ("draft_tok", draft_tok, n_draft * K), ("draft_ndist", draft_ndist, n_draft),
                           ("child_node", child_node, n_draft * K)):
        _need(name, t, dev, torch.int32, numel)
    _need_out(out, [("winner", torch.int32, n), ("word", torch.int32, n), ("accept_len", torch.int32, n_seq),
                    ("n_emitted", torch.int32, n_seq), ("emitted", torch.int32, n_seq * W),
                    ("score", torch.float32, n_seq * W), ("score_sum", torch.float64, n_seq)], dev)
    _need("status", status, dev, torch.int32, 1)
    _need("ws", ws, dev, torch.uint8)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        if top_k > 0:
            code = lib().pps_verify_tree_trunc(_ptr(p_logits), _dtype_code(p_logits), n, V, stride, ids,
                                               float(temperature), int(top_k), float(top_p), n_seq, int(gamma),
                                               _ptr(seq_off), _ptr(node_draft_row), n_draft, _ptr(draft_tok),
                                               _ptr(draft_ndist), int(K), _ptr(child_node), _ptr(out["winner"]),
                                               _ptr(out["word"]), _ptr(out["accept_len"]), _ptr(out["n_emitted"]),
                                               _ptr(out["emitted"]), _ptr(out["score"]), _ptr(out["score_sum"]),
                                               _ptr(status), _ptr(ws), ws.numel(), _stream(stream, dev))
            _check("pps_verify_tree_trunc", code)
            return out
        code = lib().pps_verify_tree(_ptr(p_logits), _dtype_code(p_logits), n, V, stride, ids, float(temperature),
                                     n_seq, int(gamma), _ptr(seq_off), _ptr(node_draft_row), n_draft,
                                     _ptr(draft_tok), _ptr(draft_ndist), int(K), _ptr(child_node),
                                     _ptr(out["winner"]), _ptr(out["word"]), _ptr(out["accept_len"]),
                                     _ptr(out["n_emitted"]), _ptr(out["emitted"]), _ptr(out["score"]),
                                     _ptr(out["score_sum"]), _ptr(status), _ptr(ws), ws.numel(),
                                     _stream(stream, dev))
    _check("pps_verify_tree", code)
    return out


def _need_detector(tokens, seg_off, n, n_seg, dev):
    if not isinstance(tokens, torch.Tensor) or tokens.dtype != torch.int32 or not tokens.is_cuda:
        raise TypeError("tokens must be a CUDA int32 tensor")
    _need("tokens", tokens, dev, torch.int32, n)
    if seg_off is not None and (seg_off.dtype != torch.int64 or not seg_off.is_cuda):
        raise TypeError("seg_off must be a CUDA int64 tensor")
    _need("seg_off", seg_off, dev, torch.int64, n_seg + 1)


def wm_score(tokens, key, ctx, pos, seg_off=None, out_score=None, out_sum=None, want_scores=True, stream=None):
    """pps_wm_score.  Returns (scores or None, sums)."""
    n = tokens.numel()
    dev = tokens.device
    n_seg = seg_off.numel() - 1 if seg_off is not None else 1
    if out_score is None and want_scores:
        out_score = torch.empty(n, dtype=torch.float32, device=dev)
    if out_sum is None:
        out_sum = torch.empty(n_seg, dtype=torch.float64, device=dev)
    _need_detector(tokens, seg_off, n, n_seg, dev)
    _need("out_score", out_score, dev, torch.float32, n)
    _need("out_sum", out_sum, dev, torch.float64, n_seg)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        code = lib().pps_wm_score(_ptr(tokens), ids, n, n_seg, _ptr(seg_off), _ptr(out_score), _ptr(out_sum),
                                  _stream(stream, dev))
    _check("pps_wm_score", code)
    return out_score, out_sum


def tree_expand(K: int, gamma: int, depth: int, draft, rows_key, rows_ctx, rows_pos, row_k, nxt: dict, child_node,
                nodes: dict, stream=None):
    """pps_tree_expand: children of depth `depth`'s rows (dynamic IID tree).  `draft` = the
    pps_draft_list (IID) outputs of those rows; writes nxt = dict(key, ctx, pos, k) of the next
    depth's rows, child_node and nodes = dict(key, ctx, pos) in place."""
    n_seq = nxt["k"].numel() // K
    dev = nxt["k"].device
    ids = _ids(rows_key, rows_ctx, rows_pos, 0, dev)
    with torch.cuda.device(dev):
        code = lib().pps_tree_expand(n_seq, int(K), int(gamma), int(depth), _ptr(draft["tok"]), _ptr(draft["mult"]),
                                     _ptr(draft["ndist"]), ids, _ptr(row_k), _ptr(nxt["key"]), _ptr(nxt["ctx"]),
                                     _ptr(nxt["pos"]), _ptr(nxt["k"]), _ptr(child_node), _ptr(nodes["key"]),
                                     _ptr(nodes["ctx"]), _ptr(nodes["pos"]), _stream(stream, dev))
    _check("pps_tree_expand", code)


def draft_hetero(q_logits, key, ctx, pos, row_block, n_blocks: int, temperature: float = 1.0, ws=None, status=None,
                 out_tok=None, out_key=None, stream=None, top_k: int = 0, top_p: float = 1.0):
    """pps_draft_hetero (pps_draft_hetero_trunc when top_k > 0): proposal row_block[r] of
    n_blocks at each row (non-identical proposals on the augmented source).  Returns the
    [n_rows] int32 tokens."""
    n, V, stride = _rows(q_logits)
    dev = q_logits.device
    if out_tok is None:
        out_tok = torch.empty(n, dtype=torch.int32, device=dev)
    if ws is None:
        ws = workspace(n, 0, dev)
    if row_block.dtype != torch.int32 or not row_block.is_cuda or not row_block.is_contiguous():
        raise TypeError("row_block must be a contiguous CUDA int32 tensor")
    _need("row_block", row_block, dev, torch.int32, n)
    _need("out_tok", out_tok, dev, torch.int32, n)
    _need("out_key", out_key, dev, torch.float32, n)
    _need("status", status, dev, torch.int32, 1)
    _need("ws", ws, dev, torch.uint8)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        if top_k > 0:
            code = lib().pps_draft_hetero_trunc(_ptr(q_logits), _dtype_code(q_logits), n, V, stride, ids,
                                                float(temperature), int(top_k), float(top_p), _ptr(row_block),
                                                int(n_blocks), _ptr(out_tok), _ptr(out_key), _ptr(status), _ptr(ws),
                                                ws.numel(), _stream(stream, dev))
            _check("pps_draft_hetero_trunc", code)
            return out_tok
        code = lib().pps_draft_hetero(_ptr(q_logits), _dtype_code(q_logits), n, V, stride, ids, float(temperature),
                                      _ptr(row_block), int(n_blocks), _ptr(out_tok), _ptr(out_key), _ptr(status),
                                      _ptr(ws), ws.numel(), _stream(stream, dev))
    _check("pps_draft_hetero", code)
    return out_tok


def hetero_expand(n_blocks: int, gamma: int, depth: int, draft_tok, rows_key, rows_ctx, rows_pos, row_owner,
                  nxt, lists: dict, nodes: dict, stream=None):
    """pps_hetero_expand: depth `depth` of the tree of n_blocks proposals.  Writes
    lists = dict(tok, ndist, child) of the depth's nodes, nodes = dict(key, ctx, pos) of
    the next depth's nodes and nxt = dict(key, ctx, pos, owner) of the next depth's
    proposal rows (None at the last depth) in place."""
    n_seq = row_owner.numel() // n_blocks
    nx = nxt or {}
    dev = row_owner.device
    ids = _ids(rows_key, rows_ctx, rows_pos, 0, dev)
    with torch.cuda.device(dev):
        code = lib().pps_hetero_expand(n_seq, int(n_blocks), int(gamma), int(depth), _ptr(draft_tok), ids,
                                       _ptr(row_owner), _ptr(nx.get("key")), _ptr(nx.get("ctx")), _ptr(nx.get("pos")),
                                       _ptr(nx.get("owner")), _ptr(lists["tok"]), _ptr(lists["ndist"]),
                                       _ptr(lists["child"]), _ptr(nodes["key"]), _ptr(nodes["ctx"]),
                                       _ptr(nodes["pos"]), _stream(stream, dev))
    _check("pps_hetero_expand", code)


def hetero_block(tokens, key, ctx, pos, n_blocks: int, out=None, stream=None):
    """pps_hetero_block: the block J of the target's augmented point for each token."""
    n = tokens.numel()
    dev = tokens.device
    if out is None:
        out = torch.empty(n, dtype=torch.int32, device=dev)
    _need_detector(tokens, None, n, 0, dev)
    _need("out", out, dev, torch.int32, n)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        code = lib().pps_hetero_block(_ptr(tokens), ids, n, int(n_blocks), _ptr(out), _stream(stream, dev))
    _check("pps_hetero_block", code)
    return out


SCORE_AARONSON, SCORE_U, SCORE_LI, SCORE_POWER_LAW = 0, 1, 2, 3


def wm_detect(tokens, key, ctx, pos, seg_off=None, kind: int = SCORE_AARONSON, param: float = 0.0,
              want_scores: bool = True, want_logp: bool = True, stream=None):
    """pps_wm_detect.  Returns (scores or None, sums, log p-values or None)."""
    n = tokens.numel()
    dev = tokens.device
    n_seg = seg_off.numel() - 1 if seg_off is not None else 1
    out_score = torch.empty(n, dtype=torch.float32, device=dev) if want_scores else None
    out_sum = torch.empty(n_seg, dtype=torch.float64, device=dev)
    out_logp = torch.empty(n_seg, dtype=torch.float64, device=dev) if want_logp else None
    _need_detector(tokens, seg_off, n, n_seg, dev)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        code = lib().pps_wm_detect(_ptr(tokens), ids, n, n_seg, _ptr(seg_off), int(kind), float(param),
                                   _ptr(out_score), _ptr(out_sum), _ptr(out_logp), _stream(stream, dev))
    _check("pps_wm_detect", code)
    return out_score, out_sum, out_logp


def philox_words(key, ctx, pos, vocab: int, arrival: int = 1, stream=None):
    n = key.numel()
    dev = key.device
    out = torch.empty(n, vocab, dtype=torch.int32, device=dev)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        _check("pps_philox_words", lib().pps_philox_words(ids, n, vocab, arrival, _ptr(out), _stream(stream, dev)))
    return out


def selftest_key_error(w_begin: int = 0, w_end: int = 1 << 32, stream=None) -> float:
    out = torch.zeros(1, dtype=torch.float32, device="cuda")
    _check("pps_selftest_key_error", lib().pps_selftest_key_error(w_begin, w_end, _ptr(out), _stream(stream)))
    return float(out.item())


def selftest_lg2_error(x_lo: float = 2.0 ** -40, x_hi: float = 2.0 ** 7, stream=None) -> float:
    """Largest |lg2.approx(x) - log2 x| over every fp32 x in [x_lo, x_hi)."""
    out = torch.zeros(1, dtype=torch.float32, device="cuda")
    _check("pps_selftest_lg2_error", lib().pps_selftest_lg2_error(float(x_lo), float(x_hi), _ptr(out),
                                                                  _stream(stream)))
    return float(out.item())


def selftest_philox_rate(n_blocks: int, out_len: int, stream=None):
    """Launch the Philox-only throughput kernel (returns the folded words)."""
    out = torch.empty(out_len, dtype=torch.int32, device="cuda")
    _check("pps_selftest_philox_rate", lib().pps_selftest_philox_rate(n_blocks, _ptr(out), out_len, _stream(stream)))
    return out


# ---------------------------------------------------------------- LM head (the race fused into the GEMM)

def _lm_operands(hidden, weight):
    """Shapes and strides of the bf16 hidden states [n, d] and LM-head matrix [V, d]."""
    for name, t in (("hidden", hidden), ("weight", weight)):
        if not isinstance(t, torch.Tensor) or not t.is_cuda or t.dim() != 2 or t.stride(1) != 1:
            raise TypeError(f"{name} must be a 2-D CUDA tensor with unit stride along d")
        if t.dtype != torch.bfloat16:
            raise TypeError(f"{name} must be bfloat16, got {t.dtype}")
    if hidden.device != weight.device:
        raise ValueError("hidden and weight must be on the same device")
    if hidden.shape[1] != weight.shape[1]:
        raise ValueError(f"hidden has d={hidden.shape[1]}, weight d={weight.shape[1]}")
    return hidden.shape[0], weight.shape[0], hidden.shape[1], hidden.stride(0), weight.stride(0)


def lmhead_workspace(n_rows: int, n_seq: int = 0, device=None) -> torch.Tensor:
    """A zeroed workspace for the fused LM-head calls."""
    nb = int(lib().pps_lmhead_workspace_size(n_rows, n_seq))
    return torch.zeros(nb, dtype=torch.uint8, device=device or "cuda")


def lmhead_logits(hidden, weight, out=None, stream=None):
    """pps_lmhead_logits: fp32 logits = hidden @ weight^T on the tensor cores (the unfused path)."""
    n, V, d, ldh, ldw = _lm_operands(hidden, weight)
    dev = hidden.device
    if out is None:
        out = torch.empty(n, V, dtype=torch.float32, device=dev)
    if out.dtype != torch.float32 or out.device != dev or out.dim() != 2 or out.stride(1) != 1 or \
            out.shape[0] < n or out.shape[1] < V:
        raise TypeError("out must be a float32 [n_rows, >= vocab] tensor on the operands' device")
    with torch.cuda.device(dev):
        code = lib().pps_lmhead_logits(_ptr(hidden), ldh, _ptr(weight), ldw, n, V, d, _ptr(out), out.stride(0),
                                       _stream(stream, dev))
    _check("pps_lmhead_logits", code)
    return out


def lmhead_draft_list(hidden, weight, key, ctx, pos, K: int, row_k=None, mode: int = DISTINCT,
                      temperature: float = 1.0, ws=None, status=None, out=None, keys: bool = True,
                      samples: bool = True, stream=None):
    """pps_lmhead_draft_list: the draft lists of pps_draft_list, computed in the LM-head GEMM's epilogue."""
    n, V, d, ldh, ldw = _lm_operands(hidden, weight)
    dev = hidden.device
    if out is None:
        out = dict(tok=torch.empty(n, K, dtype=torch.int32, device=dev),
                   key=torch.empty(n, K, dtype=torch.float32, device=dev) if keys else None,
                   mult=torch.empty(n, K, dtype=torch.int32, device=dev),
                   ndist=torch.empty(n, dtype=torch.int32, device=dev),
                   samples=torch.empty(n, K, dtype=torch.int32, device=dev) if samples else None)
    if ws is None:
        ws = lmhead_workspace(n, 0, dev)
    _need_draft(out, n, K, row_k, status, dev)
    _need("ws", ws, dev, torch.uint8)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        code = lib().pps_lmhead_draft_list(_ptr(hidden), ldh, _ptr(weight), ldw, n, V, d, ids, float(temperature),
                                           int(K), _ptr(row_k), int(mode), _ptr(out["tok"]), _ptr(out.get("key")),
                                           _ptr(out["mult"]), _ptr(out["ndist"]), _ptr(out.get("samples")),
                                           _ptr(status), _ptr(ws), ws.numel(), _stream(stream, dev))
    _check("pps_lmhead_draft_list", code)
    return out


def lmhead_verify_tree(hidden, weight, key, ctx, pos, gamma: int, seq_off, node_draft_row, draft_tok, draft_ndist,
                       child_node, temperature: float = 1.0, ws=None, status=None, out=None, stream=None):
    """pps_lmhead_verify_tree: the target race of every node, the tree walk and the scores of
    pps_verify_tree, computed in the LM-head GEMM's epilogue."""
    n, V, d, ldh, ldw = _lm_operands(hidden, weight)
    dev = hidden.device
    n_seq = seq_off.numel() - 1
    K = draft_tok.shape[1]
    W = gamma + 1
    if out is None:
        out = dict(winner=torch.empty(n, dtype=torch.int32, device=dev),
                   word=torch.empty(n, dtype=torch.int32, device=dev),
                   accept_len=torch.empty(n_seq, dtype=torch.int32, device=dev),
                   n_emitted=torch.empty(n_seq, dtype=torch.int32, device=dev),
                   emitted=torch.empty(n_seq, W, dtype=torch.int32, device=dev),
                   score=torch.empty(n_seq, W, dtype=torch.float32, device=dev),
                   score_sum=torch.empty(n_seq, dtype=torch.float64, device=dev))
    if ws is None:
        ws = lmhead_workspace(n, n_seq, dev)
    n_draft = draft_tok.shape[0]
    for name, t, numel in (("seq_off", seq_off, n_seq + 1), ("node_draft_row", node_draft_row, n),
                           ("draft_tok", draft_tok, n_draft * K), ("draft_ndist", draft_ndist, n_draft),
                           ("child_node", child_node, n_draft * K)):
        _need(name, t, dev, torch.int32, numel)
    _need_out(out, [("winner", torch.int32, n), ("word", torch.int32, n), ("accept_len", torch.int32, n_seq),
                    ("n_emitted", torch.int32, n_seq), ("emitted", torch.int32, n_seq * W),
                    ("score", torch.float32, n_seq * W), ("score_sum", torch.float64, n_seq)], dev)
    _need("status", status, dev, torch.int32, 1)
    _need("ws", ws, dev, torch.uint8)
    ids = _ids(key, ctx, pos, n, dev)
    with torch.cuda.device(dev):
        code = lib().pps_lmhead_verify_tree(_ptr(hidden), ldh, _ptr(weight), ldw, n, V, d, ids, float(temperature),
                                            n_seq, int(gamma), _ptr(seq_off), _ptr(node_draft_row), n_draft,
                                            _ptr(draft_tok), _ptr(draft_ndist), int(K), _ptr(child_node),
                                            _ptr(out["winner"]), _ptr(out["word"]), _ptr(out["accept_len"]),
                                            _ptr(out["n_emitted"]), _ptr(out["emitted"]), _ptr(out["score"]),
                                            _ptr(out["score_sum"]), _ptr(status), _ptr(ws), ws.numel(),
                                            _stream(stream, dev))
    _check("pps_lmhead_verify_tree", code)
    return out
