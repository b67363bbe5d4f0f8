"""C-ABI checks that need no GPU: the library loads, exports every entry point
include/pps.h declares, and rejects invalid arguments before launching anything."""
import ctypes
import os
import re

import pytest

from paper_2609_21858_gb300 import pps

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    txt = open(os.path.join(ROOT, "include", "pps.h")).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(pps_[a-z0-9_]+)\s*\(", txt)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("pps_draft_list", "pps_verify_tree", "pps_wm_score", "pps_workspace_size", "pps_philox_words"):
        assert n in names


def test_library_exports_every_declared_symbol():
    L = pps.lib()
    for n in _declared():
        assert hasattr(L, n), n
    assert "sm_103a" in pps.version()


def test_binding_selects_the_keyed_source_build():
    # the binding loads libpps.so (Philox4x32-10) unless told otherwise, and use_library switches
    # builds (loading a library and asking its rounds need no GPU)
    import os as _os
    assert _os.path.basename(pps.library_path(10)) == "libpps.so"
    assert _os.path.basename(pps.library_path(7)) == "libpps_r7.so"
    with pytest.raises(ValueError):
        pps.library_path(8)
    default = 10 if not _os.environ.get("PPS_PHILOX_ROUNDS") else int(_os.environ["PPS_PHILOX_ROUNDS"])
    try:
        pps.use_library(7)
        assert pps.philox_rounds() == 7 and "Philox4x32-7" in pps.version()
        pps.use_library(10)
        assert pps.philox_rounds() == 10 and "Philox4x32-10" in pps.version()
    finally:
        pps.use_library(default)
    assert pps.philox_rounds() == default


def test_both_keyed_source_builds_export_every_symbol_and_report_their_rounds():
    # libpps.so: Philox4x32-10; libpps_r7.so: the same sources built with PPS_PHILOX_ROUNDS=7
    # (loading the libraries and these two queries need no GPU)
    for rounds in (10, 7):
        L = ctypes.CDLL(pps.library_path(rounds))
        for n in _declared():
            assert hasattr(L, n), (rounds, n)
        L.pps_philox_rounds.restype = ctypes.c_int
        L.pps_version.restype = ctypes.c_char_p
        assert L.pps_philox_rounds() == rounds
        assert f"Philox4x32-{rounds}".encode() in L.pps_version()


def _ids0():
    return pps.RowIds(None, None, None)


def test_validation_rejects_bad_arguments_without_a_gpu():
    L = pps.lib()
    fake = ctypes.c_void_p(256)  # never dereferenced: every call below fails validation first
    ids = pps.RowIds(256, 256, 256)
    ws = 1 << 30

    def draft(**kw):
        a = dict(logits=fake, dtype=pps.BF16, n=4, V=100, stride=100, ids=ids, T=1.0, K=4, mode=pps.DISTINCT,
                 tok=fake, mult=fake, nd=fake, ws=fake, wsb=ws)
        a.update(kw)
        return L.pps_draft_list(a["logits"], a["dtype"], a["n"], a["V"], a["stride"], a["ids"], a["T"], a["K"], None,
                                a["mode"], a["tok"], None, a["mult"], a["nd"], None, None, a["ws"], a["wsb"], None)

    assert draft(K=0) == pps.ERR_INVALID_ARG
    assert draft(K=33) == pps.ERR_INVALID_ARG
    assert draft(K=8, V=5, stride=5) == pps.ERR_INVALID_ARG
    assert draft(stride=99) == pps.ERR_INVALID_ARG
    assert draft(T=0.0) == pps.ERR_INVALID_ARG
    assert draft(T=float("nan")) == pps.ERR_INVALID_ARG
    assert draft(dtype=7) == pps.ERR_UNSUPPORTED
    assert draft(mode=5) == pps.ERR_UNSUPPORTED
    assert draft(ids=_ids0()) == pps.ERR_INVALID_ARG
    assert draft(tok=None) == pps.ERR_INVALID_ARG
    assert draft(ws=None) == pps.ERR_WORKSPACE
    assert draft(wsb=16) == pps.ERR_WORKSPACE
    assert draft(n=0) == pps.OK  # nothing to do, nothing launched

    def verify(**kw):
        a = dict(n=10, V=100, gamma=2, n_seq=2, K=2, ws=fake, wsb=ws, seq=fake)
        a.update(kw)
        return L.pps_verify_tree(fake, pps.F32, a["n"], a["V"], a["V"], ids, 1.0, a["n_seq"], a["gamma"], a["seq"],
                                 fake, a.get("nd", 4), fake, fake, a["K"], fake, fake, fake, fake, fake, fake, fake, fake, None,
                                 a["ws"], a["wsb"], None)

    assert verify(gamma=0) == pps.ERR_INVALID_ARG
    assert verify(gamma=65) == pps.ERR_INVALID_ARG
    assert verify(n_seq=11) == pps.ERR_INVALID_ARG
    assert verify(K=0) == pps.ERR_INVALID_ARG
    assert verify(seq=None) == pps.ERR_INVALID_ARG
    assert verify(nd=-1) == pps.ERR_INVALID_ARG
    assert verify(wsb=0) == pps.ERR_WORKSPACE
    assert L.pps_wm_score(fake, ids, -1, 1, None, fake, None, None) == pps.ERR_INVALID_ARG
    assert L.pps_wm_score(fake, ids, 10, 1, None, None, None, None) == pps.ERR_INVALID_ARG
    assert L.pps_wm_score(fake, ids, 10, 0, fake, fake, None, None) == pps.ERR_INVALID_ARG
    assert L.pps_philox_words(ids, 1, 10, 0, fake, None) == pps.ERR_INVALID_ARG
    assert L.pps_selftest_key_error(0, (1 << 32) + 1, fake, None) == pps.ERR_INVALID_ARG
    assert L.pps_selftest_lg2_error(0.0, 1.0, fake, None) == pps.ERR_INVALID_ARG
    assert L.pps_selftest_lg2_error(2.0, 1.0, fake, None) == pps.ERR_INVALID_ARG
    assert L.pps_selftest_lg2_error(1.0, 2.0, None, None) == pps.ERR_INVALID_ARG


def test_workspace_size_grows_with_rows_and_sequences():
    a = pps.workspace_size(100, 1000, 8, 0)
    b = pps.workspace_size(200, 1000, 8, 0)
    c = pps.workspace_size(200, 1000, 8, 50)
    assert 0 < a < b <= c
    assert pps.status_string(pps.ERR_WORKSPACE) == "workspace missing or too small"


def test_truncated_calls_validate_top_k_and_top_p():
    L = pps.lib()
    fake = ctypes.c_void_p(256)
    ids = pps.RowIds(256, 256, 256)

    def draft(tk, tp, **kw):
        a = dict(K=4, ws=fake)
        a.update(kw)
        return L.pps_draft_list_trunc(fake, pps.BF16, 4, 100, 100, ids, 1.0, tk, tp, a["K"], None, pps.DISTINCT,
                                      fake, None, fake, fake, None, None, a["ws"], 1 << 30, None)

    def verify(tk, tp):
        return L.pps_verify_tree_trunc(fake, pps.F32, 10, 100, 100, ids, 1.0, tk, tp, 2, 2, fake, fake, 4, fake, fake,
                                       2, fake, fake, fake, fake, fake, fake, fake, fake, None, fake, 1 << 30, None)

    for tk, tp in ((0, 1.0), (-3, 1.0), (pps.MAX_TOP_K + 1, 1.0), (5, 0.0), (5, -0.5), (5, 1.01),
                   (5, float("nan"))):
        assert draft(tk, tp) == pps.ERR_INVALID_ARG, (tk, tp)
        assert verify(tk, tp) == pps.ERR_INVALID_ARG, (tk, tp)
    assert draft(5, 0.9, K=0) == pps.ERR_INVALID_ARG   # the untruncated checks still apply
    assert draft(5, 0.9, ws=None) == pps.ERR_WORKSPACE


def test_detect_validates_kind_and_parameter():
    L = pps.lib()
    fake = ctypes.c_void_p(256)
    ids = pps.RowIds(256, 256, 256)

    def detect(kind, param, out_sum=fake, out_logp=fake):
        return L.pps_wm_detect(fake, ids, 10, 1, None, kind, param, None, out_sum, out_logp, None)

    assert detect(7, 0.0) == pps.ERR_UNSUPPORTED
    for bad in (0.0, 1.0, -0.5, float("nan")):
        assert detect(pps.SCORE_LI, bad) == pps.ERR_INVALID_ARG
    for bad in (0.0, 1.5, float("nan")):
        assert detect(pps.SCORE_POWER_LAW, bad) == pps.ERR_INVALID_ARG
    assert detect(pps.SCORE_AARONSON, 0.0, out_sum=None) == pps.ERR_INVALID_ARG  # p-values need the sums


def test_tree_expand_validates_shape_arguments():
    L = pps.lib()
    fake = ctypes.c_void_p(256)
    ids = pps.RowIds(256, 256, 256)

    def expand(n_seq=4, K=4, gamma=3, depth=0, tok=fake):
        return L.pps_tree_expand(n_seq, K, gamma, depth, tok, fake, fake, ids, fake, fake, fake, fake, fake, fake,
                                 fake, fake, fake, None)

    for kw in (dict(K=0), dict(K=33), dict(gamma=0), dict(gamma=65), dict(depth=-1), dict(depth=3), dict(n_seq=-1),
               dict(tok=None)):
        assert expand(**kw) == pps.ERR_INVALID_ARG, kw
    assert expand(n_seq=0) == pps.OK


def test_hetero_entry_points_validate_arguments():
    L = pps.lib()
    fake = ctypes.c_void_p(256)
    ids = pps.RowIds(256, 256, 256)
    ws = pps.workspace_size(8, 0, 1, 0)

    def draft(n_rows=8, V=100, stride=100, T=1.0, block=fake, B=4, tok=fake, ws_bytes=ws, dtype=pps.BF16):
        return L.pps_draft_hetero(fake, dtype, n_rows, V, stride, ids, T, block, B, tok, None, None, fake, ws_bytes,
                                  None)

    for kw in (dict(B=0), dict(B=33), dict(stride=99), dict(T=0.0), dict(block=None), dict(tok=None),
               dict(n_rows=-1), dict(V=0)):
        assert draft(**kw) == pps.ERR_INVALID_ARG, kw
    assert draft(ws_bytes=ws - 1) == pps.ERR_WORKSPACE
    assert draft(dtype=7) == pps.ERR_UNSUPPORTED
    assert draft(n_rows=0) == pps.OK

    def trunc(top_k=50, top_p=1.0, B=4):
        return L.pps_draft_hetero_trunc(fake, pps.BF16, 8, 100, 100, ids, 1.0, top_k, top_p, fake, B, fake, None,
                                        None, fake, ws, None)

    for kw in (dict(top_k=0), dict(top_k=65), dict(top_p=0.0), dict(top_p=1.5), dict(B=0)):
        assert trunc(**kw) == pps.ERR_INVALID_ARG, kw

    def expand(n_seq=4, B=4, gamma=3, depth=0, tok=fake, nxt=fake):
        return L.pps_hetero_expand(n_seq, B, gamma, depth, tok, ids, fake, nxt, nxt, nxt, nxt, fake, fake, fake,
                                   fake, fake, fake, None)

    for kw in (dict(B=0), dict(B=33), dict(gamma=0), dict(gamma=65), dict(depth=-1), dict(depth=3), dict(n_seq=-1),
               dict(tok=None), dict(nxt=None)):
        assert expand(**kw) == pps.ERR_INVALID_ARG, kw
    assert expand(n_seq=0) == pps.OK

    def block(n=5, B=3, tok=fake, out=fake):
        return L.pps_hetero_block(tok, ids, n, B, out, None)

    for kw in (dict(B=0), dict(B=33), dict(n=-1), dict(tok=None), dict(out=None)):
        assert block(**kw) == pps.ERR_INVALID_ARG, kw
    assert block(n=0) == pps.OK


def _header_defines():
    txt = open(os.path.join(ROOT, "include", "pps.h")).read()
    return {m.group(1): int(m.group(2)) for m in re.finditer(r"#define\s+(PPS_[A-Z0-9_]+)\s+(\d+)u?\b", txt)}


def test_binding_constants_match_the_header():
    d = _header_defines()
    assert d["PPS_NOALLOC_MAX_ROWS"] == pps.NOALLOC_MAX_ROWS
    assert d["PPS_MAX_K"] == pps.MAX_K and d["PPS_MAX_TOP_K"] == pps.MAX_TOP_K and d["PPS_MAX_BLOCKS"] == pps.MAX_BLOCKS
    assert (d["PPS_FLAG_GUARD"], d["PPS_FLAG_LOGIT_RANGE"], d["PPS_FLAG_TREE"]) == (
        pps.FLAG_GUARD, pps.FLAG_LOGIT_RANGE, pps.FLAG_TREE)
    # the stated scratch size: a 272-byte partial list per (row + warp) slot and two counters per row
    assert d["PPS_NOALLOC_SCRATCH_BYTES"] == 272 * (d["PPS_NOALLOC_MAX_ROWS"] + d["PPS_NOALLOC_MAX_WARPS"]) + \
        8 * d["PPS_NOALLOC_MAX_ROWS"]


def test_noalloc_entry_point_rejects_bad_arguments_without_a_gpu():
    # every refusal below returns before the scratch address is looked up (no CUDA call)
    L = pps.lib()
    fake = ctypes.c_void_p(256)
    ids = pps.RowIds(256, 256, 256)

    def draft(**kw):
        a = dict(logits=fake, dtype=pps.BF16, n=4, V=100, stride=100, ids=ids, T=1.0, K=4, mode=pps.DISTINCT,
                 tok=fake, mult=fake, nd=fake)
        a.update(kw)
        return L.pps_draft_list_noalloc(a["logits"], a["dtype"], a["n"], a["V"], a["stride"], a["ids"], a["T"],
                                        a["K"], None, a["mode"], a["tok"], None, a["mult"], a["nd"], None, None, None)

    assert draft(K=0) == pps.ERR_INVALID_ARG
    assert draft(K=pps.MAX_K + 1) == pps.ERR_INVALID_ARG
    assert draft(K=8, V=5, stride=5) == pps.ERR_INVALID_ARG
    assert draft(stride=99) == pps.ERR_INVALID_ARG
    assert draft(T=0.0) == pps.ERR_INVALID_ARG
    assert draft(dtype=7) == pps.ERR_UNSUPPORTED
    assert draft(mode=5) == pps.ERR_UNSUPPORTED
    assert draft(ids=_ids0()) == pps.ERR_INVALID_ARG
    for name in ("tok", "mult", "nd"):
        assert draft(**{name: None}) == pps.ERR_INVALID_ARG, name
    assert draft(n=pps.NOALLOC_MAX_ROWS + 1) == pps.ERR_SIZE
    assert draft(n=0) == pps.OK


def test_lmhead_entry_points_validate_arguments():
    L = pps.lib()
    fake = ctypes.c_void_p(256)
    odd = ctypes.c_void_p(258)  # not 16-byte aligned
    ids = pps.RowIds(256, 256, 256)
    ws = int(L.pps_lmhead_workspace_size(8, 4))
    assert ws >= 8 * 32 * 128

    def logits(hidden=fake, ldh=64, weight=fake, ldw=64, n=8, V=100, d=64, out=fake, ldo=100):
        return L.pps_lmhead_logits(hidden, ldh, weight, ldw, n, V, d, out, ldo, None)

    for kw in (dict(d=0), dict(V=0), dict(n=-1), dict(ldh=32), dict(ldw=60), dict(ldh=68), dict(ldo=99),
               dict(weight=None), dict(hidden=None), dict(out=None), dict(hidden=odd), dict(weight=odd)):
        assert logits(**kw) == pps.ERR_INVALID_ARG, kw
    assert logits(n=0) == pps.OK

    def draft(K=4, mode=pps.DISTINCT, T=1.0, tok=fake, wsb=ws, **kw):
        a = dict(hidden=fake, ldh=64, weight=fake, ldw=64, n=8, V=100, d=64)
        a.update(kw)
        return L.pps_lmhead_draft_list(a["hidden"], a["ldh"], a["weight"], a["ldw"], a["n"], a["V"], a["d"], ids, T,
                                       K, None, mode, tok, None, fake, fake, None, None, fake, wsb, None)

    assert draft(K=0) == pps.ERR_INVALID_ARG
    assert draft(K=pps.LMHEAD_MAX_K + 1) == pps.ERR_INVALID_ARG
    assert draft(T=0.0) == pps.ERR_INVALID_ARG
    assert draft(mode=3) == pps.ERR_UNSUPPORTED
    assert draft(tok=None) == pps.ERR_INVALID_ARG
    assert draft(ldw=12) == pps.ERR_INVALID_ARG
    assert draft(wsb=16) == pps.ERR_WORKSPACE
    assert draft(n=0) == pps.OK

    def verify(gamma=2, n_seq=2, K=2, wsb=ws, seq=fake):
        return L.pps_lmhead_verify_tree(fake, 64, fake, 64, 8, 100, 64, ids, 1.0, n_seq, gamma, seq, fake, 4, fake,
                                        fake, K, fake, fake, fake, fake, fake, fake, fake, fake, None, fake, wsb, None)

    for kw in (dict(gamma=0), dict(gamma=65), dict(n_seq=9), dict(K=0), dict(seq=None)):
        assert verify(**kw) == pps.ERR_INVALID_ARG, kw
    assert verify(wsb=0) == pps.ERR_WORKSPACE
    assert _header_defines()["PPS_LMHEAD_MAX_K"] == pps.LMHEAD_MAX_K
