"""The Python binding refuses buffers the library could overrun or that live on
another device: every check raises before anything is launched."""
import pytest
import torch

from paper_2609_21858_gb300 import pps

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    pps.lib()


def _rows(n, V=64):
    g = torch.Generator(device="cuda")
    g.manual_seed(1)
    q = torch.randn(n, V, generator=g, device="cuda")
    key = torch.arange(n, dtype=torch.int64, device="cuda")
    ctx = key * 7 + 3
    pos = torch.arange(n, dtype=torch.int32, device="cuda")
    return q, key, ctx, pos


def test_short_outputs_and_ids_are_refused():
    n, K = 6, 3
    q, key, ctx, pos = _rows(n)
    short = dict(tok=torch.empty(n * K - 1, dtype=torch.int32, device="cuda"),
                 mult=torch.empty(n * K, dtype=torch.int32, device="cuda"),
                 ndist=torch.empty(n, dtype=torch.int32, device="cuda"))
    with pytest.raises(ValueError):
        pps.draft_list(q, key, ctx, pos, K, out=short)
    with pytest.raises(ValueError):
        pps.draft_list(q, key[: n - 1], ctx, pos, K)
    with pytest.raises(ValueError):
        pps.draft_list(q, key, ctx, pos, K, row_k=torch.ones(n - 1, dtype=torch.int32, device="cuda"))
    with pytest.raises(TypeError):
        pps.draft_list(q, key, ctx, pos, K, row_k=torch.ones(n, dtype=torch.int64, device="cuda"))
    with pytest.raises(ValueError):
        pps.wm_score(torch.zeros(10, dtype=torch.int32, device="cuda"), key, ctx, pos)
    with pytest.raises(ValueError):
        pps.wm_detect(torch.zeros(n, dtype=torch.int32, device="cuda"), key, ctx[: n - 1], pos)


def test_short_tree_arrays_are_refused():
    n, K = 4, 2
    p, key, ctx, pos = _rows(n)
    seq_off = torch.tensor([0, n], dtype=torch.int32, device="cuda")
    ndr = torch.tensor([0, -1, -1, -1], dtype=torch.int32, device="cuda")
    tok = torch.tensor([[1, 2]], dtype=torch.int32, device="cuda")
    nd = torch.tensor([2], dtype=torch.int32, device="cuda")
    child = torch.tensor([[1, 2]], dtype=torch.int32, device="cuda")
    v = pps.verify_tree(p, key, ctx, pos, 1, seq_off, ndr, tok, nd, child)
    torch.cuda.synchronize()
    assert v["accept_len"].numel() == 1
    with pytest.raises(ValueError):
        pps.verify_tree(p, key, ctx, pos, 1, seq_off, ndr[:3], tok, nd, child)
    with pytest.raises(ValueError):
        pps.verify_tree(p, key, ctx, pos, 1, seq_off, ndr, tok, nd, child.view(-1)[:1].view(1, 1).expand(1, 1))
    bad = {k: x for k, x in v.items()}
    bad["emitted"] = torch.empty(1, dtype=torch.int32, device="cuda")
    with pytest.raises(ValueError):
        pps.verify_tree(p, key, ctx, pos, 1, seq_off, ndr, tok, nd, child, out=bad)


def test_tensors_on_another_device_are_refused():
    if torch.cuda.device_count() < 2:
        pytest.skip("one GPU: the cross-device check needs a second device")
    n, K = 4, 2
    q, key, ctx, pos = _rows(n)
    with pytest.raises(TypeError):
        pps.draft_list(q, key.to("cuda:1"), ctx, pos, K)
