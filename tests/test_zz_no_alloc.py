"""pps_draft_list_noalloc through the C ABI.

The no-alloc entry point serves callers that cannot allocate device memory
per call or pass a workspace (fixed-pool allocators, engine plugin hooks that
only see their input and output buffers).  It runs the same draft-list
computation on a built-in scratch array, so its outputs must match those of
pps_draft_list on the same inputs, on two calls in a row (the second call
reuses the scratch the first one left behind).  The file is named to be
collected last.
"""
import numpy as np
import pytest
import torch

from paper_2609_21858_gb300 import pps, synth

pytestmark = pytest.mark.gpu


def _cases():
    # bf16 rows split across warps (several warp slices per row) and small fp32 rows
    yield synth.make_workload("zipf_k8", device="cuda", n_seq=6)
    yield synth.make_workload("tiny", device="cuda", n_seq=40, seed=9)


@pytest.mark.parametrize("mode", [pps.DISTINCT, pps.IID])
def test_noalloc_matches_the_workspace_entry_point_on_two_calls(mode):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    for wl in _cases():
        t = wl.tree
        row_k = torch.as_tensor(t.row_k).cuda()
        args = (wl.q_logits, wl.draft_key, wl.draft_ctx, wl.draft_pos, t.K)
        ref = pps.draft_list(*args, row_k=row_k, mode=mode)
        for _ in range(2):
            status = torch.zeros(1, dtype=torch.int32, device="cuda")
            got = pps.draft_list_noalloc(*args, row_k=row_k, mode=mode, status=status)
            torch.cuda.synchronize()
            assert int(status.item()) == 0
            for k in ("tok", "mult", "ndist", "samples"):
                assert torch.equal(got[k], ref[k]), k
            valid = ref["tok"] >= 0
            np.testing.assert_allclose(got["key"][valid].cpu().numpy(), ref["key"][valid].cpu().numpy(),
                                       rtol=1e-5, atol=0)


def test_noalloc_rejects_rows_beyond_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    n = pps.NOALLOC_MAX_ROWS + 1
    q = torch.zeros(n, 64, dtype=torch.bfloat16, device="cuda")
    ids = torch.zeros(n, dtype=torch.int64, device="cuda")
    pos = torch.zeros(n, dtype=torch.int32, device="cuda")
    with pytest.raises(pps.PPSError) as e:
        pps.draft_list_noalloc(q, ids, ids, pos, 4)
    assert e.value.code == pps.ERR_SIZE
