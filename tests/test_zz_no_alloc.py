"""rc_localize_mask_noalloc, the allocation-free localisation entry point.

Callers inside an allocator-free context (an inference server's plugin hook,
a program whose device memory belongs to another framework's pool, a
latency-critical loop that cannot take cudaMalloc's device-wide
synchronisation) use this variant; it keeps its scratch in a fixed array of
the library.  Its masks and dirty lists must equal those of the workspace
entry point bit for bit, also on consecutive calls that reuse the same
scratch with different problems.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_29809_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def _outputs(N):
    mask = torch.full((N,), 9, dtype=torch.uint8, device="cuda")
    idx = torch.full((N,), -3, dtype=torch.int32, device="cuda")
    cnt = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    return mask, idx, cnt


def _with_workspace(R, A_dev, ids, d, dil):
    N = d.tokens
    mask, idx, cnt = _outputs(N)
    ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8, device="cuda")
    R.rc_localize_mask(A_dev, A_dev.shape[0], N, d.text_len, d.grid_h, d.grid_w, ids, 0.5, dil,
                       mask, idx, cnt, ws)
    torch.cuda.synchronize()
    D = int(cnt.item())
    return mask.cpu(), idx[:D].cpu(), D


def _no_alloc(R, A_dev, ids, d, dil):
    N = d.tokens
    mask, idx, cnt = _outputs(N)
    R.rc_localize_mask_noalloc(A_dev, A_dev.shape[0], N, d.text_len, d.grid_h, d.grid_w, ids,
                               0.5, dil, mask, idx, cnt)
    torch.cuda.synchronize()
    D = int(cnt.item())
    return mask.cpu(), idx[:D].cpu(), D


def _check_case(R, d, seed, dil, n_delta=(3, 8)):
    A, ids = synth.blob_scores(d, seed, n_delta=n_delta)
    A_dev = torch.from_numpy(A).cuda()
    ref = _with_workspace(R, A_dev, ids, d, dil)
    got = _no_alloc(R, A_dev, ids, d, dil)
    assert got[2] == ref[2] and 0 < got[2] < d.tokens
    assert torch.equal(got[0], ref[0])
    assert torch.equal(got[1], ref[1])
    # and against the oracle's float32 localisation, bit for bit
    m_ref, idx_ref = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, dil)
    assert np.array_equal(got[0].numpy(), m_ref)
    assert np.array_equal(got[1].numpy(), idx_ref)


def test_no_alloc_matches_workspace_entry_point_on_two_calls(R):
    # two different problems in a row: the second call finds the first call's
    # data in the shared scratch and must not depend on it
    _check_case(R, synth.Dims(grid_h=64, grid_w=64), 31, 1)
    _check_case(R, synth.Dims(grid_h=32, grid_w=40), 32, 2)


def test_no_alloc_at_its_limit_then_a_small_case(R):
    # 128 x 128 tokens with 16 delta ids uses the scratch to its last byte;
    # a small problem right after it must not see the large one's data
    d = synth.Dims(grid_h=128, grid_w=128)
    assert R.rc_localize_workspace_size(d.tokens, 16) == R.RC_NOALLOC_SCRATCH_BYTES
    _check_case(R, d, 33, 1, n_delta=(16, 16))
    _check_case(R, synth.Dims(grid_h=24, grid_w=24), 34, 1, n_delta=(2, 2))


def test_no_alloc_rejects_sizes_beyond_its_scratch(R):
    d = synth.Dims(grid_h=8, grid_w=8)
    A_dev = torch.zeros((1, d.tokens, d.text_len), device="cuda")
    mask, idx, cnt = _outputs(d.tokens)
    ids = np.arange(17, dtype=np.int32)  # one more delta token than the scratch allows
    with pytest.raises(R.RCError) as ei:
        R.rc_localize_mask_noalloc(A_dev, 1, d.tokens, d.text_len, d.grid_h, d.grid_w, ids, 0.5,
                                   1, mask, idx, cnt)
    assert ei.value.status == 2 and "n_delta <= 16" in str(ei.value)
    # one token more than the scratch allows (a 113 x 145 grid)
    with pytest.raises(R.RCError) as ei:
        R.rc_localize_mask_noalloc(A_dev, 1, 113 * 145, d.text_len, 113, 145, ids[:2], 0.5, 1,
                                   mask, idx, cnt)
    assert ei.value.status == 2 and "N <= 16384" in str(ei.value)
