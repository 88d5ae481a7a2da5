"""GPU parity of the localisation scores captured from the model's own
cross-attention during a DENSE step (Section 3.2), and of the mask the
localisation kernel makes from them."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.gpu_cases import LATENT_REL_L2, Problem, block_close, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def _capture(R, p, t, ids):
    d = p.d
    lat = synth.make_latent(d, p.seed)
    latent = lat.clone().cuda()
    scores = torch.full((d.tokens, d.text_len), float("nan"), device="cuda")
    R.rc_step_capture(p.model.ctx, p.model.cache, 0, latent, t, ids, scores)
    R.rc_sync(p.model.ctx)
    cache_t = [p.cache64[(l, t)] for l in range(d.layers)]
    ref = O.step_capture(p.G64, p.layers64, p.pos64, O.to64(lat), t, cache_t, p.tkv64,
                         p.tv.astype(np.float64), p.ab.astype(np.float64), d.heads, d.grid_h,
                         d.grid_w, d.patch, d.in_ch, ids, d.text_len)
    return latent.cpu().double().numpy(), scores.cpu().double().numpy(), ref


def _normalised(col):
    lo, hi = col.min(), col.max()
    return (col - lo) / (hi - lo)


@pytest.mark.parametrize("ids", [[3], [0, 17, 63, 64, 119], [5, 9, 33, 70, 71, 100, 118, 119]])
def test_capture_scores_small(R, ids):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=20)
    p = Problem(R, d, 1234 + 500, ts=(4,))
    try:
        got_lat, got, (ref_lat, _, _, ref) = _capture(R, p, 4, np.array(ids, np.int32))
        assert rel_l2(got_lat, ref_lat) <= LATENT_REL_L2
        other = np.setdiff1d(np.arange(d.text_len), ids)
        assert np.all(got[:, other] == 0)
        block_close(got[:, ids], ref[:, ids], "captured scores")
    finally:
        p.close()


def test_capture_then_localise_512px(R):
    """28 blocks at 1024 tokens: the DENSE step's captured scores feed the
    localisation kernel; the normalised scores agree with the oracle's to
    0.02, so the masks may differ only on tokens that close to the threshold."""
    d = synth.PIXART_512
    p = Problem(R, d, 1234 + 501, ts=(0,))
    try:
        ids = np.array([4, 31, 77], np.int32)
        got_lat, got, (ref_lat, _, _, ref) = _capture(R, p, 0, ids)
        assert rel_l2(got_lat, ref_lat) <= LATENT_REL_L2
        block_close(got[:, ids], ref[:, ids], "captured scores")
        for j in ids:
            assert np.max(np.abs(_normalised(got[:, j]) - _normalised(ref[:, j]))) <= 0.02
        N = d.tokens
        ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8, device="cuda")
        mask = torch.zeros(N, dtype=torch.uint8, device="cuda")
        idx = torch.zeros(N, dtype=torch.int32, device="cuda")
        cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
        R.rc_localize_mask(torch.from_numpy(got.astype(np.float32)[None]).cuda(), 1, N, d.text_len,
                           d.grid_h, d.grid_w, ids, 0.5, 1, mask, idx, cnt, ws)
        torch.cuda.synchronize()
        m_ref, _ = O.localize_mask(ref.astype(np.float32)[None], ids, d.grid_h, d.grid_w, 0.5, 1)
        diff = np.flatnonzero(mask.cpu().numpy() != m_ref)
        if len(diff):
            # a flipped token is (or is next to, through the dilation) a token
            # whose normalised oracle score lies within 0.02 of the threshold
            near = np.zeros(N, bool)
            for j in ids:
                near |= np.abs(_normalised(ref[:, j]) - 0.5) <= 0.02
            near = near.reshape(d.grid_h, d.grid_w)
            from scipy.ndimage import binary_dilation
            near = binary_dilation(near, np.ones((3, 3), bool)).reshape(-1)
            assert np.all(near[diff]), diff[~near[diff]]
        assert 0 < int(cnt.item()) < N
    finally:
        p.close()
