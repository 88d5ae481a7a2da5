"""GPU parity of rc_localize_scores: the localisation scores of Section 3.2
computed from the cached states of the previous turn (no dense step), the
mask the localisation kernel makes from them, and a whole editing turn
scheduled by Eq. 2 (REUSE steps, then SPARSE steps) whose edit region comes
from those scores."""
import numpy as np
import pytest
import torch
from scipy.ndimage import binary_dilation

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


def _gpu_scores(R, p, t, latent, ids):
    d = p.d
    scores = torch.full((d.tokens, d.text_len), float("nan"), device="cuda")
    R.rc_localize_scores(p.model.ctx, p.model.cache, 0, t, latent, ids, scores)
    R.rc_sync(p.model.ctx)
    return scores.cpu().double().numpy()


def _ref_scores(p, t, latent64, ids):
    d = p.d
    cache_t = [p.cache64[(l, t)] for l in range(d.layers)]
    return O.cached_localization_scores(p.G64, p.layers64, p.pos64, latent64, cache_t, p.tkv64,
                                        d.heads, d.grid_h, d.grid_w, d.patch, ids, d.text_len)


def _normalised(col):
    lo, hi = col.min(), col.max()
    return (col - lo) / (hi - lo)


def _gpu_mask(R, scores, ids, d, dil=1):
    N = d.tokens
    ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8, device="cuda")
    mask = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
    R.rc_localize_mask(scores, 1, N, d.text_len, d.grid_h, d.grid_w, ids, 0.5, dil, mask, idx,
                       cnt, ws)
    torch.cuda.synchronize()
    return mask, idx, cnt


def _check_mask(mask_gpu, ref, ids, d, dil=1):
    """The GPU mask equals the oracle's except on tokens whose normalised
    oracle score lies within 0.02 of the threshold (or next to one, through
    the dilation)."""
    m_ref, _ = O.localize_mask(ref.astype(np.float32)[None], ids, d.grid_h, d.grid_w, 0.5, dil)
    diff = np.flatnonzero(mask_gpu != m_ref)
    if len(diff):
        near = np.zeros(d.tokens, bool)
        for j in ids:
            near |= np.abs(_normalised(ref[:, j]) - 0.5) <= 0.02
        if dil:
            near = binary_dilation(near.reshape(d.grid_h, d.grid_w),
                                   np.ones((2 * dil + 1, 2 * dil + 1), bool)).reshape(-1)
        assert np.all(near[diff]), diff[~near[diff]]
    return m_ref


@pytest.mark.parametrize("ids", [[3], [0, 17, 63, 64, 119], [5, 9, 33, 70, 71, 100, 118, 119]])
def test_cached_scores_small(R, ids):
    d = synth.Dims(grid_h=16, grid_w=16, layers=3, timesteps=20)
    p = Problem(R, d, 1234 + 520, ts=(7,))
    try:
        ids = np.array(ids, np.int32)
        lat = synth.make_latent(d, p.seed)
        got = _gpu_scores(R, p, 7, lat.cuda(), ids)
        ref = _ref_scores(p, 7, O.to64(lat), ids)
        other = np.setdiff1d(np.arange(d.text_len), ids)
        assert np.all(got[:, other] == 0)
        block_close(got[:, ids], ref[:, ids], "cached scores")
        # the cache is only read
        slot = p.read_slot(1, 7)
        for k in "HKV":
            assert np.array_equal(slot[k], p.cache64[(1, 7)][k])
    finally:
        p.close()


def test_cached_scores_then_localise_512px(R):
    """28 blocks at 1024 tokens: scores from the cache feed the localisation
    kernel; the normalised scores agree with the oracle's to 0.02.  (The
    synthetic states are unrelated to the text, so the regions are scattered:
    no dilation, or the union would cover the grid.)"""
    d = synth.PIXART_512
    p = Problem(R, d, 1234 + 521, ts=(3,))
    try:
        ids = np.array([4, 31, 77], np.int32)
        lat = synth.make_latent(d, p.seed)
        got = _gpu_scores(R, p, 3, lat.cuda(), ids)
        ref = _ref_scores(p, 3, O.to64(lat), ids)
        block_close(got[:, ids], ref[:, ids], "cached scores")
        for j in ids:
            assert np.max(np.abs(_normalised(got[:, j]) - _normalised(ref[:, j]))) <= 0.02
        mask, idx, cnt = _gpu_mask(R, torch.from_numpy(got.astype(np.float32)[None]).cuda(),
                                   ids, d, 0)
        _check_mask(mask.cpu().numpy(), ref, ids, d, 0)
        assert 0 < int(cnt.item()) < d.tokens
    finally:
        p.close()


def test_eq2_turn_localised_from_the_cache_1024_tokens(R):
    """One editing turn at 1024 tokens under rc_reuse_schedule (Eq. 2,
    s < tau_s: the first floor(rho T) steps REUSE, then SPARSE): at the first
    SPARSE step the new prompt's delta tokens are localised from the cached
    states, and the turn's final latent matches the oracle's."""
    d = synth.Dims(grid_h=32, grid_w=32, layers=4, timesteps=10)
    T = d.timesteps
    p = Problem(R, d, 1234 + 522, ts=tuple(range(T)))
    try:
        # the new turn's prompt: its text keys replace the previous ones
        text = synth.make_text(d, p.seed + 1)
        R.rc_set_text(p.model.ctx, p.model.cache, 0, text.cuda())
        p.tkv64 = [O.text_kv(O.to64(text), L) for L in p.layers64]
        modes = R.rc_reuse_schedule(0.3, 0.8, T, 0.2)
        assert modes.tolist() == [O.MODE_REUSE] * 2 + [O.MODE_SPARSE] * (T - 2)
        ids = np.array([6, 40, 95], np.int32)
        lat = synth.make_latent(d, p.seed)
        x = lat.clone().cuda()
        x64 = O.to64(lat)
        idx_dev = cnt = None
        idx_host = None
        for t in range(T):
            if modes[t] == O.MODE_SPARSE and idx_dev is None:
                got = _gpu_scores(R, p, t, x, ids)
                ref = _ref_scores(p, t, x64, ids)
                block_close(got[:, ids], ref[:, ids], f"cached scores at t = {t}")
                # (scattered regions on synthetic states: no dilation)
                mask, idx_dev, cnt = _gpu_mask(
                    R, torch.from_numpy(got.astype(np.float32)[None]).cuda(), ids, d, 0)
                _check_mask(mask.cpu().numpy(), ref, ids, d, 0)
                D = int(cnt.item())
                assert 0 < D < d.tokens
                idx_host = idx_dev[:D].cpu().numpy()
            R.rc_step(p.model.ctx, p.model.cache, 0, x, t, modes, idx_dev,
                      -1 if idx_dev is not None else 0, cnt)
            x64, _, _ = p.oracle_step(x64, t, int(modes[t]), idx_host)
        R.rc_sync(p.model.ctx)
        assert rel_l2(x.cpu().double().numpy(), x64) <= LATENT_REL_L2
    finally:
        p.close()
