"""2048 px (128 x 128 = 16 384 tokens): the region-sparse step at four times
the token count of the 1024 px workload.  One block against the oracle
(localised dirty set, latent and recomputed cache rows); the full 28-block
step for the property that clean cache rows are left bit-identical."""
import numpy as np
import pytest
import torch

import oracle as O
from dataclasses import replace
from paper_2608_29809_gb300 import synth
from tests.gpu_cases import LATENT_REL_L2, block_close, rel_l2
from tests.oracle_inputs import weights64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def _localize(R, d, seed, frac):
    blobs = synth.ellipse_blobs(d, seed, frac)
    A, ids = synth.indicator_scores(d, blobs, seed)
    N = d.tokens
    ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8, device="cuda")
    mask = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
    R.rc_localize_mask(torch.from_numpy(np.ascontiguousarray(A)).cuda(), A.shape[0], N,
                       A.shape[2], d.grid_h, d.grid_w, ids, 0.5, 0, mask, idx, cnt, ws)
    _, want = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
    torch.cuda.synchronize()
    D = int(cnt.item())
    assert D == len(want)
    assert np.array_equal(np.sort(idx[:D].cpu().numpy()), np.sort(want))
    return idx, cnt, want


def test_2048_one_block_matches_oracle(R):
    d = replace(synth.PIXART_2048, layers=1, timesteps=2)
    seed = 1234 + 900
    t = 1
    w = synth.make_weights(d, seed)
    m = R.Model(d, w)
    try:
        text = synth.make_text(d, seed)
        R.rc_set_text(m.ctx, m.cache, 0, text.cuda())
        tv, ab = synth.ddim_tables(d.timesteps)
        R.rc_set_schedule(m.ctx, tv, ab)
        H, K, V = synth.make_cache_slice(d, seed, 0, 0, t)
        R.rc_cache_fill(m.cache, 0, 0, t, H.cuda(), K.cuda(), V.cuda())
        idx, cnt, want_idx = _localize(R, d, seed, 0.08)
        lat = synth.make_latent(d, seed)
        x = lat.clone().cuda()
        sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
        R.rc_step(m.ctx, m.cache, 0, x, t, sched, idx, -1, cnt)
        R.rc_sync(m.ctx)
        layers64, G64, pos64 = weights64(w)
        tkv64 = [O.text_kv(O.to64(text), L) for L in layers64]
        cache_t = [{"H": O.to64(H), "K": O.to64(K), "V": O.to64(V)}]
        want, _, cache = O.step(G64, layers64, pos64, O.to64(lat), t, O.MODE_SPARSE, want_idx,
                                cache_t, tkv64, tv.astype(np.float64), ab.astype(np.float64),
                                d.heads, d.grid_h, d.grid_w, d.patch, d.in_ch)
        assert rel_l2(x.cpu().double().numpy(), want) <= LATENT_REL_L2
        n, h = d.tokens, d.hidden
        got = [torch.empty(n, h, dtype=torch.bfloat16, device="cuda") for _ in range(3)]
        R.rc_cache_read(m.cache, 0, 0, t, *got)
        torch.cuda.synchronize()
        for name, g in zip("HKV", got):
            block_close(O.to64(g.cpu())[want_idx], cache[0][name][want_idx], f"2048 {name}")
    finally:
        m.close()


def test_2048_full_depth_leaves_clean_rows(R):
    """28 blocks at 16 384 tokens, 20 % dirty: the step runs, the latent is
    finite, and the cache rows of clean tokens are bit-identical afterwards
    while the dirty rows changed."""
    d = replace(synth.PIXART_2048, timesteps=2)
    seed = 1234 + 901
    t = 0
    w = synth.make_weights(d, seed, device="cuda")
    m = R.Model(d, w)
    try:
        R.rc_set_text(m.ctx, m.cache, 0, synth.make_text(d, seed, "cuda"))
        tv, ab = synth.ddim_tables(d.timesteps)
        R.rc_set_schedule(m.ctx, tv, ab)
        before = {}
        for l in range(d.layers):
            H, K, V = synth.make_cache_slice(d, seed, 0, l, t, device="cuda")
            R.rc_cache_fill(m.cache, 0, l, t, H, K, V)
            if l in (0, 27):
                before[l] = (H.cpu(), K.cpu(), V.cpu())
        idx, cnt, want_idx = _localize(R, d, seed, 0.2)
        x = synth.make_latent(d, seed, "cuda")
        sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
        R.rc_step(m.ctx, m.cache, 0, x, t, sched, idx, -1, cnt)
        R.rc_sync(m.ctx)
        assert torch.isfinite(x).all()
        clean = np.ones(d.tokens, bool)
        clean[want_idx] = False
        clean = torch.from_numpy(clean)
        n, h = d.tokens, d.hidden
        for l, old in before.items():
            got = [torch.empty(n, h, dtype=torch.bfloat16, device="cuda") for _ in range(3)]
            R.rc_cache_read(m.cache, 0, l, t, *got)
            torch.cuda.synchronize()
            for name, g, o in zip("HKV", got, old):
                g = g.cpu()
                assert torch.equal(g[clean], o[clean]), f"layer {l} {name} clean rows changed"
                assert not torch.equal(g[~clean], o[~clean]), f"layer {l} {name} dirty rows kept"
    finally:
        m.close()
