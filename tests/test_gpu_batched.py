"""Batched serving: several sessions' denoising steps in one rc_step_batched
call (varlen dirty queries, each item over its own session's keys / values,
timestep and text), against the oracle run item by item."""
import numpy as np
import pytest
import torch

import oracle as O
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


def _localize(R, A, ids, d):
    N = d.tokens
    ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8, device="cuda")
    mask = torch.zeros(N, dtype=torch.uint8, device="cuda")
    idx = torch.zeros(N, dtype=torch.int32, device="cuda")
    cnt = torch.zeros(1, dtype=torch.int32, device="cuda")
    R.rc_localize_mask(torch.from_numpy(np.ascontiguousarray(A)).cuda(), A.shape[0], N,
                       A.shape[2], d.grid_h, d.grid_w, ids, 0.5, 0, mask, idx, cnt, ws)
    return idx, cnt


class Sessions:
    """One model with `n` sessions: shared weights, a text context and
    cache slices per session, on both sides."""

    def __init__(self, R, d, seed, n, max_batch):
        self.R, self.d, self.seed = R, d, seed
        w = synth.make_weights(d, seed)
        self.model = R.Model(d, w, sessions=n, max_batch=max_batch)
        self.layers64, self.G64, self.pos64 = weights64(w)
        self.tkv64 = []
        for s in range(n):
            text = synth.make_text(d, seed + 1000 * s)
            R.rc_set_text(self.model.ctx, self.model.cache, s, text.cuda())
            ctx64 = O.to64(text)
            self.tkv64.append([O.text_kv(ctx64, L) for L in self.layers64])
        tv, ab = synth.ddim_tables(d.timesteps)
        self.tv, self.ab = tv.astype(np.float64), ab.astype(np.float64)
        R.rc_set_schedule(self.model.ctx, tv, ab)
        self.cache64 = {}

    def fill(self, s, t):
        for l in range(self.d.layers):
            H, K, V = synth.make_cache_slice(self.d, self.seed, s, l, t)
            self.R.rc_cache_fill(self.model.cache, s, l, t, H.cuda(), K.cuda(), V.cuda())
            self.cache64[(s, l, t)] = {"H": O.to64(H), "K": O.to64(K), "V": O.to64(V)}
        torch.cuda.synchronize()

    def oracle(self, s, latent64, t, mode, idx):
        d = self.d
        cache_t = [self.cache64[(s, l, t)] for l in range(d.layers)]
        return O.step(self.G64, self.layers64, self.pos64, latent64, t, mode, idx, cache_t,
                      self.tkv64[s], self.tv, self.ab, d.heads, d.grid_h, d.grid_w, d.patch,
                      d.in_ch)

    def read(self, s, l, t):
        n, h = self.d.tokens, self.d.hidden
        H, K, V = (torch.empty(n, h, dtype=torch.bfloat16, device="cuda") for _ in range(3))
        self.R.rc_cache_read(self.model.cache, s, l, t, H, K, V)
        torch.cuda.synchronize()
        return {"H": O.to64(H.cpu()), "K": O.to64(K.cpu()), "V": O.to64(V.cpu())}

    def close(self):
        self.model.close()


def test_c5_batched_eight_sessions_1024(R):
    """8 concurrent 512 px sessions (1024 tokens, 28 blocks, T = 20), each at
    its own timestep with its own text and a ragged dirty fraction drawn from
    U(2 %, 35 %): one rc_step_batched call, dirty counts left on the device."""
    d = synth.PIXART_512
    seed = 1234 + 400
    n = 8
    S = Sessions(R, d, seed, n, max_batch=n)
    try:
        rng = np.random.default_rng(seed)
        items, ref = [], []
        fracs = rng.uniform(0.02, 0.35, size=n)
        ts = rng.integers(0, d.timesteps, size=n)
        for s in range(n):
            t = int(ts[s])
            S.fill(s, t)
            blobs = synth.ellipse_blobs(d, seed + s, float(fracs[s]))
            A, ids = synth.indicator_scores(d, blobs, seed + s)
            idx_d, cnt = _localize(R, A, ids, d)
            _, idx = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
            lat = synth.make_latent(d, seed + s)
            items.append(dict(session=s, latent=lat.clone().cuda(), t=t, mode=O.MODE_SPARSE,
                              dirty_idx=idx_d, D=-1, dirty_count=cnt))
            ref.append((idx, O.to64(lat), t))
        torch.cuda.synchronize()
        counts = [int(it["dirty_count"].item()) for it in items]
        assert counts == [len(r[0]) for r in ref]
        assert len(set(counts)) > 1  # ragged
        R.rc_step_batched(S.model.ctx, S.model.cache, items)
        R.rc_sync(S.model.ctx)
        for s, (it, (idx, lat64, t)) in enumerate(zip(items, ref)):
            got = it["latent"].cpu().double().numpy()
            want, eps, cache = S.oracle(s, lat64, t, O.MODE_SPARSE, idx)
            assert rel_l2(got, want) <= LATENT_REL_L2, s
            for l in (0, d.layers - 1):
                sl = S.read(s, l, t)
                for k in ("H", "K", "V"):
                    block_close(sl[k][idx], cache[l][k][idx], f"session {s} layer {l} {k}")
    finally:
        S.close()


def test_batched_mixed_modes_match_single_steps(R):
    """A batch mixing SPARSE (host and device counts), DENSE and REUSE items
    on a 16 x 16 grid matches the oracle item by item and the library's own
    one-item rc_step."""
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=20)
    seed = 1234 + 401
    S = Sessions(R, d, seed, 4, max_batch=4)
    try:
        modes = [O.MODE_SPARSE, O.MODE_SPARSE, O.MODE_DENSE, O.MODE_REUSE]
        ts = [3, 3, 5, 7]
        items, ref = [], []
        for s in range(4):
            S.fill(s, ts[s])
            idx = np.flatnonzero(synth.rectangle_mask(d, seed + s)).astype(np.int32)
            lat = synth.make_latent(d, seed + s)
            it = dict(session=s, latent=lat.clone().cuda(), t=ts[s], mode=modes[s])
            if modes[s] == O.MODE_SPARSE:
                it["dirty_idx"] = torch.from_numpy(idx).cuda()
                if s == 0:
                    it["D"] = len(idx)
                else:
                    it["D"] = -1
                    it["dirty_count"] = torch.tensor([len(idx)], dtype=torch.int32).cuda()
            items.append(it)
            ref.append((idx, O.to64(lat)))
        R.rc_step_batched(S.model.ctx, S.model.cache, items)
        R.rc_sync(S.model.ctx)
        batched = [it["latent"].cpu().double().numpy() for it in items]
        for s in range(4):
            want, _, _ = S.oracle(s, ref[s][1], ts[s], modes[s], ref[s][0])
            assert rel_l2(batched[s], want) <= LATENT_REL_L2, s
        # the same steps one at a time, from the same caches
        for s in range(4):
            S.fill(s, ts[s])
            it = items[s]
            lat = torch.from_numpy(ref[s][1].astype(np.float32)).cuda()
            sched = np.full(d.timesteps, modes[s], np.uint8)
            R.rc_step(S.model.ctx, S.model.cache, s, lat, ts[s], sched, it.get("dirty_idx"),
                      it.get("D", 0), it.get("dirty_count"))
            R.rc_sync(S.model.ctx)
            assert rel_l2(batched[s], lat.cpu().double().numpy()) <= 1e-3, s
    finally:
        S.close()


def test_batched_rejects_bad_items(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=1, timesteps=4)
    S = Sessions(R, d, 7, 2, max_batch=2)
    try:
        lat = [synth.make_latent(d, 7).cuda() for _ in range(3)]
        same = [dict(session=0, latent=lat[0], t=1, mode=O.MODE_DENSE),
                dict(session=0, latent=lat[1], t=1, mode=O.MODE_DENSE)]
        with pytest.raises(R.RCError) as ei:
            R.rc_step_batched(S.model.ctx, S.model.cache, same)
        assert ei.value.status == 1
        three = [dict(session=s % 2, latent=lat[s], t=s, mode=O.MODE_DENSE) for s in range(3)]
        with pytest.raises(R.RCError):
            R.rc_step_batched(S.model.ctx, S.model.cache, three)
        bad = [dict(session=0, latent=lat[0], t=0, mode=O.MODE_SPARSE, dirty_idx=None, D=5)]
        with pytest.raises(R.RCError):
            R.rc_step_batched(S.model.ctx, S.model.cache, bad)
    finally:
        S.close()
