"""CUDA Graph replay of rc_step: one capture, replayed with new dirty-set
contents, matches the oracle and the direct rc_step."""
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


class Setup:
    def __init__(self, R, d, seed, t, host_cache=False):
        self.R, self.d, self.seed, self.t = R, d, seed, t
        self.w = synth.make_weights(d, seed)
        self.m = R.Model(d, self.w, host_cache=host_cache)
        text = synth.make_text(d, seed)
        R.rc_set_text(self.m.ctx, self.m.cache, 0, text.cuda())
        tv, ab = synth.ddim_tables(d.timesteps)
        self.tv, self.ab = tv.astype(np.float64), ab.astype(np.float64)
        R.rc_set_schedule(self.m.ctx, tv, ab)
        layers64, self.G64, self.pos64 = weights64(self.w)
        self.layers64 = layers64
        self.tkv64 = [O.text_kv(O.to64(text), L) for L in layers64]
        self.fill()

    def fill(self):
        self.cache64 = []
        for l in range(self.d.layers):
            H, K, V = synth.make_cache_slice(self.d, self.seed, 0, l, self.t)
            self.R.rc_cache_fill(self.m.cache, 0, l, self.t, H.cuda(), K.cuda(), V.cuda())
            self.cache64.append({"H": O.to64(H), "K": O.to64(K), "V": O.to64(V)})
        torch.cuda.synchronize()

    def oracle(self, lat, mode, idx):
        d = self.d
        return O.step(self.G64, self.layers64, self.pos64, O.to64(lat), self.t, mode, idx,
                      self.cache64, self.tkv64, self.tv, self.ab, d.heads, d.grid_h, d.grid_w,
                      d.patch, d.in_ch)

    def read(self, l):
        n, h = self.d.tokens, self.d.hidden
        H, K, V = (torch.empty(n, h, dtype=torch.bfloat16, device="cuda") for _ in range(3))
        self.R.rc_cache_read(self.m.cache, 0, l, self.t, H, K, V)
        torch.cuda.synchronize()
        return {"H": O.to64(H.cpu()), "K": O.to64(K.cpu()), "V": O.to64(V.cpu())}


def test_graph_replays_follow_the_dirty_buffers(R):
    """One SPARSE graph (D = -1, device count), replayed for three different
    regions written into the same index / count buffers, each from a fresh
    cache and latent: latent and the recomputed cache rows against the
    oracle, and the latent against a direct rc_step."""
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=4)
    S = Setup(R, d, 1234 + 800, t=2)
    try:
        N = d.tokens
        idx_buf = torch.zeros(N, dtype=torch.int32, device="cuda")
        cnt_buf = torch.zeros(1, dtype=torch.int32, device="cuda")
        lat_buf = torch.zeros_like(synth.make_latent(d, 0)).cuda()
        sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
        g = R.rc_step_graph_create(S.m.ctx, S.m.cache, 0, lat_buf, S.t, sched, idx_buf, -1,
                                   cnt_buf)
        try:
            n0 = R.rc_launch_count()
            regions = [np.flatnonzero(synth.rectangle_mask(d, 1234 + 800 + i)).astype(np.int32)
                       for i in range(2)] + [np.arange(0, N, 5, dtype=np.int32)]
            for i, idx in enumerate(regions):
                S.fill()
                lat = synth.make_latent(d, 1234 + 810 + i)
                lat_buf.copy_(lat.cuda())
                idx_buf.zero_()
                idx_buf[:len(idx)] = torch.from_numpy(idx).cuda()
                cnt_buf.fill_(len(idx))
                R.rc_graph_launch(g)
                R.rc_sync(S.m.ctx)
                got = lat_buf.cpu()
                want, _, cache = S.oracle(lat, O.MODE_SPARSE, idx)
                assert rel_l2(got.double().numpy(), want) <= LATENT_REL_L2, i
                for l in range(d.layers):
                    sl = S.read(l)
                    for k in ("H", "K", "V"):
                        block_close(sl[k][idx], cache[l][k][idx], f"region {i} layer {l} {k}")
                # the direct step from the same cache and latent
                S.fill()
                x = lat.clone().cuda()
                R.rc_step(S.m.ctx, S.m.cache, 0, x, S.t, sched, torch.from_numpy(idx).cuda(),
                          len(idx), None)
                R.rc_sync(S.m.ctx)
                assert rel_l2(x.cpu().double().numpy(), got.double().numpy()) <= 1e-3, i
            assert R.rc_launch_count() > n0
        finally:
            R.rc_graph_destroy(g)
    finally:
        S.m.close()


def test_graph_dense_and_reuse(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=4)
    S = Setup(R, d, 1234 + 801, t=1)
    try:
        for mode in (O.MODE_DENSE, O.MODE_REUSE):
            S.fill()
            lat = synth.make_latent(d, 1234 + 820 + mode)
            x = lat.clone().cuda()
            sched = np.full(d.timesteps, mode, np.uint8)
            g = R.rc_step_graph_create(S.m.ctx, S.m.cache, 0, x, S.t, sched, None, 0, None)
            try:
                R.rc_graph_launch(g)
                R.rc_sync(S.m.ctx)
            finally:
                R.rc_graph_destroy(g)
            want, _, _ = S.oracle(lat, mode, np.zeros(0, np.int32))
            assert rel_l2(x.cpu().double().numpy(), want) <= LATENT_REL_L2, mode
    finally:
        S.m.close()


def test_graph_refusals(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=1, timesteps=4)
    S = Setup(R, d, 1234 + 802, t=0, host_cache=True)
    try:
        x = synth.make_latent(d, 3).cuda()
        sched = np.full(d.timesteps, O.MODE_DENSE, np.uint8)
        with pytest.raises(R.RCError) as ei:
            R.rc_step_graph_create(S.m.ctx, S.m.cache, 0, x, 0, sched, None, 0, None)
        assert ei.value.status == 1
        with pytest.raises(R.RCError):
            R.rc_step_graph_create(S.m.ctx, S.m.cache, 0, x, 4, sched, None, 0, None)
    finally:
        S.m.close()
    S = Setup(R, d, 1234 + 803, t=0)
    try:
        x = synth.make_latent(d, 3).cuda()
        sched = np.full(d.timesteps, O.MODE_DENSE, np.uint8)
        R.rc_probe_enable(S.m.ctx, R.RC_PROBE_GEMM, 8)
        with pytest.raises(R.RCError):
            R.rc_step_graph_create(S.m.ctx, S.m.cache, 0, x, 0, sched, None, 0, None)
        R.rc_probe_enable(S.m.ctx, R.RC_PROBE_OFF, 0)
    finally:
        S.m.close()
