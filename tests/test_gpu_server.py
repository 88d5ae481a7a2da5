"""The cross-session scheduler (rc_server_*): turns join while others run,
ticks batch up to max_items of them in round robin, and every session's
turn ends with the latent the oracle gives for its steps run in order."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.gpu_cases import LATENT_REL_L2, rel_l2
from tests.test_gpu_batched import Sessions

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def test_server_session_joins_mid_run(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=5)
    T = d.timesteps
    seed = 1234 + 700
    S = Sessions(R, d, seed, 3, max_batch=2)
    srv = None
    try:
        for s in range(3):
            for t in range(T):
                S.fill(s, t)
        scheds = [np.full(T, O.MODE_SPARSE, np.uint8),
                  O.schedule_first_k_dense(2, T),
                  np.array([O.MODE_REUSE] * 2 + [O.MODE_SPARSE] * (T - 2), np.uint8)]
        idx = [np.flatnonzero(synth.rectangle_mask(d, seed + s)).astype(np.int32)
               for s in range(3)]
        lat = [synth.make_latent(d, seed + s) for s in range(3)]
        x = [v.clone().cuda() for v in lat]
        idx_dev = [torch.from_numpy(i).cuda() for i in idx]
        cnt1 = torch.tensor([len(idx[1])], dtype=torch.int32).cuda()
        srv = R.rc_server_create(S.model.ctx, S.model.cache, 2)
        R.rc_server_admit(srv, 0, x[0], scheds[0], idx_dev[0], len(idx[0]), None)
        R.rc_server_admit(srv, 1, x[1], scheds[1], idx_dev[1], -1, cnt1)
        with pytest.raises(R.RCError):  # its turn is running
            R.rc_server_admit(srv, 0, x[0], scheds[0], idx_dev[0], len(idx[0]), None)
        ticks = [R.rc_server_tick(srv, 2), R.rc_server_tick(srv, 2)]
        assert ticks == [[0, 1], [0, 1]]
        assert R.rc_server_state(srv, 0) == 2 and R.rc_server_state(srv, 2) == -1
        # a third session joins while the two others are at t = 2
        R.rc_server_admit(srv, 2, x[2], scheds[2], idx_dev[2], len(idx[2]), None)
        while R.rc_server_running(srv):
            ticks.append(R.rc_server_tick(srv, 2))
        assert R.rc_server_tick(srv, 2) == []
        R.rc_sync(S.model.ctx)
        # round robin: the newcomer goes first, and every turn advances at
        # least every other tick while three are running
        assert ticks[2][0] == 2
        steps = {s: sum(s in tk for tk in ticks) for s in range(3)}
        assert steps == {0: T, 1: T, 2: T}
        for s in range(3):
            seen = [i for i, tk in enumerate(ticks) if s in tk]
            assert max(np.diff(seen)) <= 2
        for s in range(3):
            x64 = O.to64(lat[s])
            for t in range(T):
                x64, _, _ = S.oracle(s, x64, t, int(scheds[s][t]), idx[s])
            assert rel_l2(x[s].cpu().double().numpy(), x64) <= LATENT_REL_L2, s
    finally:
        if srv:
            R.rc_server_destroy(srv)
        S.close()


def test_server_rejects_bad_arguments(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=1, timesteps=3)
    S = Sessions(R, d, 9, 2, max_batch=2)
    srv = None
    try:
        with pytest.raises(R.RCError):
            R.rc_server_create(S.model.ctx, S.model.cache, 3)  # above max_batch
        srv = R.rc_server_create(S.model.ctx, S.model.cache, 2)
        x = synth.make_latent(d, 9).cuda()
        with pytest.raises(R.RCError):  # session out of range
            R.rc_server_admit(srv, 2, x, np.zeros(3, np.uint8), None, 0, None)
        with pytest.raises(R.RCError):  # no mode
            R.rc_server_admit(srv, 0, x, np.full(3, 7, np.uint8), None, 0, None)
        with pytest.raises(R.RCError):  # SPARSE without a dirty list
            R.rc_server_admit(srv, 0, x, np.ones(3, np.uint8), None, 4, None)
        assert R.rc_server_running(srv) == 0
    finally:
        if srv:
            R.rc_server_destroy(srv)
        S.close()
