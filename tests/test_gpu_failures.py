"""Failure paths on the GPU, made without faulting it: a bounded device wait
that nothing ends gives up and is reported by rc_sync as RC_ERR_TIMEOUT, an
allocation beyond the device's memory returns RC_ERR_OOM, and in both cases
the context goes on working (a step afterwards matches the oracle)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.gpu_cases import LATENT_REL_L2, Problem, rel_l2

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def _step_matches(R, p):
    d = p.d
    idx = np.flatnonzero(synth.rectangle_mask(d, p.seed)).astype(np.int32)
    lat = synth.make_latent(d, p.seed)
    x = lat.clone().cuda()
    sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
    R.rc_step(p.model.ctx, p.model.cache, 0, x, 0, sched, torch.from_numpy(idx).cuda(),
              len(idx), None)
    R.rc_sync(p.model.ctx)
    want, _, _ = p.oracle_step(O.to64(lat), 0, O.MODE_SPARSE, idx)
    assert rel_l2(x.cpu().double().numpy(), want) <= LATENT_REL_L2


def test_bounded_wait_times_out_and_the_context_survives(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=2)
    p = Problem(R, d, 1234 + 800, ts=(0,))
    try:
        R.rc_selftest_wait(p.model.ctx, 20000, True)  # the flag is raised: no timeout
        R.rc_sync(p.model.ctx)
        R.rc_selftest_wait(p.model.ctx, 20000, False)  # nothing raises it: 20 ms, then give up
        with pytest.raises(R.RCError) as ei:
            R.rc_sync(p.model.ctx)
        assert ei.value.status == 5
        R.rc_sync(p.model.ctx)  # the error word was cleared
        _step_matches(R, p)
        with pytest.raises(R.RCError):
            R.rc_selftest_wait(p.model.ctx, 0, False)
    finally:
        p.close()


def test_allocation_beyond_the_device_is_refused_and_the_context_survives(R):
    d = synth.Dims(grid_h=64, grid_w=64, layers=28, timesteps=20)
    ctx = R.rc_create(R.dims_struct(d))
    try:
        free, total = torch.cuda.mem_get_info()
        per_session = d.timesteps * d.layers * 3 * d.tokens * d.hidden * 2
        sessions = int(total // per_session) + 2  # more than the whole device holds
        with pytest.raises(R.RCError) as ei:
            R.rc_cache_create(ctx, sessions)
        assert ei.value.status == 3
    finally:
        R.rc_destroy(ctx)
    p = Problem(R, synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=2), 1234 + 801, ts=(0,))
    try:
        _step_matches(R, p)
    finally:
        p.close()
