"""rc_set_deterministic: with the gated residual GEMMs on whole tiles, a
region-sparse step repeated from the same state gives the same bits
(direct and from a CUDA graph), and still matches the oracle.  Shapes of the
1024 px model (4096 tokens, hidden 1152) with two blocks and ~20 % dirty, the
row count where the default schedule splits the residual reductions."""
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


@pytest.fixture(scope="module")
def prob(R):
    p = Problem(R, synth.Dims(grid_h=64, grid_w=64, layers=2), 1234 + 950, ts=(4,))
    yield p
    p.close()


def _reset(R, p, t):
    for l in range(p.d.layers):
        H, K, V = synth.make_cache_slice(p.d, p.seed, 0, l, t)
        R.rc_cache_fill(p.model.cache, 0, l, t, H.cuda(), K.cuda(), V.cuda())
    torch.cuda.synchronize()


def _slots(R, p, t):
    n, h = p.d.tokens, p.d.hidden
    out = []
    for l in range(p.d.layers):
        H, K, V = (torch.empty(n, h, dtype=torch.bfloat16, device="cuda") for _ in range(3))
        R.rc_cache_read(p.model.cache, 0, l, t, H, K, V)
        out += [H, K, V]
    torch.cuda.synchronize()
    return [a.cpu() for a in out]


def test_deterministic_step_repeats_bitwise(R, prob):
    p, d, t = prob, prob.d, 4
    idx = np.flatnonzero(np.any(synth.ellipse_blobs(d, p.seed, 0.2), axis=0)).astype(np.int32)
    assert 700 <= len(idx) <= 950
    lat = synth.make_latent(d, p.seed)
    idx_d = torch.from_numpy(idx).cuda()
    cnt = torch.tensor([len(idx)], dtype=torch.int32, device="cuda")
    sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
    R.rc_set_deterministic(p.model.ctx, True)
    try:
        runs = []
        for _ in range(2):
            _reset(R, p, t)
            x = lat.clone().cuda()
            R.rc_step(p.model.ctx, p.model.cache, 0, x, t, sched, idx_d, -1, cnt)
            R.rc_sync(p.model.ctx)
            runs.append((x.cpu(), _slots(R, p, t)))
        # the same step from a CUDA graph captured in this mode, replayed twice
        x = lat.clone().cuda()
        g = R.rc_step_graph_create(p.model.ctx, p.model.cache, 0, x, t, sched, idx_d, -1, cnt)
        try:
            for _ in range(2):
                _reset(R, p, t)
                x.copy_(lat.cuda())
                R.rc_graph_launch(g)
                R.rc_sync(p.model.ctx)
                runs.append((x.cpu(), _slots(R, p, t)))
        finally:
            R.rc_graph_destroy(g)
    finally:
        R.rc_set_deterministic(p.model.ctx, False)
    for lat_i, slots_i in runs[1:]:
        assert torch.equal(lat_i, runs[0][0])
        for a, b in zip(slots_i, runs[0][1]):
            assert torch.equal(a, b)
    ref, _, _ = p.oracle_step(O.to64(lat), t, O.MODE_SPARSE, idx)
    assert rel_l2(runs[0][0].double().numpy(), ref) <= LATENT_REL_L2
    _reset(R, p, t)


def test_deterministic_flag_rejects_null_context(R):
    with pytest.raises(R.RCError):
        R.rc_set_deterministic(None, True)
