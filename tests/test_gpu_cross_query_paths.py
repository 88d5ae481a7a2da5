"""The two forms of the cross-attention query projection.  While the dirty
rows are fewer than 2048 or their count lives on the device, the projection
is folded into the text keys (one cross-attention kernel on x, five GEMMs per
block); with 2048 or more rows known on the host it runs as its own GEMM
(CTA pairs) before the cross-attention (six GEMMs per block).  Both sides of
the switch, and the dense step, against the oracle."""
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


@pytest.fixture(scope="module")
def problem(R):
    # 64 x 48 grid = 3072 tokens, so that a sparse step can hold 2047 or
    # 2048 dirty rows with clean rows left over
    d = synth.Dims(grid_h=64, grid_w=48, layers=2, timesteps=2)
    p = Problem(R, d, 1234 + 1100, ts=(1,))
    yield p
    p.close()


def _refill(R, p, t):
    for l in range(p.d.layers):
        H, K, V = synth.make_cache_slice(p.d, p.seed, 0, l, t)
        R.rc_cache_fill(p.model.cache, 0, l, t, H.cuda(), K.cuda(), V.cuda())
    torch.cuda.synchronize()


@pytest.mark.parametrize("case", ["sparse_2047", "sparse_2048", "dense"])
def test_cross_query_fold_switch(R, problem, case):
    p, d, t = problem, problem.d, 1
    rng = np.random.default_rng(p.seed + len(case))
    if case == "dense":
        mode, idx, gemms = O.MODE_DENSE, np.arange(d.tokens, dtype=np.int32), 6
    else:
        D = int(case.split("_")[1])
        mode, gemms = O.MODE_SPARSE, 5 if D < 2048 else 6
        idx = np.sort(rng.choice(d.tokens, D, replace=False)).astype(np.int32)
    _refill(R, p, t)
    lat = synth.make_latent(d, p.seed + 7)
    x = lat.clone().cuda()
    sched = np.full(d.timesteps, mode, np.uint8)
    cap = 8 * d.layers
    R.rc_probe_enable(p.model.ctx, R.RC_PROBE_GEMM, cap)
    if mode == O.MODE_DENSE:
        R.rc_step(p.model.ctx, p.model.cache, 0, x, t, sched, None, 0, None)
    else:
        R.rc_step(p.model.ctx, p.model.cache, 0, x, t, sched, torch.from_numpy(idx).cuda(),
                  len(idx), None)
    R.rc_sync(p.model.ctx)
    each = R.rc_probe_read_each(p.model.ctx, cap)
    R.rc_probe_enable(p.model.ctx, R.RC_PROBE_OFF, 0)
    assert len(each) == gemms * d.layers, f"{case}: {len(each)} GEMM launches"
    want, _, cache = p.oracle_step(O.to64(lat), t, mode,
                                   idx if mode == O.MODE_SPARSE else np.zeros(0, np.int32))
    err = rel_l2(x.cpu().double().numpy(), want)
    assert err <= LATENT_REL_L2, f"{case}: latent rel L2 {err:.2e}"
    for l in range(d.layers):
        sl = p.read_slot(l, t)
        for k in ("H", "K", "V"):
            block_close(sl[k][idx], cache[l][k][idx], f"{case} layer {l} {k}")
