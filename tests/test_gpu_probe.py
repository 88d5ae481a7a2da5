"""The timing probe records one event pair per launch of the chosen kernel
class (5 GEMMs, 2 attentions, 2 LayerNorm modulations per block) without
changing what the step computes."""
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


def test_probe_counts_and_step_unchanged(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=3, timesteps=4)
    p = Problem(R, d, 1234 + 990, ts=(2,))
    try:
        idx = np.flatnonzero(synth.rectangle_mask(d, p.seed)).astype(np.int32)
        lat = synth.make_latent(d, p.seed)
        want, _, _ = p.oracle_step(O.to64(lat), 2, O.MODE_SPARSE, idx)
        sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
        # five GEMMs per block: the cross-query projection is folded into the
        # text keys when the text fits one cross-attention pass
        per_block = {R.RC_PROBE_GEMM: 5, R.RC_PROBE_ATTENTION: 2, R.RC_PROBE_LN: 2}
        for which, k in per_block.items():
            for l in range(d.layers):  # the same cache for every run
                H, K, V = synth.make_cache_slice(d, p.seed, 0, l, 2)
                R.rc_cache_fill(p.model.cache, 0, l, 2, H.cuda(), K.cuda(), V.cuda())
            cap = 64
            R.rc_probe_enable(p.model.ctx, which, cap)
            x = lat.clone().cuda()
            R.rc_step(p.model.ctx, p.model.cache, 0, x, 2, sched, torch.from_numpy(idx).cuda(),
                      len(idx), None)
            R.rc_sync(p.model.ctx)
            each = R.rc_probe_read_each(p.model.ctx, cap)
            R.rc_probe_enable(p.model.ctx, R.RC_PROBE_OFF, 0)
            assert len(each) == k * d.layers, which
            assert all(t > 0 for t in each), which
            assert rel_l2(x.cpu().double().numpy(), want) <= LATENT_REL_L2, which
    finally:
        p.close()
