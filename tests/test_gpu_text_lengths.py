"""Text conditioning of other lengths than 120 tokens.  Up to 128 text
tokens the cross-attention runs in one pass with the query projection folded
into the keys (padded key rows masked out of the softmax); above 128 the
query projection is a GEMM and the cross-attention the stream-K kernel over
64-key blocks with a ragged last block.  1 token (softmax over a single key),
77 (ragged), 128 (the one-pass limit) and 200 against the oracle, with the
dirty count read on the device and given on the host."""
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


@pytest.mark.parametrize("M", [1, 77, 128, 200])
def test_text_length_sparse_step(R, M):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=2, text_len=M)
    t = 1
    p = Problem(R, d, 1234 + 1200 + M, ts=(t,))
    try:
        idx = np.flatnonzero(synth.rectangle_mask(d, p.seed)).astype(np.int32)
        lat = synth.make_latent(d, p.seed)
        want, _, cache = p.oracle_step(O.to64(lat), t, O.MODE_SPARSE, idx)
        sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
        di = torch.from_numpy(idx).cuda()
        cnt = torch.tensor([len(idx)], dtype=torch.int32, device="cuda")
        for on_device in (True, False):
            for l in range(d.layers):
                H, K, V = synth.make_cache_slice(d, p.seed, 0, l, t)
                R.rc_cache_fill(p.model.cache, 0, l, t, H.cuda(), K.cuda(), V.cuda())
            x = lat.clone().cuda()
            if on_device:
                R.rc_step(p.model.ctx, p.model.cache, 0, x, t, sched, di, -1, cnt)
            else:
                R.rc_step(p.model.ctx, p.model.cache, 0, x, t, sched, di, len(idx), None)
            R.rc_sync(p.model.ctx)
            what = f"M {M} count on {'device' if on_device else 'host'}"
            err = rel_l2(x.cpu().double().numpy(), want)
            assert err <= LATENT_REL_L2, f"{what}: latent rel L2 {err:.2e}"
            for l in range(d.layers):
                sl = p.read_slot(l, t)
                for k in ("H", "K", "V"):
                    block_close(sl[k][idx], cache[l][k][idx], f"{what} layer {l} {k}")
    finally:
        p.close()
