"""Cache export / import: a session written to a file and read into another
cache (device or host tier) gives back every slot and the text keys/values
bit for bit, and a step from the imported cache matches the oracle.  A
session whose text keys may be stale (an import that failed part-way, layer
weights set again after rc_set_text) is refused until its text is set."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.gpu_cases import LATENT_REL_L2, rel_l2
from tests.oracle_inputs import weights64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    from paper_2608_29809_gb300 import build as B
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def _slots(R, m, d, s):
    out = []
    for t in range(d.timesteps):
        for l in range(d.layers):
            bufs = [torch.empty(d.tokens, d.hidden, dtype=torch.bfloat16, device="cuda")
                    for _ in range(3)]
            R.rc_cache_read(m.cache, s, l, t, *bufs)
            out.append([b.cpu() for b in bufs])
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("host_tier", [False, True])
def test_export_import_round_trip(R, tmp_path, host_tier):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=3)
    seed = 1234 + 950
    w = synth.make_weights(d, seed)
    src = R.Model(d, w, sessions=2)
    dst = R.Model(d, w, sessions=3, host_cache=host_tier)
    path = str(tmp_path / "session.rccache")
    try:
        text = synth.make_text(d, seed)
        R.rc_set_text(src.ctx, src.cache, 1, text.cuda())
        cache64 = {}
        for t in range(d.timesteps):
            for l in range(d.layers):
                H, K, V = synth.make_cache_slice(d, seed, 1, l, t)
                R.rc_cache_fill(src.cache, 1, l, t, H.cuda(), K.cuda(), V.cuda())
                cache64[(l, t)] = {"H": O.to64(H), "K": O.to64(K), "V": O.to64(V)}
        R.rc_cache_export(src.cache, 1, path)
        R.rc_cache_import(dst.cache, 2, path)
        a, b = _slots(R, src, d, 1), _slots(R, dst, d, 2)
        for x, y in zip(a, b):
            for u, v in zip(x, y):
                assert torch.equal(u, v)
        # the imported session steps (its text keys/values came with it)
        tv, ab = synth.ddim_tables(d.timesteps)
        R.rc_set_schedule(dst.ctx, tv, ab)
        idx = np.flatnonzero(synth.rectangle_mask(d, seed)).astype(np.int32)
        lat = synth.make_latent(d, seed)
        x = lat.clone().cuda()
        sched = np.full(d.timesteps, O.MODE_SPARSE, np.uint8)
        R.rc_step(dst.ctx, dst.cache, 2, x, 1, sched, torch.from_numpy(idx).cuda(), len(idx),
                  None)
        R.rc_sync(dst.ctx)
        layers64, G64, pos64 = weights64(w)
        tkv64 = [O.text_kv(O.to64(text), L) for L in layers64]
        want, _, _ = O.step(G64, layers64, pos64, O.to64(lat), 1, O.MODE_SPARSE, idx,
                            [cache64[(l, 1)] for l in range(d.layers)], tkv64,
                            tv.astype(np.float64), ab.astype(np.float64), d.heads, d.grid_h,
                            d.grid_w, d.patch, d.in_ch)
        assert rel_l2(x.cpu().double().numpy(), want) <= LATENT_REL_L2
    finally:
        src.close()
        dst.close()


def test_import_refuses_other_dims_and_bad_files(R, tmp_path):
    d = synth.Dims(grid_h=16, grid_w=16, layers=1, timesteps=2)
    w = synth.make_weights(d, 3)
    m = R.Model(d, w)
    d2 = synth.Dims(grid_h=16, grid_w=16, layers=1, timesteps=3)
    m2 = R.Model(d2, synth.make_weights(d2, 3))
    try:
        path = str(tmp_path / "a.rccache")
        R.rc_cache_export(m.cache, 0, path)
        with pytest.raises(R.RCError) as ei:
            R.rc_cache_import(m2.cache, 0, path)
        assert ei.value.status == 2
        bad = tmp_path / "bad.rccache"
        bad.write_bytes(b"not a cache file at all")
        with pytest.raises(R.RCError) as ei:
            R.rc_cache_import(m.cache, 0, str(bad))
        assert ei.value.status == 8
        with pytest.raises(R.RCError) as ei:
            R.rc_cache_import(m.cache, 0, str(tmp_path / "missing.rccache"))
        assert ei.value.status == 8
        short = tmp_path / "short.rccache"
        short.write_bytes(open(path, "rb").read()[:1000])
        with pytest.raises(R.RCError) as ei:
            R.rc_cache_import(m.cache, 0, str(short))
        assert ei.value.status == 8
        with pytest.raises(R.RCError):
            R.rc_cache_export(m.cache, 5, path)
    finally:
        m.close()
        m2.close()


def _reuse_step(R, m, d, x):
    sched = np.full(d.timesteps, O.MODE_REUSE, np.uint8)
    R.rc_step(m.ctx, m.cache, 0, x, 0, sched, None, 0, None)
    R.rc_sync(m.ctx)


def test_failed_import_and_new_weights_leave_the_text_unset(R, tmp_path):
    d = synth.Dims(grid_h=16, grid_w=16, layers=2, timesteps=2)
    w = synth.make_weights(d, 5)
    m = R.Model(d, w)
    try:
        tv, ab = synth.ddim_tables(d.timesteps)
        R.rc_set_schedule(m.ctx, tv, ab)
        text = synth.make_text(d, 5).cuda()
        R.rc_set_text(m.ctx, m.cache, 0, text)
        x = synth.make_latent(d, 5).cuda()
        _reuse_step(R, m, d, x)
        path = str(tmp_path / "s.rccache")
        R.rc_cache_export(m.cache, 0, path)
        # a short file past a good header: the slots were partly overwritten
        short = tmp_path / "short.rccache"
        short.write_bytes(open(path, "rb").read()[:100000])
        with pytest.raises(R.RCError) as ei:
            R.rc_cache_import(m.cache, 0, str(short))
        assert ei.value.status == 8
        with pytest.raises(R.RCError) as ei:
            _reuse_step(R, m, d, x)
        assert ei.value.status == 7 and "text" in str(ei.value)
        R.rc_cache_import(m.cache, 0, path)  # a whole file restores the session
        _reuse_step(R, m, d, x)
        # new weights for a layer: the text keys and folded keys are stale
        w2 = synth.make_weights(d, 6).to("cuda")
        R.rc_set_layer_weights(m.ctx, 1, w2.layers[1])
        with pytest.raises(R.RCError) as ei:
            _reuse_step(R, m, d, x)
        assert ei.value.status == 7 and "rc_set_text" in str(ei.value)
        R.rc_set_text(m.ctx, m.cache, 0, text)
        _reuse_step(R, m, d, x)
    finally:
        m.close()
