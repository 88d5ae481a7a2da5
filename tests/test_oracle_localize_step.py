"""Pins of the oracle's localisation, timestep, patch, final-layer, DDIM,
step and schedule arithmetic (CPU only)."""
import math
import os

import numpy as np
import pytest
import scipy.ndimage as ndi
import torch
import torch.nn.functional as F

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import rng, weights64

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------ localisation
def _read_localize_golden():
    sec, data = None, {"scores": [], "union": [], "mask": []}
    for ln in open(os.path.join(GOLDEN, "localize_6x6.txt")):
        ln = ln.strip()
        if not ln or ln.startswith("#"):
            continue
        if ln.startswith("["):
            sec = ln[1:-1]
            continue
        data[sec].append([float(v) for v in ln.split()])
    return (np.array(data["scores"], np.float32)[None], np.array(data["union"], np.uint8),
            np.array(data["mask"], np.uint8))


def test_localize_golden_6x6():
    A, union, mask = _read_localize_golden()
    m, idx = O.localize_mask(A, [1, 3], 6, 6, 0.5, 1)
    assert np.array_equal(m.reshape(6, 6), mask)
    assert np.array_equal(idx, np.flatnonzero(mask.reshape(-1)))
    m0, _ = O.localize_mask(A, [1, 3], 6, 6, 0.5, 0)
    assert np.array_equal(m0.reshape(6, 6), union)
    # ">=" at the boundary: a strict comparison would drop token 31
    m_strict, _ = O.localize_mask(A, [1, 3], 6, 6, np.nextafter(np.float32(0.5), 1), 0)
    assert m_strict[31] == 0 and m0[31] == 1


@pytest.mark.parametrize("pos", [(0, 0), (0, 5), (3, 0), (3, 4), (7, 7)])
def test_localize_one_hot_dilates_to_clipped_square(pos):
    gh, gw = 8, 8
    A = np.zeros((1, gh * gw, 5), np.float32)
    A[0, pos[0] * gw + pos[1], 2] = 1.0
    m, idx = O.localize_mask(A, [2], gh, gw, 0.5, 1)
    ys = range(max(0, pos[0] - 1), min(gh, pos[0] + 2))
    xs = range(max(0, pos[1] - 1), min(gw, pos[1] + 2))
    want = sorted(y * gw + x for y in ys for x in xs)
    assert idx.tolist() == want
    corner = pos in [(0, 0), (7, 7)]
    if corner:
        assert len(idx) == 4


def test_localize_constant_column_is_empty():
    A = np.full((1, 16, 3), 0.25, np.float32)
    m, idx = O.localize_mask(A, [0, 1, 2], 4, 4, 0.5, 1)
    assert m.sum() == 0 and idx.size == 0


def test_localize_non_finite_column_is_dropped():
    # NaN or +-Inf anywhere in a delta column: the min-max normalisation is
    # undefined, the column gives no token, the other columns are unaffected
    gh, gw = 6, 6
    A = np.zeros((1, gh * gw, 4), np.float32)
    A[0, 7, 1] = 1.0
    A[0, 20, 2] = 1.0
    for bad in (np.nan, np.inf, -np.inf):
        B = A.copy()
        B[0, 30, 2] = bad
        m, idx = O.localize_mask(B, [1, 2], gh, gw, 0.5, 0)
        assert idx.tolist() == [7]
        m, idx = O.localize_mask(B, [2], gh, gw, 0.0, 0)
        assert idx.size == 0
    # finite slices whose f32 sum overflows: the mean is +Inf, dropped too
    C = np.stack([A[0], A[0]])
    C[:, 20, 2] = 3.0e38
    m, idx = O.localize_mask(C, [1, 2], gh, gw, 0.5, 0)
    assert idx.tolist() == [7]


def test_localize_plateau_rectangle_grows_by_one():
    gh, gw = 10, 12
    A = rng(3).uniform(0, 0.3, (1, gh * gw, 4)).astype(np.float32)
    g = np.zeros((gh, gw), bool)
    g[3:6, 4:9] = True
    A[0, g.reshape(-1), 1] = 1.0
    m, _ = O.localize_mask(A, [1], gh, gw, 0.5, 1)
    want = np.zeros((gh, gw), bool)
    want[2:7, 3:10] = True
    assert np.array_equal(m.reshape(gh, gw).astype(bool), want)


def test_localize_matches_scipy_dilation_and_union_properties():
    d = synth.Dims(grid_h=20, grid_w=24, text_len=30)
    A, ids = synth.blob_scores(d, 5, n_delta=(3, 5))
    for r in (0, 1, 2):
        m, idx = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, r)
        m0, _ = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
        ref = ndi.binary_dilation(m0.reshape(d.grid_h, d.grid_w).astype(bool),
                                  structure=np.ones((2 * r + 1, 2 * r + 1), bool)) if r else \
            m0.reshape(d.grid_h, d.grid_w).astype(bool)
        assert np.array_equal(m.reshape(d.grid_h, d.grid_w).astype(bool), ref)
        assert np.array_equal(idx, np.flatnonzero(m))
        assert np.all(np.diff(idx) > 0)
    # order-free, idempotent union
    m1, _ = O.localize_mask(A, ids, d.grid_h, d.grid_w)
    m2, _ = O.localize_mask(A, list(ids[::-1]) + list(ids), d.grid_h, d.grid_w)
    assert np.array_equal(m1, m2)
    # the union contains each token's own region
    for j in ids:
        mj, _ = O.localize_mask(A, [j], d.grid_h, d.grid_w)
        assert np.all(m1 >= mj)


def test_localize_mean_over_slices():
    gh, gw, M = 4, 4, 3
    base = rng(4).uniform(0, 1, (gh * gw, M)).astype(np.float32)
    # two slices whose float32 mean is exactly `base` (x + x = 2x is exact)
    A2 = np.stack([base, base])
    for j in range(M):
        a, _ = O.localize_mask(base[None], [j], gh, gw, 0.5, 0)
        b, _ = O.localize_mask(A2, [j], gh, gw, 0.5, 0)
        assert np.array_equal(a, b)
    # a column split as 0 and 2x across two slices is the same mean
    A2b = np.stack([np.zeros_like(base), base * 2])
    a, _ = O.localize_mask(base[None], [0, 1, 2], gh, gw)
    b, _ = O.localize_mask(A2b, [0, 1, 2], gh, gw)
    assert np.array_equal(a, b)


def test_localize_indicator_scores_reproduce_ellipses():
    d = synth.Dims(grid_h=32, grid_w=32)
    blobs = synth.ellipse_blobs(d, 7, 0.2)
    A, ids = synth.indicator_scores(d, blobs, 7)
    m, idx = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
    union = np.any(np.stack(blobs), axis=0)
    assert np.array_equal(m.astype(bool), union)
    assert abs(union.mean() - 0.2) <= 0.005 + 1.0 / d.tokens


# ---------------------------------------------------------- timestep embed
def test_timestep_embedding_closed_form():
    e0 = O.timestep_embedding(0.0, 256)
    assert np.array_equal(e0, np.concatenate([np.ones(128), np.zeros(128)]))
    e1 = O.timestep_embedding(1.0, 256)
    assert e1[0] == math.cos(1.0) and e1[128] == math.sin(1.0)
    w_last = 10000.0 ** (-127 / 128)
    assert abs(e1[127] - math.cos(w_last)) < 1e-15
    e = O.timestep_embedding(500.0, 8)
    for k in range(4):
        w = math.exp(-math.log(10000.0) * k / 4)
        assert abs(e[k] - math.cos(500 * w)) < 1e-12
        assert abs(e[4 + k] - math.sin(500 * w)) < 1e-12


def test_t_embed_and_t_block_against_torch_modules():
    d = synth.TINY
    w = synth.make_weights(d, 31)
    _, G, _ = weights64(w)
    t = 437.0
    f = torch.from_numpy(O.timestep_embedding(t, d.freq_dim))
    h = F.linear(f, torch.from_numpy(G["W_t1"]), torch.from_numpy(G["b_t1"]))
    h = F.linear(F.silu(h), torch.from_numpy(G["W_t2"]), torch.from_numpy(G["b_t2"]))
    assert np.allclose(O.t_embed(t, G), h.numpy(), rtol=0, atol=1e-13)
    tb = F.linear(F.silu(h), torch.from_numpy(G["W_tb"]), torch.from_numpy(G["b_tb"]))
    assert np.allclose(O.t_block(h.numpy(), G), tb.numpy().reshape(6, -1), rtol=0, atol=1e-13)


# ------------------------------------------------------- patches and final
def test_patch_embed_matches_conv2d():
    d = synth.Dims(hidden=32, heads=2, mlp=64, grid_h=3, grid_w=5)
    w = synth.make_weights(d, 41)
    _, G, pos = weights64(w)
    lat = rng(41).standard_normal(d.latent_shape)
    rows = np.array([0, 4, 7, 14])
    got = O.patch_embed(lat, rows, G, pos, d.patch)
    conv = F.conv2d(torch.from_numpy(lat)[None], torch.from_numpy(G["W_e"]).view(
        d.hidden, d.in_ch, d.patch, d.patch), torch.from_numpy(G["b_e"]), stride=d.patch)
    ref = conv[0].reshape(d.hidden, -1).T.numpy() + pos
    assert np.allclose(got, ref[rows], rtol=0, atol=1e-13)


def test_unpatchify_hand_indices():
    gh, gw, p, C = 2, 3, 2, 8
    out = np.arange(gh * gw * p * p * C, dtype=float).reshape(gh * gw, p * p * C)
    img = O.unpatchify(out, gh, gw, p)
    assert img.shape == (C, gh * p, gw * p)
    # token n = gy*gw + gx, sub-position (py, px), channel c -> out[n][(py*p+px)*C + c]
    for (gy, gx, py, px, c) in [(0, 0, 0, 0, 0), (1, 2, 1, 1, 7), (0, 1, 1, 0, 3), (1, 0, 0, 1, 5)]:
        n = gy * gw + gx
        assert img[c, gy * p + py, gx * p + px] == out[n, (py * p + px) * C + c]
    lat = rng(5).standard_normal((4, 6, 10))
    P = O.patchify(lat, 2)
    # (c, py, px) ordering of a patch vector: token (gy=1, gx=2) of a 3x5 grid
    assert np.array_equal(P[1 * 5 + 2], lat[:, 2:4, 4:6].reshape(-1))


def test_final_layer_zero_weight_gives_bias_image():
    d = synth.Dims(hidden=32, heads=2, mlp=64, grid_h=3, grid_w=4)
    w = synth.make_weights(d, 51)
    _, G, _ = weights64(w)
    G["W_f"] = np.zeros_like(G["W_f"])
    H = rng(51).standard_normal((d.tokens, d.hidden))
    eps = O.final_layer(H, rng(52).standard_normal(d.hidden), G, d.grid_h, d.grid_w, d.patch,
                        d.in_ch)
    for c in range(d.in_ch):
        for y in range(d.grid_h * 2):
            for x in range(d.grid_w * 2):
                assert eps[c, y, x] == G["b_f"][((y % 2) * 2 + (x % 2)) * d.out_ch + c]


def test_final_layer_matches_torch_composition():
    d = synth.Dims(hidden=32, heads=2, mlp=64, grid_h=3, grid_w=4)
    w = synth.make_weights(d, 53)
    _, G, _ = weights64(w)
    H = rng(53).standard_normal((d.tokens, d.hidden))
    temb = rng(54).standard_normal(d.hidden)
    got = O.final_layer(H, temb, G, d.grid_h, d.grid_w, d.patch, d.in_ch)
    t = torch.from_numpy
    y = F.layer_norm(t(H), (d.hidden,), eps=1e-6)
    y = y * (1 + t(G["table_f"][1] + temb)) + t(G["table_f"][0] + temb)
    out = F.linear(y, t(G["W_f"]), t(G["b_f"]))
    # channel-fastest patch outputs -> image via pixel_shuffle on (c, py, px) order
    out = out.view(d.grid_h, d.grid_w, 2, 2, d.out_ch).permute(4, 2, 3, 0, 1)
    img = F.pixel_shuffle(out.reshape(1, d.out_ch * 4, d.grid_h, d.grid_w), 2)[0]
    assert np.allclose(got, img[:d.in_ch].numpy(), rtol=0, atol=1e-12)


# ------------------------------------------------------------------- DDIM
def test_ddim_closed_forms():
    r = rng(61)
    x = r.standard_normal((4, 6, 6))
    eps0 = np.zeros_like(x)
    assert np.allclose(O.ddim_update(x, eps0, 0.3, 0.6), x * math.sqrt(0.6 / 0.3))
    x0, e = r.standard_normal(x.shape), r.standard_normal(x.shape)
    xt = math.sqrt(0.25) * x0 + math.sqrt(0.75) * e
    assert np.allclose(O.ddim_update(xt, e, 0.25, 0.81), 0.9 * x0 + math.sqrt(0.19) * e)
    assert np.allclose(O.ddim_update(xt, e, 0.25, 1.0), x0)


def test_ddim_tables():
    tv, ab = synth.ddim_tables(20)
    assert tv[0] == 999 and tv[-1] == 0 and len(ab) == 21 and ab[-1] == 1.0
    assert np.all(np.diff(ab) > 0)


# ------------------------------------------------------------------- step
def _step_problem(d, seed):
    w = synth.make_weights(d, seed)
    layers, G, pos = weights64(w)
    ctx = O.to64(synth.make_text(d, seed))
    tkv = [O.text_kv(ctx, L) for L in layers]
    cache = [dict(zip("HKV", (O.to64(a) for a in synth.make_cache_slice(d, seed, 0, l, 0))))
             for l in range(d.layers)]
    lat = O.to64(synth.make_latent(d, seed))
    tv, ab = synth.ddim_tables(d.timesteps)
    return layers, G, pos, tkv, cache, lat, tv.astype(float), ab.astype(float)


def _run(d, prob, mode, idx, t=1, cache=None):
    layers, G, pos, tkv, c0, lat, tv, ab = prob
    return O.step(G, layers, pos, lat, t, mode, idx, c0 if cache is None else cache, tkv, tv, ab,
                  d.heads, d.grid_h, d.grid_w, d.patch, d.in_ch)


def test_step_reuse_zero_final_weight_closed_form():
    d = synth.TINY
    prob = _step_problem(d, 71)
    prob[1]["W_f"] = np.zeros_like(prob[1]["W_f"])
    lat = prob[5]
    ab = prob[7]
    x_next, eps, newc = _run(d, prob, O.MODE_REUSE, None, t=2)
    bf = prob[1]["b_f"]
    want_eps = np.empty_like(lat)
    for c in range(d.in_ch):
        for y in range(lat.shape[1]):
            for x in range(lat.shape[2]):
                want_eps[c, y, x] = bf[((y % 2) * 2 + (x % 2)) * d.out_ch + c]
    assert np.array_equal(eps, want_eps)
    x0 = (lat - math.sqrt(1 - ab[2]) * want_eps) / math.sqrt(ab[2])
    assert np.allclose(x_next, math.sqrt(ab[3]) * x0 + math.sqrt(1 - ab[3]) * want_eps)
    for l in range(d.layers):
        for k in "HKV":
            assert np.array_equal(newc[l][k], prob[4][l][k])


def test_step_sparse_all_dirty_equals_dense():
    d = synth.TINY
    prob = _step_problem(d, 72)
    a = _run(d, prob, O.MODE_DENSE, None)
    b = _run(d, prob, O.MODE_SPARSE, np.arange(d.tokens))
    assert np.array_equal(a[0], b[0])
    for l in range(d.layers):
        for k in "HKV":
            assert np.array_equal(a[2][l][k], b[2][l][k])


def test_step_dense_cache_is_a_fixed_point_of_sparse():
    d = synth.TINY
    prob = _step_problem(d, 73)
    xa, ea, ca = _run(d, prob, O.MODE_DENSE, None)
    for idx in ([0, 5], [3, 4, 7, 8, 12]):
        xb, eb, cb = _run(d, prob, O.MODE_SPARSE, np.array(idx), cache=ca)
        assert np.allclose(xb, xa, rtol=0, atol=1e-12)
        for l in range(d.layers):
            assert np.allclose(cb[l]["H"], ca[l]["H"], rtol=0, atol=1e-12)
    # REUSE on the dense cache gives the dense step's latent too
    xc, _, _ = _run(d, prob, O.MODE_REUSE, None, cache=ca)
    assert np.allclose(xc, xa, rtol=0, atol=1e-12)


def test_step_sparse_leaves_clean_rows_of_every_layer():
    d = synth.TINY
    prob = _step_problem(d, 74)
    idx = np.array([1, 2, 9])
    _, _, c = _run(d, prob, O.MODE_SPARSE, idx)
    clean = np.setdiff1d(np.arange(d.tokens), idx)
    for l in range(d.layers):
        for k in "HKV":
            assert np.array_equal(c[l][k][clean], prob[4][l][k][clean])
            assert not np.allclose(c[l][k][idx], prob[4][l][k][idx])


# -------------------------------------------------------------- schedules
def test_eq2_golden():
    for ln in open(os.path.join(GOLDEN, "eq2_reuse_cutoff.txt")):
        if ln.startswith("#") or not ln.strip():
            continue
        T, s, tau, want = ln.split()
        assert O.reuse_cutoff(float(s), float(tau), int(T)) == int(want)
        sched = O.schedule_eq2(float(s), float(tau), int(T))
        assert int((sched == O.MODE_REUSE).sum()) == int(want)
        assert np.all(sched[:int(want)] == O.MODE_REUSE)


def test_eq1_cosine():
    e = rng(8).standard_normal(16)
    assert abs(O.cosine_similarity(e, 3 * e) - 1) < 1e-15
    assert abs(O.cosine_similarity(e, -e) + 1) < 1e-15
    f = np.zeros(16)
    f[0], e2 = 1.0, np.zeros(16)
    e2[1] = 2.0
    assert O.cosine_similarity(f, e2) == 0.0


def test_turn_k_table():
    table = {1.0: 2, 0.8: 2, 0.76: 2, 0.75: 4, 0.6: 4, 0.5: 6, 0.3: 6, 0.25: 8, 0.0: 8}
    for s, k in table.items():
        assert O.k_from_similarity(s) == k
    sch = O.schedule_first_k_dense(6, 20)
    assert sch.tolist() == [0] * 6 + [1] * 14
