"""Pins of the oracle's localisation scores from the model's own
cross-attention (Section 3.2): each fixes a value by something other than the
oracle's own formula (a library softmax, the attention output computed by a
different routine, closed forms, a brute-force loop, invariants)."""
import math

import numpy as np
import torch

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import rng, small_problem, weights64

TINY = synth.TINY


def test_cross_attention_maps_library_softmax_and_rows():
    p = small_problem(TINY, 81)
    L = p["layers"][0]
    tk, tv = O.text_kv(p["ctx"], L)
    maps = O.cross_attention_maps(p["x"], tk, L, TINY.heads)
    assert maps.shape == (TINY.heads, TINY.tokens, TINY.text_len)
    assert np.allclose(maps.sum(-1), 1.0, atol=1e-13)
    q = O.linear(p["x"], L["W_xq"], L["b_xq"])
    dh = TINY.head_dim
    for h in range(TINY.heads):
        c = slice(h * dh, (h + 1) * dh)
        s = torch.from_numpy(q[:, c] @ tk[:, c].T / math.sqrt(dh))
        assert np.allclose(maps[h], torch.softmax(s, -1).numpy(), rtol=0, atol=1e-14)


def test_cross_attention_maps_reproduce_the_attention_output():
    p = small_problem(TINY, 82)
    L = p["layers"][1]
    tk, tv = O.text_kv(p["ctx"], L)
    maps = O.cross_attention_maps(p["x"], tk, L, TINY.heads)
    dh = TINY.head_dim
    o = np.concatenate([maps[h] @ tv[:, h * dh:(h + 1) * dh] for h in range(TINY.heads)], 1)
    want = O.cross_attention(p["x"], tk, tv, L, TINY.heads)
    assert np.allclose(O.linear(o, L["W_xo"], L["b_xo"]), want, rtol=0, atol=1e-12)


def test_cross_attention_maps_brute_force_entry():
    p = small_problem(TINY, 83)
    L = p["layers"][0]
    tk, _ = O.text_kv(p["ctx"], L)
    maps = O.cross_attention_maps(p["x"], tk, L, TINY.heads)
    q = O.linear(p["x"], L["W_xq"], L["b_xq"])
    dh = TINY.head_dim
    for h, i, j in [(0, 0, 0), (3, 15, 7), (2, 9, 4)]:
        num = [math.exp(sum(q[i, h * dh + e] * tk[m, h * dh + e] for e in range(dh)) / math.sqrt(dh))
               for m in range(TINY.text_len)]
        assert abs(maps[h, i, j] - num[j] / sum(num)) < 1e-14


def _problem(d, seed):
    w = synth.make_weights(d, seed)
    layers, G, pos = weights64(w)
    ctx = O.to64(synth.make_text(d, seed))
    tkv = [O.text_kv(ctx, L) for L in layers]
    cache = [dict(zip("HKV", (O.to64(a) for a in synth.make_cache_slice(d, seed, 0, l, 0))))
             for l in range(d.layers)]
    lat = O.to64(synth.make_latent(d, seed))
    tv, ab = synth.ddim_tables(d.timesteps)
    return layers, G, pos, tkv, cache, lat, tv.astype(float), ab.astype(float)


def _capture(d, prob, ids, t=1):
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    return O.step_capture(G, layers, pos, lat, t, cache, tkv, tv, ab, d.heads, d.grid_h, d.grid_w,
                          d.patch, d.in_ch, ids, d.text_len)


def test_step_capture_is_the_dense_step_and_rows_sum_to_one():
    d = TINY
    prob = _problem(d, 84)
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    x_next, eps, newc, scores = _capture(d, prob, np.arange(d.text_len))
    ref = O.step(G, layers, pos, lat, 1, O.MODE_DENSE, None, cache, tkv, tv, ab, d.heads,
                 d.grid_h, d.grid_w, d.patch, d.in_ch)
    assert np.array_equal(x_next, ref[0]) and np.array_equal(eps, ref[1])
    for l in range(d.layers):
        for k in "HKV":
            assert np.array_equal(newc[l][k], ref[2][l][k])
    # the mean over heads and layers of probability rows is a probability row
    assert np.allclose(scores.sum(1), 1.0, atol=1e-12)
    assert np.all(scores > 0)


def test_step_capture_only_delta_columns_and_uniform_closed_form():
    d = TINY
    prob = _problem(d, 85)
    ids = np.array([1, 6])
    scores = _capture(d, prob, ids)[3]
    other = np.setdiff1d(np.arange(d.text_len), ids)
    assert np.all(scores[:, other] == 0) and np.all(scores[:, ids] > 0)
    # a zero query projection makes every head attend uniformly: 1 / M
    for L in prob[0]:
        L["W_xq"] = np.zeros_like(L["W_xq"])
        L["b_xq"] = np.zeros_like(L["b_xq"])
    scores = _capture(d, prob, ids)[3]
    assert np.allclose(scores[:, ids], 1.0 / d.text_len, rtol=0, atol=1e-15)
