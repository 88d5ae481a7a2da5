"""Pins of the oracle's localisation scores taken from the cached states of
the previous turn (Section 3.2's a_j, aggregated over heads and layers, for a
turn that recomputes nothing densely).  Each pin fixes the value by something
other than the oracle's own formula: a brute-force loop over layers, heads
and text tokens with torch-built inputs, a closed form, the dense capture
step (an independent code path) on a model whose self-attention gate is
zero, and which cached states the scores may depend on."""
import math

import numpy as np
import torch
import torch.nn.functional as F

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import weights64

D = synth.Dims(hidden=64, heads=4, mlp=128, layers=3, grid_h=4, grid_w=5, text_len=8,
               timesteps=3, freq_dim=32)


def _problem(d, seed, t=1):
    w = synth.make_weights(d, seed)
    layers, G, pos = weights64(w)
    ctx = O.to64(synth.make_text(d, seed))
    tkv = [O.text_kv(ctx, L) for L in layers]
    cache = [dict(zip("HKV", (O.to64(a) for a in synth.make_cache_slice(d, seed, 0, l, t))))
             for l in range(d.layers)]
    lat = O.to64(synth.make_latent(d, seed))
    tv, ab = synth.ddim_tables(d.timesteps)
    return dict(layers=layers, G=G, pos=pos, ctx=ctx, tkv=tkv, cache=cache, lat=lat,
                tv=tv.astype(float), ab=ab.astype(float))


def _scores(d, p, ids, cache=None, lat=None):
    return O.cached_localization_scores(p["G"], p["layers"], p["pos"],
                                        p["lat"] if lat is None else lat,
                                        p["cache"] if cache is None else cache, p["tkv"],
                                        d.heads, d.grid_h, d.grid_w, d.patch, ids, d.text_len)


def test_rows_are_probabilities_and_only_delta_columns_are_written():
    p = _problem(D, 91)
    all_ids = np.arange(D.text_len)
    s = _scores(D, p, all_ids)
    assert np.allclose(s.sum(1), 1.0, atol=1e-12) and np.all(s > 0)
    ids = np.array([0, 5])
    s2 = _scores(D, p, ids)
    other = np.setdiff1d(all_ids, ids)
    assert np.all(s2[:, other] == 0)
    assert np.array_equal(s2[:, ids], s[:, ids])


def test_zero_query_projection_gives_uniform_scores():
    p = _problem(D, 92)
    for L in p["layers"]:
        L["W_xq"] = np.zeros_like(L["W_xq"])
        L["b_xq"] = np.zeros_like(L["b_xq"])
    ids = np.array([2, 7])
    assert np.allclose(_scores(D, p, ids)[:, ids], 1.0 / D.text_len, rtol=0, atol=1e-15)


def test_brute_force_entries():
    p = _problem(D, 93)
    t = torch.from_numpy
    # the state entering block 0: patch embedding (a strided convolution) + pos
    conv = F.conv2d(t(p["lat"])[None], t(p["G"]["W_e"]).view(D.hidden, D.in_ch, D.patch,
                                                              D.patch),
                    t(p["G"]["b_e"]), stride=D.patch)
    h0 = (conv[0].reshape(D.hidden, -1).T + t(p["pos"])).numpy()
    dh = D.head_dim
    ids = np.array([1, 6])
    s = _scores(D, p, ids)
    for i, j in [(0, 1), (7, 6), (19, 1), (12, 6)]:
        acc = 0.0
        for l, L in enumerate(p["layers"]):
            x = h0[i] if l == 0 else p["cache"][l - 1]["H"][i]
            q = F.linear(t(x), t(L["W_xq"]), t(L["b_xq"])).numpy()
            k = F.linear(t(p["ctx"]), t(L["W_xkv"]), t(L["b_xkv"])).numpy()[:, :D.hidden]
            for h in range(D.heads):
                e = [math.exp(sum(q[h * dh + c] * k[m, h * dh + c] for c in range(dh)) /
                              math.sqrt(dh)) for m in range(D.text_len)]
                acc += e[j] / sum(e)
        assert abs(s[i, j] - acc / (D.layers * D.heads)) < 1e-13


def test_equals_the_dense_capture_when_the_self_attention_gate_is_zero():
    # with gate_msa = 0 the cross-attention of block l reads exactly the
    # block's input H^l, so the scores the dense step captures equal the
    # scores computed afterwards from the cache that step wrote
    p = _problem(D, 94)
    h = D.hidden
    p["G"]["W_tb"][2 * h:3 * h] = 0.0
    p["G"]["b_tb"][2 * h:3 * h] = 0.0
    for L in p["layers"]:
        L["table"][2] = 0.0
    ids = np.array([0, 3, 7])
    _, _, newc, cap = O.step_capture(p["G"], p["layers"], p["pos"], p["lat"], 1, p["cache"],
                                     p["tkv"], p["tv"], p["ab"], D.heads, D.grid_h, D.grid_w,
                                     D.patch, D.in_ch, ids, D.text_len)
    got = _scores(D, p, ids, cache=newc)
    assert np.array_equal(got, cap)


def test_depends_on_the_latent_and_block_inputs_only():
    p = _problem(D, 95)
    ids = np.array([4])
    base = _scores(D, p, ids)
    # the last block's output is no block's input: changing it changes nothing
    c = [dict(x) for x in p["cache"]]
    c[-1] = dict(c[-1], H=c[-1]["H"] + 1.0)
    assert np.array_equal(_scores(D, p, ids, cache=c), base)
    # cached K, V of the self-attention are not read either
    c = [dict(x, K=x["K"] * 2, V=-x["V"]) for x in p["cache"]]
    assert np.array_equal(_scores(D, p, ids, cache=c), base)
    # the output of block 0 (input of block 1) and the latent (input of block 0) are
    c = [dict(x) for x in p["cache"]]
    c[0] = dict(c[0], H=c[0]["H"] + 1.0)
    assert not np.allclose(_scores(D, p, ids, cache=c), base)
    assert not np.allclose(_scores(D, p, ids, lat=p["lat"] * 0.5), base)
