"""Pins of how the oracle's denoising step wires the timestep conditioning
(reading A11 of the backbone, adaLN-single, and the sampler; Section 3.3 for
the DENSE / SPARSE / REUSE modes of a step).

With every block matrix zero, a block's update no longer depends on its
input: the self-attention of identical value rows returns b_v, the text
cross-attention of identical key rows returns b_xv, and the MLP returns
gelu(b_1).  After the zero projections only the biases survive, so block l
adds  g1_l * b_o,l + b_xo,l + g2_l * b_2,l  with the gates
g1_l = table_l[2] + tb[2], g2_l = table_l[5] + tb[5], where
tb = W_tb silu(temb) + b_tb and temb = MLP(sinusoid(t_values[t])) of the
step's own timestep.  The final layer modulates with table_f + temb.  The
expected values below are composed from those facts with torch library
calls; none of the oracle's step, block or final-layer code is used.

Each test fails if the step drops tb from the modulation, takes the
timestep value of another step, or hands the final layer tb (or nothing)
instead of temb.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import weights64

T = torch.from_numpy


def _problem(d, seed):
    w = synth.make_weights(d, seed)
    layers, G, pos = weights64(w)
    for L in layers:  # zero every block matrix, keep biases and tables
        for k in synth.LAYER_MATS:
            L[k] = np.zeros_like(L[k])
    ctx = O.to64(synth.make_text(d, seed))
    tkv = [O.text_kv(ctx, L) for L in layers]
    cache = [dict(zip("HKV", (O.to64(a) for a in synth.make_cache_slice(d, seed, 0, l, 0))))
             for l in range(d.layers)]
    lat = O.to64(synth.make_latent(d, seed))
    tv, ab = synth.ddim_tables(d.timesteps)
    return layers, G, pos, tkv, cache, lat, tv.astype(float), ab.astype(float)


def _temb_tb(G, t_value, d):
    """Timestep embedding and adaLN-single vector, from torch modules."""
    half = d.freq_dim // 2
    k = torch.arange(half, dtype=torch.float64)
    a = float(t_value) * torch.exp(-math.log(10000.0) * k / half)
    f = torch.cat([torch.cos(a), torch.sin(a)])
    h = F.linear(F.silu(F.linear(f, T(G["W_t1"]), T(G["b_t1"]))), T(G["W_t2"]), T(G["b_t2"]))
    tb = F.linear(F.silu(h), T(G["W_tb"]), T(G["b_tb"])).reshape(6, d.hidden)
    return h, tb


def _embedded(G, pos, lat, d):
    """Patch embedding of every token (a strided convolution) plus pos."""
    conv = F.conv2d(T(lat)[None], T(G["W_e"]).view(d.hidden, d.in_ch, d.patch, d.patch),
                    T(G["b_e"]), stride=d.patch)
    return conv[0].reshape(d.hidden, -1).T + T(pos)


def _block_update(L, tb):
    g1 = T(L["table"][2]) + tb[2]
    g2 = T(L["table"][5]) + tb[5]
    return g1 * T(L["b_o"]) + T(L["b_xo"]) + g2 * T(L["b_2"])


def _final_eps(G, H, temb, d):
    y = F.layer_norm(H, (d.hidden,), eps=1e-6)
    y = y * (1 + T(G["table_f"][1]) + temb) + T(G["table_f"][0]) + temb
    out = F.linear(y, T(G["W_f"]), T(G["b_f"]))
    out = out.view(d.grid_h, d.grid_w, d.patch, d.patch, d.out_ch).permute(4, 2, 3, 0, 1)
    img = F.pixel_shuffle(out.reshape(1, d.out_ch * d.patch ** 2, d.grid_h, d.grid_w), d.patch)[0]
    return img[:d.in_ch].numpy()


def _ddim(x, eps, ab_t, ab_n):
    x0 = (x - math.sqrt(1 - ab_t) * eps) / math.sqrt(ab_t)
    return math.sqrt(ab_n) * x0 + math.sqrt(1 - ab_n) * eps


def _run(d, prob, mode, idx, t):
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    return O.step(G, layers, pos, lat, t, mode, idx, cache, tkv, tv, ab, d.heads, d.grid_h,
                  d.grid_w, d.patch, d.in_ch)


def _close(a, b):
    a, b = np.asarray(a, float), np.asarray(b, float)
    assert np.allclose(a, b, rtol=1e-12, atol=1e-12), float(np.abs(a - b).max())


D = synth.Dims(hidden=64, heads=4, mlp=128, layers=3, grid_h=4, grid_w=6, text_len=8,
               timesteps=5, freq_dim=32)


@pytest.mark.parametrize("t", [0, 2, 4])
def test_dense_step_conditioning_closed_form(t):
    prob = _problem(D, 81)
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    temb, tb = _temb_tb(G, tv[t], D)
    x = _embedded(G, pos, lat, D)
    Hs = []
    for L in layers:
        x = x + _block_update(L, tb)
        Hs.append(x.numpy())
    eps = _final_eps(G, x, temb, D)
    x_next, eps_o, newc = _run(D, prob, O.MODE_DENSE, None, t)
    _close(eps_o, eps)
    _close(x_next, _ddim(lat, eps, ab[t], ab[t + 1]))
    for l, L in enumerate(layers):
        _close(newc[l]["H"], Hs[l])
        # K, V of every token are the biases of the zero projection
        h = D.hidden
        _close(newc[l]["K"], np.broadcast_to(L["b_qkv"][h:2 * h], (D.tokens, h)))
        _close(newc[l]["V"], np.broadcast_to(L["b_qkv"][2 * h:], (D.tokens, h)))


@pytest.mark.parametrize("t", [1, 3])
def test_sparse_step_conditioning_closed_form(t):
    prob = _problem(D, 82)
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    idx = np.array([0, 5, 6, 13, 23])
    clean = np.setdiff1d(np.arange(D.tokens), idx)
    temb, tb = _temb_tb(G, tv[t], D)
    x = _embedded(G, pos, lat, D)[idx]
    for L in layers:
        x = x + _block_update(L, tb)
    H = T(cache[-1]["H"]).clone()
    H[idx] = x
    eps = _final_eps(G, H, temb, D)
    x_next, eps_o, newc = _run(D, prob, O.MODE_SPARSE, idx, t)
    _close(eps_o, eps)
    _close(x_next, _ddim(lat, eps, ab[t], ab[t + 1]))
    _close(newc[-1]["H"][idx], x.numpy())
    assert np.array_equal(newc[-1]["H"][clean], cache[-1]["H"][clean])


@pytest.mark.parametrize("t", [0, 3])
def test_reuse_step_final_layer_takes_the_steps_own_embedding(t):
    prob = _problem(D, 83)
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    temb, _ = _temb_tb(G, tv[t], D)
    eps = _final_eps(G, T(cache[-1]["H"]), temb, D)
    x_next, eps_o, _ = _run(D, prob, O.MODE_REUSE, None, t)
    _close(eps_o, eps)
    _close(x_next, _ddim(lat, eps, ab[t], ab[t + 1]))


def test_neighbouring_timesteps_give_different_results():
    # the pins above are only sensitive to the timestep if the conditioning
    # actually varies between steps on this problem
    prob = _problem(D, 84)
    G, tv = prob[1], prob[6]
    a, ta = _temb_tb(G, tv[1], D)
    b, tb_ = _temb_tb(G, tv[2], D)
    assert float((a - b).abs().max()) > 1e-3 and float((ta - tb_).abs().max()) > 1e-3
    assert float(ta[2].abs().max()) > 1e-3 and float(ta[5].abs().max()) > 1e-3


def test_capture_step_conditioning_and_uniform_scores():
    # zero text-key projection: every text key is b_xk, so each delta token
    # gets probability 1 / M in every head and layer
    prob = _problem(D, 85)
    layers, G, pos, tkv, cache, lat, tv, ab = prob
    t = 2
    temb, tb = _temb_tb(G, tv[t], D)
    x = _embedded(G, pos, lat, D)
    for L in layers:
        x = x + _block_update(L, tb)
    eps = _final_eps(G, x, temb, D)
    ids = [1, 6]
    x_next, eps_o, newc, scores = O.step_capture(G, layers, pos, lat, t, cache, tkv, tv, ab,
                                                D.heads, D.grid_h, D.grid_w, D.patch, D.in_ch,
                                                ids, D.text_len)
    _close(eps_o, eps)
    _close(x_next, _ddim(lat, eps, ab[t], ab[t + 1]))
    want = np.zeros((D.tokens, D.text_len))
    want[:, ids] = 1.0 / D.text_len
    _close(scores, want)
