"""Pins of the oracle's block arithmetic (CPU only).

Each test fixes a value by something other than the oracle itself: a library
routine that implements the same textbook operation, a closed form, a
brute-force scalar loop, or an invariant that a dropped term, a wrong sign, a
wrong index or a transposed operand would break.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import rng, small_problem

TINY = synth.TINY


# ------------------------------------------------------------------ pieces
def test_layer_norm_hand_row_and_library():
    x = np.array([[1.0, 2.0, 3.0, 4.0]])
    want = (x - 2.5) / math.sqrt(1.25 + 1e-6)          # mean 2.5, biased var 1.25
    assert np.allclose(O.layer_norm(x), want, rtol=0, atol=1e-15)
    y = rng(1).standard_normal((7, 33)) * 3 + 1
    ref = F.layer_norm(torch.from_numpy(y), (33,), eps=1e-6).numpy()
    assert np.allclose(O.layer_norm(y), ref, rtol=0, atol=1e-12)
    z = O.layer_norm(y)
    assert np.allclose(z.mean(1), 0, atol=1e-13)
    assert np.allclose(z.var(1), 1, atol=1e-5)


def test_gelu_tanh_points_and_library():
    z = np.linspace(-8, 8, 101)
    ref = F.gelu(torch.from_numpy(z), approximate="tanh").numpy()
    assert np.allclose(O.gelu_tanh(z), ref, rtol=0, atol=1e-12)
    assert O.gelu_tanh(np.array(0.0)) == 0.0
    assert abs(O.gelu_tanh(np.array(20.0)) - 20.0) < 1e-12
    assert abs(O.gelu_tanh(np.array(-20.0))) < 1e-12
    assert abs(O.gelu_tanh(np.array(1.0)) - 0.8411919906082768) < 1e-9


def test_modulate_closed_form():
    y = rng(2).standard_normal((3, 5))
    sh, sc = rng(3).standard_normal(5), rng(4).standard_normal(5)
    assert np.allclose(O.modulate(np.zeros_like(y), sh, sc), sh)
    assert np.allclose(O.modulate(y, sh, -np.ones(5)), sh)
    assert np.allclose(O.modulate(y, np.zeros(5), np.zeros(5)), y)


def test_softmax_rows():
    s = rng(5).standard_normal((6, 9)) * 4
    p = O.softmax(s)
    assert np.allclose(p.sum(1), 1, atol=1e-14)
    assert np.allclose(O.softmax(np.array([0.0, math.log(2.0)])), [1 / 3, 2 / 3])


def test_attention_matches_sdpa():
    r = rng(6)
    h, dh = 4, 16
    q = r.standard_normal((10, h * dh))
    k = r.standard_normal((23, h * dh))
    v = r.standard_normal((23, h * dh))
    got = O.multihead_attention(q, k, v, h)
    tq = torch.from_numpy(q).view(10, h, dh).transpose(0, 1)
    tk = torch.from_numpy(k).view(23, h, dh).transpose(0, 1)
    tv = torch.from_numpy(v).view(23, h, dh).transpose(0, 1)
    ref = F.scaled_dot_product_attention(tq, tk, tv).transpose(0, 1).reshape(10, h * dh)
    assert np.allclose(got, ref.numpy(), rtol=0, atol=1e-12)


def test_attention_special_cases():
    r = rng(7)
    h, dh = 2, 8
    v = r.standard_normal((5, h * dh))
    k = r.standard_normal((5, h * dh))
    # zero query: uniform average of the values
    out = O.multihead_attention(np.zeros((3, h * dh)), k, v, h)
    assert np.allclose(out, np.tile(v.mean(0), (3, 1)))
    # one key: that key's value
    out = O.multihead_attention(r.standard_normal((2, h * dh)), k[:1], v[:1], h)
    assert np.allclose(out, np.tile(v[0], (2, 1)))
    # heads are contiguous column blocks: head 0 selects key 1, head 1 key 3
    q = np.zeros((1, h * dh))
    kk = np.zeros((5, h * dh))
    q[0, 0] = 1.0
    q[0, dh] = 1.0
    kk[1, 0] = 200.0
    kk[3, dh] = 200.0
    out = O.multihead_attention(q, kk, v, h)
    assert np.allclose(out[0, :dh], v[1, :dh])
    assert np.allclose(out[0, dh:], v[3, dh:])
    # scale 1/sqrt(dh): two keys whose scores differ by sqrt(dh)*ln 3
    q = np.zeros((1, dh))
    k2 = np.zeros((2, dh))
    q[0, 0] = 1.0
    k2[0, 0] = math.sqrt(dh) * math.log(3.0)
    v2 = np.array([[1.0] * dh, [0.0] * dh])
    out = O.multihead_attention(q, k2, v2, 1)
    assert np.allclose(out, 0.75)


# ------------------------------------------------------------------- blocks
def _zero_mats(layers):
    L = dict(layers)
    for k in L:
        if k.startswith("W_"):
            L[k] = np.zeros_like(L[k])
    return L


def test_dense_block_zero_weights_closed_form():
    p = small_problem(TINY, 11)
    L = _zero_mats(p["layers"][0])
    tkv = O.text_kv(p["ctx"], L)
    x = p["x"]
    out, K, V = O.dense_block(x, L, p["m6"], tkv, TINY.heads)
    g1, g2 = p["m6"][2], p["m6"][5]
    want = x + g1 * L["b_o"] + L["b_xo"] + g2 * L["b_2"]
    assert np.allclose(out, want, rtol=0, atol=1e-14)
    d = TINY.hidden
    assert np.allclose(K, np.tile(L["b_qkv"][d:2 * d], (x.shape[0], 1)))
    assert np.allclose(V, np.tile(L["b_qkv"][2 * d:], (x.shape[0], 1)))


def test_dense_block_zero_gates_keep_only_cross_attention():
    p = small_problem(TINY, 12)
    L = p["layers"][0]
    m6 = p["m6"].copy()
    m6[2] = 0.0
    m6[5] = 0.0
    tkv = O.text_kv(p["ctx"], L)
    out, _, _ = O.dense_block(p["x"], L, m6, tkv, TINY.heads)
    # single text token: the cross-attention softmax is 1, output = v' W_xo + b
    ctx1 = p["ctx"][:1]
    tk1, tv1 = O.text_kv(ctx1, L)
    out1, _, _ = O.dense_block(p["x"], L, m6, (tk1, tv1), TINY.heads)
    want1 = p["x"] + np.tile(tv1[0] @ L["W_xo"].T + L["b_xo"], (p["x"].shape[0], 1))
    assert np.allclose(out1, want1, rtol=0, atol=1e-12)
    assert not np.allclose(out, out1)


def _brute_block(x, L, m6, ctx, heads):
    """Scalar-loop dense block written straight from the definitions."""
    N, d = len(x), len(x[0])
    dh = d // heads
    F_ = len(L["b_1"])

    def lin(row, W, b):
        return [sum(row[i] * W[o][i] for i in range(len(row))) + b[o] for o in range(len(b))]

    def ln(row):
        mu = sum(row) / len(row)
        var = sum((a - mu) ** 2 for a in row) / len(row)
        return [(a - mu) / math.sqrt(var + 1e-6) for a in row]

    def attn(qs, ks, vs):
        out = []
        for qr in qs:
            o = [0.0] * d
            for h in range(heads):
                sc = [sum(qr[h * dh + e] * kr[h * dh + e] for e in range(dh)) / math.sqrt(dh)
                      for kr in ks]
                mx = max(sc)
                ex = [math.exp(s - mx) for s in sc]
                z = sum(ex)
                for e in range(dh):
                    o[h * dh + e] = sum(ex[j] / z * vs[j][h * dh + e] for j in range(len(ks)))
            out.append(o)
        return out

    sh1, sc1, g1, sh2, sc2, g2 = m6
    a = [[v * (1 + sc1[i]) + sh1[i] for i, v in enumerate(ln(r))] for r in x]
    qkv = [lin(r, L["W_qkv"], L["b_qkv"]) for r in a]
    q = [r[:d] for r in qkv]
    k = [r[d:2 * d] for r in qkv]
    v = [r[2 * d:] for r in qkv]
    o = attn(q, k, v)
    x1 = [[x[n][i] + g1[i] * y for i, y in enumerate(lin(o[n], L["W_o"], L["b_o"]))]
          for n in range(N)]
    kv = [lin(r, L["W_xkv"], L["b_xkv"]) for r in ctx]
    tk = [r[:d] for r in kv]
    tv = [r[d:] for r in kv]
    qx = [lin(r, L["W_xq"], L["b_xq"]) for r in x1]
    ox = attn(qx, tk, tv)
    x2 = [[x1[n][i] + y for i, y in enumerate(lin(ox[n], L["W_xo"], L["b_xo"]))]
          for n in range(N)]
    x3 = []
    for n in range(N):
        a2 = [v_ * (1 + sc2[i]) + sh2[i] for i, v_ in enumerate(ln(x2[n]))]
        hdn = lin(a2, L["W_1"], L["b_1"])
        u = [0.5 * z * (1 + math.tanh(math.sqrt(2 / math.pi) * (z + 0.044715 * z ** 3)))
             for z in hdn]
        assert len(u) == F_
        y = lin(u, L["W_2"], L["b_2"])
        x3.append([x2[n][i] + g2[i] * y[i] for i in range(d)])
    return x3, k, v


def test_dense_block_brute_force_float64_tiny():
    """hidden 64, 4 heads, 16 tokens, MLP 256, 8 text tokens."""
    p = small_problem(TINY, 13)
    L = p["layers"][0]
    # make the attention non-trivial: scale the weights up from N(0, 0.02)
    L = {k: (v * 10.0 if k.startswith("W_") else v) for k, v in L.items()}
    tolist = lambda a: a.tolist()  # noqa: E731
    bx, bk, bv = _brute_block(tolist(p["x"]), {k: tolist(v) for k, v in L.items()},
                              [tolist(r) for r in p["m6"]], tolist(p["ctx"]), TINY.heads)
    out, K, V = O.dense_block(p["x"], L, p["m6"], O.text_kv(p["ctx"], L), TINY.heads)
    for a, b in ((out, bx), (K, bk), (V, bv)):
        b = np.array(b)
        assert np.linalg.norm(a - b) <= 1e-12 * np.linalg.norm(b)


# ------------------------------------------------- region block invariants
def _region(p, idx, cache=None, x=None):
    L = p["layers"][0]
    x = p["x"] if x is None else x
    idx = np.asarray(idx)
    return O.region_block(x[idx], idx, p["cache"] if cache is None else cache, L, p["m6"],
                          O.text_kv(p["ctx"], L), TINY.heads)


def test_region_all_dirty_equals_dense_exactly():
    p = small_problem(TINY, 21)
    L = p["layers"][0]
    N = TINY.tokens
    dense, K, V = O.dense_block(p["x"], L, p["m6"], O.text_kv(p["ctx"], L), TINY.heads)
    cache, out = _region(p, np.arange(N))
    assert np.array_equal(cache["H"], dense)
    assert np.array_equal(cache["K"], K)
    assert np.array_equal(cache["V"], V)
    assert np.array_equal(out, dense)


def test_region_all_clean_returns_cache_unchanged():
    p = small_problem(TINY, 22)
    cache, out = _region(p, np.array([], dtype=np.int64))
    for k in "HKV":
        assert np.array_equal(cache[k], p["cache"][k])
    assert out.shape == (0, TINY.hidden)


def test_region_dirty_order_invariance():
    p = small_problem(TINY, 23)
    idx = np.array([1, 4, 5, 9, 14])
    c1, o1 = _region(p, idx)
    perm = np.array([3, 0, 4, 2, 1])
    c2, o2 = _region(p, idx[perm])
    for k in "HKV":
        assert np.array_equal(c1[k], c2[k])
    assert np.array_equal(o1[perm], o2)


def test_region_self_consistent_with_dense_cache():
    """A cache written by the dense block on x0 is a fixed point: recomputing
    any subset of tokens from x0 reproduces the dense result."""
    p = small_problem(TINY, 24)
    L = p["layers"][0]
    dense, K, V = O.dense_block(p["x"], L, p["m6"], O.text_kv(p["ctx"], L), TINY.heads)
    cache = {"H": dense, "K": K, "V": V}
    for idx in ([0], [3, 7, 8], list(range(0, 16, 3))):
        c, _ = _region(p, idx, cache=cache)
        for k, ref in (("H", dense), ("K", K), ("V", V)):
            assert np.allclose(c[k], ref, rtol=0, atol=1e-13)


def test_region_clean_rows_untouched_and_dirty_rows_use_fresh_kv():
    p = small_problem(TINY, 25)
    idx = np.array([2, 6, 11])
    c, out = _region(p, idx)
    clean = np.setdiff1d(np.arange(TINY.tokens), idx)
    for k in "HKV":
        assert np.array_equal(c[k][clean], p["cache"][k][clean])
    assert np.array_equal(c["H"][idx], out)
    # fresh K/V of the dirty rows: the qkv projection of the modulated rows
    L = p["layers"][0]
    _, k, v = O.qkv_rows(p["x"][idx], L, p["m6"][0], p["m6"][1])
    assert np.array_equal(c["K"][idx], k)
    assert np.array_equal(c["V"][idx], v)
    # and the result differs from attending over the stale cached K/V
    K_stale = p["cache"]["K"]
    q, _, _ = O.qkv_rows(p["x"][idx], L, p["m6"][0], p["m6"][1])
    o_stale = O.multihead_attention(q, K_stale, p["cache"]["V"], TINY.heads)
    o_fresh = O.multihead_attention(q, c["K"], c["V"], TINY.heads)
    assert not np.allclose(o_stale, o_fresh)


def test_region_single_dirty_token_attends_all_tokens():
    """One dirty token with its fresh key made dominant for head 0 must take
    that head's value; with a clean key dominant instead, that cached value."""
    p = small_problem(TINY, 26)
    L = p["layers"][0]
    N, dh = TINY.tokens, TINY.head_dim
    cache = {k: v.copy() for k, v in p["cache"].items()}
    q, _, _ = O.qkv_rows(p["x"][[5]], L, p["m6"][0], p["m6"][1])
    # make cached key 9 align strongly with the query in head 0
    cache["K"][9, :dh] = q[0, :dh] * 1e4
    c, _ = _region(p, [5], cache=cache)
    o = O.multihead_attention(q, c["K"], c["V"], TINY.heads)
    assert np.allclose(o[0, :dh], cache["V"][9, :dh], atol=1e-6)
    assert N == 16
