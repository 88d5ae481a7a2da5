"""The CUDA path computes the cross-attention logits with the query
projection folded into the text keys, once per turn: per head h,
(x W_xq,h^T + b_h) K_h^T = x G_h^T + kb_h with G_h = K_h W_xq,h and
kb_h = K_h b_h.  That reassociation gives the oracle's cross-attention
(Section 4.1 backbone, the text cross-attention of the block) up to float64
rounding, at the tiny and the PixArt-alpha head shapes."""
import math

import numpy as np
import pytest

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import small_problem


def folded_cross_attention(x, tk, tv, Lw, heads):
    d = x.shape[1]
    dh = d // heads
    W, b = Lw["W_xq"], Lw["b_xq"]
    outs = []
    for h in range(heads):
        cols = slice(h * dh, (h + 1) * dh)
        Kh, Vh = tk[:, cols], tv[:, cols]
        G = Kh @ W[cols, :]          # [M][d]
        kb = Kh @ b[cols]            # [M]
        s = (x @ G.T + kb) / math.sqrt(dh)
        p = np.exp(s - s.max(axis=1, keepdims=True))
        p /= p.sum(axis=1, keepdims=True)
        outs.append(p @ Vh)
    return O.linear(np.concatenate(outs, axis=1), Lw["W_xo"], Lw["b_xo"])


@pytest.mark.parametrize("dims", [synth.TINY,
                                  synth.Dims(grid_h=2, grid_w=3, layers=1, text_len=120),
                                  synth.Dims(grid_h=2, grid_w=2, layers=1, text_len=7)])
def test_folded_query_projection_gives_the_same_cross_attention(dims):
    P = small_problem(dims, 1234 + 1300)
    L = P["layers"][0]
    tk, tv = O.text_kv(P["ctx"], L)
    x = P["x"]
    want = O.cross_attention(x, tk, tv, L, dims.heads)
    got = folded_cross_attention(x, tk, tv, L, dims.heads)
    assert np.linalg.norm(got - want) <= 1e-12 * np.linalg.norm(want)


def test_fold_catches_a_dropped_query_bias():
    """The key-bias term kb_h carries the query bias: without it the result
    moves by far more than rounding."""
    dims = synth.TINY
    P = small_problem(dims, 1234 + 1301)
    L = dict(P["layers"][0])
    tk, tv = O.text_kv(P["ctx"], L)
    want = O.cross_attention(P["x"], tk, tv, L, dims.heads)
    L0 = dict(L, b_xq=np.zeros_like(L["b_xq"]))
    got = folded_cross_attention(P["x"], tk, tv, L0, dims.heads)
    assert np.linalg.norm(got - want) > 1e-6 * np.linalg.norm(want)
