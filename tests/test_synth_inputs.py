"""The seeded synthetic inputs that stand in for the paper's editing
workloads and the PixArt-alpha weights: each generator produces the shapes,
distributions and structure the workload recipe states, and the same seed
always gives the same tensor."""
import numpy as np
import pytest
import torch

from paper_2608_29809_gb300 import synth

D1024 = synth.PIXART_1024
D256 = synth.Dims(grid_h=16, grid_w=16)


def test_rectangle_mask_is_one_rectangle_of_35_to_42_tokens():
    for seed in range(20):
        m = synth.rectangle_mask(D256, seed).reshape(D256.grid_h, D256.grid_w)
        assert 35 <= m.sum() <= 42
        ys, xs = np.nonzero(m)
        box = m[ys.min():ys.max() + 1, xs.min():xs.max() + 1]
        assert box.all(), "not a filled axis-aligned rectangle"
        assert np.array_equal(m, synth.rectangle_mask(D256, seed).reshape(m.shape))


@pytest.mark.parametrize("frac", [0.05, 0.10, 0.20, 0.40])
def test_ellipse_union_hits_the_dirty_fraction(frac):
    for seed in (1, 2, 3):
        blobs = synth.ellipse_blobs(D1024, seed, frac)
        assert 1 <= len(blobs) <= 3
        union = np.logical_or.reduce(blobs)
        assert abs(union.mean() - frac) <= 0.005
        again = synth.ellipse_blobs(D1024, seed, frac)
        assert all(np.array_equal(a, b) for a, b in zip(blobs, again))


def test_indicator_scores_mark_each_blob_in_its_delta_column():
    blobs = synth.ellipse_blobs(D1024, 9, 0.2)
    A, ids = synth.indicator_scores(D1024, blobs, 9)
    assert A.shape == (1, D1024.tokens, D1024.text_len) and A.dtype == np.float32
    assert len(set(ids.tolist())) == len(blobs)
    for j, b in zip(ids, blobs):
        col = A[0, :, j]
        assert col[b].min() >= 0.6 and col[~b].max() <= 0.4
    others = np.setdiff1d(np.arange(D1024.text_len), ids)
    assert 0.0 <= A[0][:, others].min() and A[0][:, others].max() <= 1.0


def test_blob_scores_are_row_softmaxes_with_3_to_8_delta_tokens():
    d = synth.PIXART_512
    for seed in range(5):
        A, ids = synth.blob_scores(d, seed)
        assert A.shape == (1, d.tokens, d.text_len)
        assert np.allclose(A[0].sum(axis=1), 1.0, atol=1e-5) and (A > 0).all()
        assert 3 <= len(ids) <= 8 and len(set(ids.tolist())) == len(ids)
        # each delta token's column peaks where its bump was added
        assert all(A[0, :, j].max() > 5 * A[0].mean() for j in ids)


def test_tensors_are_seeded_per_name():
    d = synth.Dims(grid_h=4, grid_w=4, layers=2, timesteps=2)
    a = synth.make_cache_slice(d, 5, 0, 1, 1)
    b = synth.make_cache_slice(d, 5, 0, 1, 1)
    assert all(torch.equal(x, y) for x, y in zip(a, b))
    others = [synth.make_cache_slice(d, 5, 0, 0, 1), synth.make_cache_slice(d, 5, 0, 1, 0),
              synth.make_cache_slice(d, 5, 1, 1, 1), synth.make_cache_slice(d, 6, 0, 1, 1)]
    for o in others:
        assert not any(torch.equal(x, y) for x, y in zip(a, o))
    H, K, V = a
    assert not torch.equal(H, K) and not torch.equal(K, V)
    assert H.dtype == torch.bfloat16 and H.shape == (d.tokens, d.hidden)


def test_weight_shapes_and_distributions():
    d = synth.Dims(grid_h=4, grid_w=4, layers=2)
    w = synth.make_weights(d, 3)
    for L in w.layers:
        for name, shp in synth.layer_shapes(d).items():
            assert tuple(L[name].shape) == shp, name
            assert L[name].dtype == (torch.bfloat16 if name.startswith("W_") else torch.float32)
    big = w.layers[0]["W_1"].float()
    assert abs(big.std().item() - 0.02) < 0.001 and abs(big.mean().item()) < 0.001
    assert not torch.equal(w.layers[0]["W_1"], w.layers[1]["W_1"])


def test_sincos_positions():
    d = synth.Dims(grid_h=4, grid_w=6)
    P = synth.sincos_pos_table(d).double().numpy()
    q = d.hidden // 4
    assert P.shape == (d.tokens, d.hidden)
    # token 0 is (y, x) = (0, 0): every sine 0, every cosine 1
    assert np.allclose(P[0, :q], 0) and np.allclose(P[0, q:2 * q], 1)
    # token y * W + x: the first half encodes y, the second x, each as
    # [sin(p w_k) | cos(p w_k)] with w_k = 10000^(-k / q)
    y, x, k = 2, 5, 7
    w = 10000.0 ** (-k / q)
    r = P[y * d.grid_w + x]
    assert np.isclose(r[k], np.sin(y * w), atol=1e-6)
    assert np.isclose(r[q + k], np.cos(y * w), atol=1e-6)
    assert np.isclose(r[2 * q + k], np.sin(x * w), atol=1e-6)
    assert np.isclose(r[3 * q + k], np.cos(x * w), atol=1e-6)
