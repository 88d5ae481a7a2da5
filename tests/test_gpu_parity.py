"""GPU parity: the CUDA path through the C ABI against the oracle on the same
seeded inputs."""
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


def _dev_i32(a):
    return torch.as_tensor(np.asarray(a, np.int32)).cuda()


# ------------------------------------------------------------- localisation
def _gpu_mask(R, A, ids, gh, gw, thr=0.5, dil=1):
    S, N, M = A.shape
    ws = torch.empty(R.rc_localize_workspace_size(N, len(ids)), dtype=torch.uint8, device="cuda")
    mask = torch.full((N,), 7, dtype=torch.uint8, device="cuda")
    idx = torch.full((N,), -5, dtype=torch.int32, device="cuda")
    cnt = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    R.rc_localize_mask(torch.from_numpy(np.ascontiguousarray(A)).cuda(), S, N, M, gh, gw, ids,
                       thr, dil, mask, idx, cnt, ws)
    torch.cuda.synchronize()
    D = int(cnt.item())
    return mask.cpu().numpy(), idx.cpu().numpy()[:D], D


@pytest.mark.parametrize("grid,dil,seed", [((32, 32), 1, 1), ((64, 64), 1, 2), ((32, 32), 0, 3),
                                           ((64, 64), 2, 4), ((17, 23), 1, 5)])
def test_localize_bit_exact_blob_scores(R, grid, dil, seed):
    d = synth.Dims(grid_h=grid[0], grid_w=grid[1])
    A, ids = synth.blob_scores(d, seed)
    m, idx, D = _gpu_mask(R, A, ids, d.grid_h, d.grid_w, 0.5, dil)
    m_ref, idx_ref = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, dil)
    assert np.array_equal(m, m_ref)
    assert D == len(idx_ref)
    assert np.array_equal(idx, idx_ref)


def test_localize_bit_exact_multi_slice_and_thresholds(R):
    d = synth.Dims(grid_h=32, grid_w=32)
    rng = np.random.default_rng(9)
    A = rng.random((5, d.tokens, d.text_len), dtype=np.float32) ** 3
    ids = np.array([1, 17, 64, 119], np.int32)
    for thr in (0.05, 0.3, 0.5, 0.9):
        m, idx, D = _gpu_mask(R, A, ids, d.grid_h, d.grid_w, thr, 1)
        m_ref, idx_ref = O.localize_mask(A, ids, d.grid_h, d.grid_w, thr, 1)
        assert np.array_equal(m, m_ref) and np.array_equal(idx, idx_ref)


def test_localize_edge_cases(R):
    # constant columns: empty mask, D = 0
    A = np.full((1, 64, 8), 0.125, np.float32)
    m, idx, D = _gpu_mask(R, A, np.array([0, 3]), 8, 8)
    assert D == 0 and m.sum() == 0
    # golden 6x6 example
    from tests.test_oracle_localize_step import _read_localize_golden
    A, _, mask = _read_localize_golden()
    m, idx, D = _gpu_mask(R, A, np.array([1, 3]), 6, 6)
    assert np.array_equal(m.reshape(6, 6), mask)
    # everything dirty: single token grid-wide plateau
    A = np.zeros((1, 300, 4), np.float32)
    A[0, :, 2] = 1.0
    A[0, 7, 2] = 0.0
    m, idx, D = _gpu_mask(R, A, np.array([2]), 15, 20, 0.5, 1)
    assert D == 300 and np.array_equal(idx, np.arange(300))


def test_localize_non_finite_columns_give_no_token(R):
    # a delta column whose scores hold NaN or +-Inf contributes nothing; the
    # finite columns beside it still do (bit-exact with the oracle)
    d = synth.Dims(grid_h=32, grid_w=32)
    A, ids = synth.blob_scores(d, 11, n_delta=(4, 4))
    A = A.copy()
    A[0, 5, ids[0]] = np.nan
    A[0, 700, ids[1]] = np.inf
    A[0, 3, ids[2]] = -np.inf
    m, idx, D = _gpu_mask(R, A, ids, d.grid_h, d.grid_w, 0.5, 1)
    m_ref, idx_ref = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 1)
    m_last, _ = O.localize_mask(A, ids[3:], d.grid_h, d.grid_w, 0.5, 1)
    assert np.array_equal(m_ref, m_last) and D > 0
    assert np.array_equal(m, m_ref) and np.array_equal(idx, idx_ref)
    # two slices whose finite sum overflows to +Inf in f32: the mean is
    # non-finite and the column drops out on both sides
    A2 = np.stack([A[0], A[0]])
    A2[:, :, ids[3]] = np.nan_to_num(A2[:, :, ids[3]])
    A2[:, 9, ids[3]] = 3.0e38
    m2, idx2, D2 = _gpu_mask(R, A2, ids[3:], d.grid_h, d.grid_w, 0.5, 1)
    assert D2 == 0 and m2.sum() == 0


def test_localize_indicator_ellipses_4096(R):
    d = synth.PIXART_1024
    for f in (0.05, 0.1, 0.2, 0.4):
        blobs = synth.ellipse_blobs(d, 1234 + 200, f)
        A, ids = synth.indicator_scores(d, blobs, 1234 + 200)
        m, idx, D = _gpu_mask(R, A, ids, d.grid_h, d.grid_w, 0.5, 0)
        m_ref, idx_ref = O.localize_mask(A, ids, d.grid_h, d.grid_w, 0.5, 0)
        assert np.array_equal(m, m_ref) and np.array_equal(idx, idx_ref)
        assert abs(D / d.tokens - f) <= 0.0051


# -------------------------------------------------------------------- GEMM
# the tile width is chosen on the device from the row count: these shapes
# take 64 (1, 37, 128, 1000 rows), 128 (300 x 3456), 192 (831 x 3456) and 256
# (831 x 4608); from 2048 rows (known on the host) CTA pairs share M = 256
# MMAs, including a ragged last pair (2900 rows: 23 row tiles) and split k.
# When every CTA holds one tile, tiles up to 192 wide are issued by two MMA
# threads (even / odd k-blocks into two accumulators): 2, 3 and 19 k-blocks
# give them equal and unequal shares, 1 k-block leaves the second idle.
@pytest.mark.parametrize("rows,n,k", [(1, 128, 64), (37, 1152, 1152), (128, 256, 4608),
                                      (300, 3456, 1152), (1000, 1152, 4608), (831, 3456, 1152),
                                      (831, 4608, 1152), (2048, 1152, 1152), (2900, 1152, 4608),
                                      (3001, 3456, 1152), (4096, 4608, 1152), (96, 384, 128),
                                      (200, 256, 192), (831, 1152, 1216), (500, 640, 64)])
def test_linear_matches_fp64(R, rows, n, k):
    g = torch.Generator().manual_seed(rows * 7 + n)
    x = torch.randn(rows, k, generator=g).to(torch.bfloat16)
    W = (torch.randn(n, k, generator=g) * 0.02).to(torch.bfloat16)
    b = torch.randn(n, generator=g)
    d = synth.Dims(grid_h=2, grid_w=2, layers=1)
    ctx = R.rc_create(R.dims_struct(d))
    try:
        y = torch.full((rows, n), float("nan"), device="cuda")
        R.rc_linear(ctx, x.cuda(), W.cuda(), b.cuda(), y, rows, n, k)
        R.rc_sync(ctx)
    finally:
        R.rc_destroy(ctx)
    ref = O.linear(O.to64(x), O.to64(W), O.to64(b))
    got = y.cpu().double().numpy()
    assert np.max(np.abs(got - ref)) <= 1e-4 * (1 + np.max(np.abs(ref)))


# --------------------------------------------------------------- attention
# Key splits across the shapes (two CTAs per SM on 152 SMs): 831 x 4096 is
# cut into 304 equal ranges (3-4 pieces per pair); 205 x 4096, 410 x 4096
# and 100 x 16384 into 256 ranges aligned to the pairs (8, 4 and 16 pieces
# per pair, beyond the combine's unrolled depths); 37 x 3000 into 188 equal
# ranges over 47 key blocks per pair (12-13 pieces, ragged last block).
@pytest.mark.parametrize("Nq,Nk,ld_kv", [(1, 120, 2304), (37, 256, 1152), (200, 1024, 1152),
                                         (831, 4096, 1152), (128, 120, 2304), (300, 4096, 1152),
                                         (205, 4096, 1152), (410, 4096, 1152),
                                         (100, 16384, 1152), (37, 3000, 1152)])
def test_attention_matches_fp64(R, Nq, Nk, ld_kv):
    d = synth.PIXART_1024
    g = torch.Generator().manual_seed(Nq * 31 + Nk)
    h = d.hidden
    Q = torch.randn(Nq, h, generator=g).to(torch.bfloat16)
    KV = (torch.randn(Nk, ld_kv, generator=g) * 1.5).to(torch.bfloat16)
    Vsrc = torch.randn(Nk, ld_kv, generator=g).to(torch.bfloat16)
    ctx = R.rc_create(R.dims_struct(d))
    try:
        out = torch.full((Nq, h), float("nan"), dtype=torch.bfloat16, device="cuda")
        Kd, Vd = KV.cuda(), Vsrc.cuda()
        R.rc_attention(ctx, Q.cuda(), h, Kd, Vd, ld_kv, Nq, Nk, out, h)
        R.rc_sync(ctx)
    finally:
        R.rc_destroy(ctx)
    got = out.cpu().double().numpy()
    want = O.multihead_attention(O.to64(Q), O.to64(KV[:, :h]), O.to64(Vsrc[:, :h]), d.heads)
    # Raw attention outputs, not block outputs: the output is bf16 (half an
    # ulp is up to 2^-8 of an element's size) and so is P (each probability
    # off by up to 2^-8 of itself, which a row that attends to few keys
    # passes on to its outputs at their own scale), while the output RMS
    # shrinks like 1/sqrt(effective keys), so such rows hold elements many
    # times the RMS.  Bound: relative L2 <= 1e-2, per element
    # |err| <= 2^-7 |want| + 2e-2 x RMS, cosine >= 0.9999.
    err = got - want
    rms = np.sqrt(np.mean(want ** 2))
    assert np.linalg.norm(err) <= 1e-2 * np.linalg.norm(want), f"Nq={Nq} Nk={Nk} rel L2"
    excess = np.abs(err) - (2.0 ** -7 * np.abs(want) + 2e-2 * rms)
    assert np.max(excess) <= 0, f"Nq={Nq} Nk={Nk}: {np.max(np.abs(err)):.2e}"
    cos = float((got * want).sum() / (np.linalg.norm(got) * np.linalg.norm(want)))
    assert cos >= 0.9999, cos


# ------------------------------------------------------------- one block
@pytest.fixture(scope="module")
def block_problem(R):
    p = Problem(R, synth.ONE_BLOCK_256, 1234 + 100)
    yield p
    p.close()


def _run_block(R, p, idx, x, t=0, use_count=False):
    d = p.d
    mod6 = synth.make_mod6(d, p.model.w.layers[0]["table"].cpu(), p.seed)
    hidden = x.clone().cuda()
    idx_d = _dev_i32(idx if len(idx) else [0])
    if use_count:
        cnt = _dev_i32([len(idx)])
        R.rc_block_forward_region(p.model.ctx, p.model.cache, 0, 0, t, hidden, idx_d, -1, cnt,
                                  mod6.cuda())
    else:
        R.rc_block_forward_region(p.model.ctx, p.model.cache, 0, 0, t, hidden, idx_d, len(idx),
                                  None, mod6.cuda())
    R.rc_sync(p.model.ctx)
    return hidden.cpu(), O.to64(mod6)


def _oracle_block(p, idx, x, m6, cache):
    return O.region_block(O.to64(x)[idx], np.asarray(idx), cache, p.layers64[0], m6, p.tkv64[0],
                          p.d.heads)


@pytest.mark.parametrize("use_count", [False, True])
def test_block_region_parity_c1(R, block_problem, use_count):
    """One PixArt-alpha block, 256 tokens, ~15 % dirty rectangle (fp32 in/out)."""
    p = block_problem
    d = p.d
    t = 0
    base = p.read_slot(0, t)
    idx = np.flatnonzero(synth.rectangle_mask(d, p.seed))
    assert 35 <= len(idx) <= 42
    x = synth.make_hidden(d, p.seed)
    hidden, m6 = _run_block(R, p, idx, x, t, use_count)
    ref_cache, ref_out = _oracle_block(p, idx, x, m6, base)
    block_close(hidden.numpy()[idx], ref_out, "block output rows")
    after = p.read_slot(0, t)
    clean = np.setdiff1d(np.arange(d.tokens), idx)
    for k in "HKV":
        assert np.array_equal(after[k][clean], base[k][clean]), f"clean rows of {k} changed"
        block_close(after[k][idx], ref_cache[k][idx], f"cache {k} dirty rows")
    # rows outside idx of `hidden` are untouched
    assert torch.equal(hidden[clean], x[clean])
    # restore the slot for the other tests
    H, K, V = synth.make_cache_slice(d, p.seed, 0, 0, t)
    R.rc_cache_fill(p.model.cache, 0, 0, t, H.cuda(), K.cuda(), V.cuda())


def test_block_all_dirty_and_empty(R, block_problem):
    p = block_problem
    d = p.d
    base = p.read_slot(0, 0)
    x = synth.make_hidden(d, p.seed + 1)
    # D = 0: nothing changes
    hidden, _ = _run_block(R, p, np.array([], np.int64), x)
    assert torch.equal(hidden, x)
    after = p.read_slot(0, 0)
    for k in "HKV":
        assert np.array_equal(after[k], base[k])
    # all dirty, in a permuted order: equals the dense block
    perm = np.random.default_rng(3).permutation(d.tokens)
    hidden, m6 = _run_block(R, p, perm, x)
    dense, K, V = O.dense_block(O.to64(x), p.layers64[0], m6, p.tkv64[0], d.heads)
    block_close(hidden.numpy(), dense, "all-dirty block vs dense")
    after = p.read_slot(0, 0)
    block_close(after["K"], K, "dense K")
    block_close(after["V"], V, "dense V")
    H, K, V = synth.make_cache_slice(d, p.seed, 0, 0, 0)
    R.rc_cache_fill(p.model.cache, 0, 0, 0, H.cuda(), K.cuda(), V.cuda())


def test_block_bad_index_is_reported(R, block_problem):
    p = block_problem
    x = synth.make_hidden(p.d, p.seed)
    with pytest.raises(R.RCError) as ei:
        _run_block(R, p, np.array([3, 5000]), x)
    assert ei.value.status == 6
    H, K, V = synth.make_cache_slice(p.d, p.seed, 0, 0, 0)
    R.rc_cache_fill(p.model.cache, 0, 0, 0, H.cuda(), K.cuda(), V.cuda())
    torch.cuda.synchronize()


# ------------------------------------------------------------------ steps
@pytest.fixture(scope="module")
def step_problem(R):
    d = synth.Dims(grid_h=16, grid_w=16, layers=4, timesteps=20)
    p = Problem(R, d, 4321, ts=(3,))
    yield p
    p.close()


def _gpu_step(R, p, lat, t, mode, idx, use_count=False):
    sched = np.full(p.d.timesteps, mode, np.uint8)
    latent = lat.clone().cuda()
    if mode == O.MODE_SPARSE:
        idx_d = _dev_i32(idx if len(idx) else [0])
        cnt = _dev_i32([len(idx)]) if use_count else None
        R.rc_step(p.model.ctx, p.model.cache, 0, latent, t, sched, idx_d,
                  -1 if use_count else len(idx), cnt)
    else:
        R.rc_step(p.model.ctx, p.model.cache, 0, latent, t, sched, None, 0, None)
    R.rc_sync(p.model.ctx)
    return latent.cpu().double().numpy()


def _reset(R, p, t):
    for l in range(p.d.layers):
        H, K, V = synth.make_cache_slice(p.d, p.seed, 0, l, t)
        R.rc_cache_fill(p.model.cache, 0, l, t, H.cuda(), K.cuda(), V.cuda())
    torch.cuda.synchronize()


@pytest.mark.parametrize("mode", [O.MODE_SPARSE, O.MODE_DENSE, O.MODE_REUSE])
def test_step_parity_small(R, step_problem, mode):
    p = step_problem
    t = 3
    _reset(R, p, t)
    lat = synth.make_latent(p.d, p.seed)
    idx = np.flatnonzero(synth.rectangle_mask(p.d, p.seed))
    got = _gpu_step(R, p, lat, t, mode, idx, use_count=(mode == O.MODE_SPARSE))
    ref, eps, cache = p.oracle_step(O.to64(lat), t, mode, idx)
    assert rel_l2(got, ref) <= LATENT_REL_L2
    # the model output itself, recovered from the update, at block tolerance
    ab_t, ab_n = float(p.ab[t]), float(p.ab[t + 1])
    x = O.to64(lat)
    c_x = np.sqrt(ab_n / ab_t)
    c_e = np.sqrt(1 - ab_n) - np.sqrt(ab_n) * np.sqrt(1 - ab_t) / np.sqrt(ab_t)
    block_close((got - c_x * x) / c_e, eps, "eps")
    last = p.read_slot(p.d.layers - 1, t)
    block_close(last["H"], cache[-1]["H"], "H of the last block")
    _reset(R, p, t)


def test_step_after_schedule_change(R, step_problem):
    """The per-timestep embeddings are computed once per schedule: after
    rc_set_schedule with other timestep values, a step uses the new ones."""
    p = step_problem
    t = 3
    lat = synth.make_latent(p.d, p.seed)
    idx = np.flatnonzero(synth.rectangle_mask(p.d, p.seed))
    _reset(R, p, t)
    _gpu_step(R, p, lat, t, O.MODE_SPARSE, idx)  # embeddings of the first schedule
    tv0 = p.tv
    tv1 = (np.float32(999.0) - tv0).astype(np.float32)  # the schedule reversed
    ref0, _, _ = p.oracle_step(O.to64(lat), t, O.MODE_SPARSE, idx)
    try:
        R.rc_set_schedule(p.model.ctx, tv1, p.ab)
        p.tv = tv1
        _reset(R, p, t)
        got = _gpu_step(R, p, lat, t, O.MODE_SPARSE, idx)
        ref, _, _ = p.oracle_step(O.to64(lat), t, O.MODE_SPARSE, idx)
        # the two schedules give results far apart, so stale embeddings fail
        assert rel_l2(ref0, ref) > 2 * LATENT_REL_L2
        assert rel_l2(got, ref) <= LATENT_REL_L2
    finally:
        R.rc_set_schedule(p.model.ctx, tv0, p.ab)
        p.tv = tv0
        _reset(R, p, t)


@pytest.fixture(scope="module")
def c2_problem(R):
    p = Problem(R, synth.PIXART_512, 1234 + 200, ts=(5,))
    yield p
    p.close()


def test_step_c2_localized_sparse(R, c2_problem):
    """Full 28-block step at 512 px (1024 tokens): the dirty set comes from the
    localisation kernel on a random score map with 3-8 delta tokens."""
    p = c2_problem
    d = p.d
    A, ids = synth.blob_scores(d, p.seed)
    mask, idx, D = _gpu_mask(R, A, ids, d.grid_h, d.grid_w, 0.5, 1)
    assert 0 < D < d.tokens
    t = 5
    lat = synth.make_latent(d, p.seed)
    got = _gpu_step(R, p, lat, t, O.MODE_SPARSE, idx)
    ref, eps, cache = p.oracle_step(O.to64(lat), t, O.MODE_SPARSE, idx)
    assert rel_l2(got, ref) <= LATENT_REL_L2
    ab_t, ab_n = float(p.ab[t]), float(p.ab[t + 1])
    x = O.to64(lat)
    c_x = np.sqrt(ab_n / ab_t)
    c_e = np.sqrt(1 - ab_n) - np.sqrt(ab_n) * np.sqrt(1 - ab_t) / np.sqrt(ab_t)
    block_close((got - c_x * x) / c_e, eps, "eps")
    for l in (0, 13, 27):
        s = p.read_slot(l, t)
        block_close(s["H"][idx], cache[l]["H"][idx], f"H rows, layer {l}")
        block_close(s["K"][idx], cache[l]["K"][idx], f"K rows, layer {l}")
