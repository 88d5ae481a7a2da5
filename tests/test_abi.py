"""The C-ABI library builds, loads and exports every symbol of the header;
host-side validation rejects bad arguments before anything is launched.
CPU only: no call here reaches the GPU."""
import ctypes as C

import numpy as np
import pytest

from paper_2608_29809_gb300 import build as B


@pytest.fixture(scope="module")
def R():
    B.build()
    from paper_2608_29809_gb300 import regioncache
    return regioncache


def test_every_header_symbol_is_exported(R):
    names = R.header_symbols()
    assert len(names) >= 18
    lib = C.CDLL(R.LIB_PATH)
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing
    for n in ("rc_localize_mask", "rc_block_forward_region", "rc_step"):
        assert n in names


def test_status_strings(R):
    assert R.rc_status_string(0) == "ok"
    assert "index" in R.rc_status_string(6)
    assert R.rc_status_string(99) == "unknown status"


def test_create_rejects_bad_dims_without_touching_the_gpu(R):
    from paper_2608_29809_gb300 import synth
    bad = [synth.Dims(hidden=1152, heads=15), synth.Dims(hidden=1152, heads=12),
           synth.Dims(mlp=4600), synth.Dims(grid_h=200, grid_w=100), synth.Dims(layers=0)]
    for d in bad:
        with pytest.raises(R.RCError) as ei:
            R.rc_create(R.dims_struct(d))
        assert ei.value.status in (1, 2)
        assert R.rc_last_error()


def test_localize_rejects_bad_arguments(R):
    ws = C.c_void_p(256)  # never dereferenced: validation fails first
    ids = np.array([3, 200], np.int32)
    lib = R._lib

    def call(S=1, N=16, M=8, gh=4, gw=4, ids=ids[:1], thr=0.5, dil=1, ws_bytes=1 << 20):
        return lib.rc_localize_mask(256, S, N, M, gh, gw, ids.ctypes.data, len(ids), thr, dil,
                                    256, 256, 256, ws, ws_bytes, None)

    assert call(gh=3) == 2                       # N != grid_h * grid_w
    assert call(ids=ids) == 1                    # delta id 200 >= M
    assert call(dil=-1) == 1
    assert call(thr=float("nan")) == 1
    assert call(ws_bytes=8) == 1                 # workspace too small
    assert call(S=0) == 2
    assert lib.rc_localize_mask(256, 1, 16, 8, 4, 4, ids.ctypes.data, 0, 0.5, 1, 256, 256, 256,
                                ws, 1 << 20, None) == 1


def test_workspace_size_grows_with_n(R):
    a = R.rc_localize_workspace_size(1024, 4)
    b = R.rc_localize_workspace_size(4096, 4)
    assert 0 < a < b
    assert R.rc_localize_workspace_size(0, 4) == 0


def test_no_alloc_scratch_equals_the_workspace_at_its_limits(R):
    # the fixed scratch of rc_localize_mask_noalloc is exactly the workspace
    # of its largest allowed problem, and anything larger is refused before
    # the device is touched
    assert R.RC_NOALLOC_SCRATCH_BYTES == R.rc_localize_workspace_size(
        R.RC_NOALLOC_MAX_TOKENS, R.RC_NOALLOC_MAX_DELTA)
    assert R.rc_localize_workspace_size(R.RC_NOALLOC_MAX_TOKENS + 1, R.RC_NOALLOC_MAX_DELTA) > \
        R.RC_NOALLOC_SCRATCH_BYTES
    ids = np.arange(2, dtype=np.int32)
    lib = R._lib
    st = lib.rc_localize_mask_noalloc(256, 1, 113 * 145, 8, 113, 145, ids.ctypes.data, 2, 0.5, 1,
                                      256, 256, 256, None)
    assert st == 2 and "16384" in R.rc_last_error()
    ids17 = np.arange(17, dtype=np.int32)
    st = lib.rc_localize_mask_noalloc(256, 1, 64, 32, 8, 8, ids17.ctypes.data, 17, 0.5, 1, 256,
                                      256, 256, None)
    assert st == 2 and "n_delta <= 16" in R.rc_last_error()


def test_null_handles_are_rejected(R):
    lib = R._lib
    assert lib.rc_step(None, None, 0, None, 0, None, None, 0, None, None) == 1
    assert lib.rc_block_forward_region(None, None, 0, 0, 0, None, None, 0, None, None, None) == 1
    assert lib.rc_sync(None, None) == 1
    assert lib.rc_linear(None, None, None, None, None, 1, 128, 64, None) == 1


# --------------------------------------------- Eq. 1 / Eq. 2 (host-only entry points)
def test_reuse_schedule_matches_eq2_golden_and_oracle(R):
    import os
    import oracle as O
    golden = os.path.join(os.path.dirname(__file__), "golden", "eq2_reuse_cutoff.txt")
    for ln in open(golden):
        if ln.startswith("#") or not ln.strip():
            continue
        T, s, tau, tr = ln.split()
        modes = R.rc_reuse_schedule(float(s), float(tau), int(T))
        assert int((modes == R.RC_MODE_REUSE).sum()) == int(tr)
        assert np.array_equal(modes, O.schedule_eq2(float(s), float(tau), int(T)))
        assert np.all(modes[:int(tr)] == R.RC_MODE_REUSE) and np.all(modes[int(tr):] == R.RC_MODE_SPARSE)
    with pytest.raises(R.RCError):
        R.rc_reuse_schedule(0.1, 0.5, 0)
    with pytest.raises(R.RCError):
        R.rc_reuse_schedule(0.1, 0.5, 20, rho=1.5)


def test_prompt_similarity_eq1(R):
    import oracle as O
    g = np.random.default_rng(5)
    for dim in (1, 7, 4096):
        a = g.standard_normal(dim).astype(np.float32)
        b = g.standard_normal(dim).astype(np.float32)
        s = R.rc_prompt_similarity(a, b)
        assert abs(s - O.cosine_similarity(a, b)) <= 1e-6
        assert abs(R.rc_prompt_similarity(a, a) - 1.0) <= 1e-6
        assert abs(R.rc_prompt_similarity(a, -a) + 1.0) <= 1e-6
    with pytest.raises(R.RCError):
        R.rc_prompt_similarity(np.zeros(4, np.float32), np.ones(4, np.float32))
