"""ctypes binding of the C ABI in include/regioncache.h.

Argument marshalling only: every function below forwards to the entry point
of the same name in libregioncache.so; tensors are passed as raw device
pointers.  The library is loaded from the package's ``_build`` directory and
importing this module fails loudly when it is missing (there is no fallback).
A non-OK status raises ``RCError``.
"""
from __future__ import annotations

import ctypes as C
import os
import re

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libregioncache.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "regioncache.h")

RC_OK = 0
RC_MODE_DENSE, RC_MODE_SPARSE, RC_MODE_REUSE = 0, 1, 2
STATUS = {0: "RC_OK", 1: "RC_ERR_INVALID_ARG", 2: "RC_ERR_SHAPE", 3: "RC_ERR_OOM",
          4: "RC_ERR_CUDA", 5: "RC_ERR_TIMEOUT", 6: "RC_ERR_DEVICE_ASSERT", 7: "RC_ERR_STATE",
          8: "RC_ERR_IO"}


class RCError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class rc_dims(C.Structure):
    _fields_ = [(n, C.c_int) for n in ("hidden", "heads", "mlp", "layers", "grid_h", "grid_w",
                                       "patch", "in_ch", "out_ch", "text_len", "timesteps",
                                       "freq_dim", "max_batch")]


RC_MAX_BATCH = 16


def header_define(name: str) -> int:
    """Integer value of a ``#define`` of the header (read from the file)."""
    m = re.search(r"^#define\s+" + re.escape(name) + r"\s+(\d+)\b", open(HEADER).read(), re.M)
    if not m:
        raise KeyError(name)
    return int(m.group(1))


RC_NOALLOC_MAX_TOKENS = header_define("RC_NOALLOC_MAX_TOKENS")
RC_NOALLOC_MAX_DELTA = header_define("RC_NOALLOC_MAX_DELTA")
RC_NOALLOC_SCRATCH_BYTES = header_define("RC_NOALLOC_SCRATCH_BYTES")


class rc_batch_item(C.Structure):
    _fields_ = [("session", C.c_int), ("latent", C.c_void_p), ("t", C.c_int), ("mode", C.c_int),
                ("dirty_idx", C.c_void_p), ("D", C.c_int), ("dirty_count", C.c_void_p)]


LAYER_FIELDS = ("W_qkv", "b_qkv", "W_o", "b_o", "W_xq", "b_xq", "W_xkv", "b_xkv", "W_xo",
                "b_xo", "W_1", "b_1", "W_2", "b_2", "table")
GLOBAL_FIELDS = ("W_e", "b_e", "pos", "W_t1", "b_t1", "W_t2", "b_t2", "W_tb", "b_tb", "table_f",
                 "W_f", "b_f")


class rc_layer_weights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in LAYER_FIELDS]


class rc_global_weights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in GLOBAL_FIELDS]


def load_library(path: str = LIB_PATH) -> C.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"libregioncache.so not built at {path}; run "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    lib = C.CDLL(path)
    P, I, F, S = C.c_void_p, C.c_int, C.c_float, C.c_size_t
    sig = {
        "rc_create": (I, [C.POINTER(rc_dims), C.POINTER(P)]),
        "rc_destroy": (None, [P]),
        "rc_set_layer_weights": (I, [P, I, C.POINTER(rc_layer_weights)]),
        "rc_set_global_weights": (I, [P, C.POINTER(rc_global_weights)]),
        "rc_set_schedule": (I, [P, P, P]),
        "rc_set_deterministic": (I, [P, I]),
        "rc_cache_create": (I, [P, I, C.POINTER(P)]),
        "rc_cache_create_host": (I, [P, I, C.POINTER(P)]),
        "rc_cache_export": (I, [P, I, C.c_char_p]),
        "rc_cache_import": (I, [P, I, C.c_char_p]),
        "rc_step_graph_create": (I, [P, P, I, P, I, P, P, I, P, C.POINTER(P)]),
        "rc_graph_launch": (I, [P, P]),
        "rc_graph_destroy": (None, [P]),
        "rc_cache_destroy": (None, [P]),
        "rc_cache_fill": (I, [P, I, I, I, P, P, P, P]),
        "rc_cache_read": (I, [P, I, I, I, P, P, P, P]),
        "rc_set_text": (I, [P, P, I, P, P]),
        "rc_localize_workspace_size": (S, [I, I]),
        "rc_localize_mask": (I, [P, I, I, I, I, I, P, I, F, I, P, P, P, P, S, P]),
        "rc_localize_mask_noalloc": (I, [P, I, I, I, I, I, P, I, F, I, P, P, P, P]),
        "rc_localize_scores": (I, [P, P, I, I, P, P, I, P, P]),
        "rc_server_create": (I, [P, P, I, C.POINTER(P)]),
        "rc_server_destroy": (None, [P]),
        "rc_server_admit": (I, [P, I, P, P, P, I, P]),
        "rc_server_tick": (I, [P, P, P, C.POINTER(I)]),
        "rc_server_state": (I, [P, I, C.POINTER(I)]),
        "rc_server_running": (I, [P]),
        "rc_selftest_wait": (I, [P, I, I, P]),
        "rc_block_forward_region": (I, [P, P, I, I, I, P, P, I, P, P, P]),
        "rc_step": (I, [P, P, I, P, I, P, P, I, P, P]),
        "rc_step_batched": (I, [P, P, C.POINTER(rc_batch_item), I, P]),
        "rc_step_capture": (I, [P, P, I, P, I, P, I, P, P]),
        "rc_prompt_similarity": (I, [P, P, I, C.POINTER(F)]),
        "rc_reuse_schedule": (I, [F, F, F, I, P]),
        "rc_step_dense": (I, [P, P, I, P, I, P]),
        "rc_linear": (I, [P, P, P, P, P, I, I, I, P]),
        "rc_attention": (I, [P, P, I, P, P, I, I, I, P, I, P]),
        "rc_sync": (I, [P, P]),
        "rc_probe_enable": (I, [P, I, I]),
        "rc_probe_read": (I, [P, C.POINTER(C.c_double), C.POINTER(I)]),
        "rc_probe_read_each": (I, [P, C.POINTER(C.c_float), I, C.POINTER(I)]),
        "rc_launch_count": (C.c_uint64, []),
        "rc_status_string": (C.c_char_p, [I]),
        "rc_last_error": (C.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


def header_symbols(path: str = HEADER):
    """Names of the entry points declared in the header."""
    text = open(path).read()
    return sorted(set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(rc_\w+)\s*\(", text, re.M)))


_lib = load_library()


def _check(status):
    if status != RC_OK:
        raise RCError(status, _lib.rc_last_error().decode())


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


# ----------------------------------------------------- one call per entry point
def rc_create(dims) -> int:
    h = C.c_void_p()
    _check(_lib.rc_create(C.byref(dims), C.byref(h)))
    return h.value


def rc_destroy(ctx):
    _lib.rc_destroy(ctx)


def rc_set_layer_weights(ctx, layer, tensors: dict):
    w = rc_layer_weights(*[_ptr(tensors[n]) for n in LAYER_FIELDS])
    _check(_lib.rc_set_layer_weights(ctx, layer, C.byref(w)))


def rc_set_global_weights(ctx, tensors: dict):
    w = rc_global_weights(*[_ptr(tensors[n]) for n in GLOBAL_FIELDS])
    _check(_lib.rc_set_global_weights(ctx, C.byref(w)))


def rc_set_schedule(ctx, t_values, alpha_bar):
    tv = np.ascontiguousarray(t_values, np.float32)
    ab = np.ascontiguousarray(alpha_bar, np.float32)
    _check(_lib.rc_set_schedule(ctx, tv.ctypes.data, ab.ctypes.data))


def rc_set_deterministic(ctx, on: bool):
    _check(_lib.rc_set_deterministic(ctx, 1 if on else 0))


def rc_cache_create(ctx, sessions) -> int:
    h = C.c_void_p()
    _check(_lib.rc_cache_create(ctx, sessions, C.byref(h)))
    return h.value


def rc_cache_create_host(ctx, sessions) -> int:
    h = C.c_void_p()
    _check(_lib.rc_cache_create_host(ctx, sessions, C.byref(h)))
    return h.value


def rc_cache_export(cache, session, path):
    _check(_lib.rc_cache_export(cache, session, os.fsencode(path)))


def rc_cache_import(cache, session, path):
    _check(_lib.rc_cache_import(cache, session, os.fsencode(path)))


def rc_cache_destroy(cache):
    _lib.rc_cache_destroy(cache)


def rc_cache_fill(cache, session, layer, t, H, K, V, stream=None):
    _check(_lib.rc_cache_fill(cache, session, layer, t, _ptr(H), _ptr(K), _ptr(V),
                              _stream(stream)))


def rc_cache_read(cache, session, layer, t, H, K, V, stream=None):
    _check(_lib.rc_cache_read(cache, session, layer, t, _ptr(H), _ptr(K), _ptr(V),
                              _stream(stream)))


def rc_set_text(ctx, cache, session, text, stream=None):
    _check(_lib.rc_set_text(ctx, cache, session, _ptr(text), _stream(stream)))


def rc_localize_workspace_size(N, n_delta) -> int:
    return int(_lib.rc_localize_workspace_size(N, n_delta))


def rc_localize_mask(xattn, S, N, M, grid_h, grid_w, delta_ids, threshold, dilation, mask,
                     dirty_idx, dirty_count, workspace, stream=None):
    ids = np.ascontiguousarray(delta_ids, np.int32)
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    _check(_lib.rc_localize_mask(_ptr(xattn), S, N, M, grid_h, grid_w, ids.ctypes.data,
                                 len(ids), float(threshold), dilation, _ptr(mask),
                                 _ptr(dirty_idx), _ptr(dirty_count), _ptr(workspace), ws_bytes,
                                 _stream(stream)))


def rc_localize_mask_noalloc(xattn, S, N, M, grid_h, grid_w, delta_ids, threshold, dilation,
                             mask, dirty_idx, dirty_count, stream=None):
    ids = np.ascontiguousarray(delta_ids, np.int32)
    _check(_lib.rc_localize_mask_noalloc(_ptr(xattn), S, N, M, grid_h, grid_w, ids.ctypes.data,
                                         len(ids), float(threshold), dilation, _ptr(mask),
                                         _ptr(dirty_idx), _ptr(dirty_count), _stream(stream)))


def rc_localize_scores(ctx, cache, session, t, latent, delta_ids, scores, stream=None):
    ids = np.ascontiguousarray(delta_ids, np.int32)
    _check(_lib.rc_localize_scores(ctx, cache, session, t, _ptr(latent), ids.ctypes.data,
                                   len(ids), _ptr(scores), _stream(stream)))


def rc_server_create(ctx, cache, max_items) -> int:
    out = C.c_void_p()
    _check(_lib.rc_server_create(ctx, cache, max_items, C.byref(out)))
    return out.value


def rc_server_destroy(server):
    _lib.rc_server_destroy(server)


def rc_server_admit(server, session, latent, schedule, dirty_idx, D, dirty_count):
    sch = np.ascontiguousarray(schedule, np.uint8)
    _check(_lib.rc_server_admit(server, session, _ptr(latent), sch.ctypes.data, _ptr(dirty_idx),
                                D, _ptr(dirty_count)))


def rc_server_tick(server, max_items, stream=None):
    """One tick; returns the list of sessions it stepped."""
    buf = (C.c_int * max(1, max_items))()
    n = C.c_int()
    _check(_lib.rc_server_tick(server, _stream(stream), buf, C.byref(n)))
    return [buf[i] for i in range(n.value)]


def rc_server_state(server, session) -> int:
    t = C.c_int()
    _check(_lib.rc_server_state(server, session, C.byref(t)))
    return t.value


def rc_server_running(server) -> int:
    return int(_lib.rc_server_running(server))


def rc_block_forward_region(ctx, cache, session, layer, t, hidden, dirty_idx, D, dirty_count,
                            mod6, stream=None):
    _check(_lib.rc_block_forward_region(ctx, cache, session, layer, t, _ptr(hidden),
                                        _ptr(dirty_idx), D, _ptr(dirty_count), _ptr(mod6),
                                        _stream(stream)))


def rc_step(ctx, cache, session, latent, t, schedule, dirty_idx, D, dirty_count, stream=None):
    sch = np.ascontiguousarray(schedule, np.uint8)
    _check(_lib.rc_step(ctx, cache, session, _ptr(latent), t, sch.ctypes.data, _ptr(dirty_idx),
                        D, _ptr(dirty_count), _stream(stream)))


def rc_step_graph_create(ctx, cache, session, latent, t, schedule, dirty_idx, D,
                         dirty_count) -> int:
    sch = np.ascontiguousarray(schedule, np.uint8)
    h = C.c_void_p()
    _check(_lib.rc_step_graph_create(ctx, cache, session, _ptr(latent), t, sch.ctypes.data,
                                     _ptr(dirty_idx), D, _ptr(dirty_count), C.byref(h)))
    return h.value


def rc_graph_launch(graph, stream=None):
    _check(_lib.rc_graph_launch(graph, _stream(stream)))


def rc_graph_destroy(graph):
    _lib.rc_graph_destroy(graph)


def rc_step_batched(ctx, cache, items, stream=None):
    """items: sequence of dicts with session, latent, t, mode and, for SPARSE,
    dirty_idx, D (-1: device count) and dirty_count."""
    arr = (rc_batch_item * max(1, len(items)))()
    for i, it in enumerate(items):
        arr[i] = rc_batch_item(it["session"], _ptr(it["latent"]), it["t"], it["mode"],
                               _ptr(it.get("dirty_idx")), it.get("D", 0),
                               _ptr(it.get("dirty_count")))
    _check(_lib.rc_step_batched(ctx, cache, arr, len(items), _stream(stream)))


def rc_step_capture(ctx, cache, session, latent, t, delta_ids, scores, stream=None):
    ids = np.ascontiguousarray(delta_ids, np.int32)
    _check(_lib.rc_step_capture(ctx, cache, session, _ptr(latent), t, ids.ctypes.data, len(ids),
                                _ptr(scores), _stream(stream)))


def rc_prompt_similarity(e_minus, e_plus):
    a = np.ascontiguousarray(e_minus, np.float32)
    b = np.ascontiguousarray(e_plus, np.float32)
    if a.shape != b.shape:
        raise ValueError("embeddings of different sizes")
    out = C.c_float()
    _check(_lib.rc_prompt_similarity(a.ctypes.data, b.ctypes.data, a.size, C.byref(out)))
    return out.value


def rc_reuse_schedule(s, tau_s, T, rho=0.2):
    modes = np.zeros(T, np.uint8)
    _check(_lib.rc_reuse_schedule(s, tau_s, rho, T, modes.ctypes.data))
    return modes


def rc_step_dense(ctx, cache, session, latent, t, stream=None):
    _check(_lib.rc_step_dense(ctx, cache, session, _ptr(latent), t, _stream(stream)))


def rc_linear(ctx, x, W, b, y, rows, n, k, stream=None):
    _check(_lib.rc_linear(ctx, _ptr(x), _ptr(W), _ptr(b), _ptr(y), rows, n, k, _stream(stream)))


def rc_attention(ctx, Q, ldq, K, V, ldkv, Nq, Nk, O, ldo, stream=None):
    _check(_lib.rc_attention(ctx, _ptr(Q), ldq, _ptr(K), _ptr(V), ldkv, Nq, Nk, _ptr(O), ldo,
                             _stream(stream)))


def rc_selftest_wait(ctx, timeout_us, set_flag, stream=None):
    _check(_lib.rc_selftest_wait(ctx, timeout_us, 1 if set_flag else 0, _stream(stream)))


def rc_sync(ctx, stream=None):
    _check(_lib.rc_sync(ctx, _stream(stream)))


RC_PROBE_OFF, RC_PROBE_GEMM, RC_PROBE_ATTENTION, RC_PROBE_LN = 0, 1, 2, 3


def rc_probe_enable(ctx, which, capacity):
    _check(_lib.rc_probe_enable(ctx, which, capacity))


def rc_probe_read(ctx):
    ms, n = C.c_double(), C.c_int()
    _check(_lib.rc_probe_read(ctx, C.byref(ms), C.byref(n)))
    return ms.value, n.value


def rc_probe_read_each(ctx, capacity):
    """Per-launch device times (ms, launch order) of the recorded launches."""
    buf = (C.c_float * max(1, capacity))()
    n = C.c_int()
    _check(_lib.rc_probe_read_each(ctx, buf, capacity, C.byref(n)))
    return [buf[i] for i in range(min(n.value, capacity))]


def rc_launch_count() -> int:
    return int(_lib.rc_launch_count())


def rc_status_string(s) -> str:
    return _lib.rc_status_string(s).decode()


def rc_last_error() -> str:
    return _lib.rc_last_error().decode()


# ------------------------------------------------------- convenience wrapper
def dims_struct(d, max_batch: int = 1) -> rc_dims:
    return rc_dims(d.hidden, d.heads, d.mlp, d.layers, d.grid_h, d.grid_w, d.patch, d.in_ch,
                   d.out_ch, d.text_len, d.timesteps, d.freq_dim, max_batch)


class Model:
    """Owns a context, device copies of the weights (kept alive here) and a
    cache; thin sugar over the entry points for tests and the benchmark."""

    def __init__(self, dims, weights, sessions=1, device="cuda", max_batch=1, host_cache=False):
        self.dims = dims
        self.w = weights.to(device)
        self.ctx = rc_create(dims_struct(dims, max_batch))
        for l, L in enumerate(self.w.layers):
            rc_set_layer_weights(self.ctx, l, L)
        g = dict(self.w.glob)
        g["pos"] = self.w.pos
        rc_set_global_weights(self.ctx, g)
        self.cache = (rc_cache_create_host if host_cache else rc_cache_create)(self.ctx, sessions)

    def close(self):
        if self.cache:
            rc_cache_destroy(self.cache)
            self.cache = None
        if self.ctx:
            rc_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
