"""Seeded synthetic workloads for the region-sparse DiT step.

This module only draws inputs: weights of a PixArt-alpha-shaped DiT, cached
hidden/K/V states, text contexts, latents, cross-attention score maps and
dirty-region masks.  It holds none of the method's arithmetic (no layer norm,
attention, localisation or scheduling); both the CUDA path and the oracle
consume what it returns.

All random draws go through ``torch.Generator`` seeded per tensor, so a tensor
is reproducible on its own regardless of the order in which tensors are drawn.
Weight matrices are stored as bf16 (the CUDA path's storage type); biases,
modulation tables and the positional table are fp32.  The oracle reads the
same values upcast to float64.

Shapes follow PixArt-alpha at 512 px / 1024 px (hidden 1152, 16 heads of 72,
MLP 4608, 28 blocks, patch 2, 4 latent channels, 8 output channels, 120 text
tokens); the paper's workloads (Section 4.1) are multi-turn edits whose
unchanged region covers most of the image, so masks are compact blobs.
"""
from __future__ import annotations

import math
import zlib
from dataclasses import dataclass, field

import numpy as np
import torch


@dataclass(frozen=True)
class Dims:
    hidden: int = 1152
    heads: int = 16
    mlp: int = 4608
    layers: int = 28
    grid_h: int = 64
    grid_w: int = 64
    patch: int = 2
    in_ch: int = 4
    out_ch: int = 8
    text_len: int = 120
    timesteps: int = 20
    freq_dim: int = 256

    @property
    def head_dim(self) -> int:
        return self.hidden // self.heads

    @property
    def tokens(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def patch_dim(self) -> int:
        return self.in_ch * self.patch * self.patch

    @property
    def final_dim(self) -> int:
        return self.patch * self.patch * self.out_ch

    @property
    def latent_shape(self) -> tuple:
        return (self.in_ch, self.grid_h * self.patch, self.grid_w * self.patch)


PIXART_512 = Dims(grid_h=32, grid_w=32)
PIXART_1024 = Dims(grid_h=64, grid_w=64)
PIXART_2048 = Dims(grid_h=128, grid_w=128)
ONE_BLOCK_256 = Dims(grid_h=16, grid_w=16, layers=1)
TINY = Dims(hidden=64, heads=4, mlp=256, layers=2, grid_h=4, grid_w=4, text_len=8,
            timesteps=4, freq_dim=32)

MODE_DENSE, MODE_SPARSE, MODE_REUSE = 0, 1, 2

LAYER_MATS = ("W_qkv", "W_o", "W_xq", "W_xkv", "W_xo", "W_1", "W_2")
LAYER_VECS = ("b_qkv", "b_o", "b_xq", "b_xkv", "b_xo", "b_1", "b_2", "table")
GLOBAL_MATS = ("W_e", "W_t1", "W_t2", "W_tb", "W_f")
GLOBAL_VECS = ("b_e", "b_t1", "b_t2", "b_tb", "table_f", "b_f")


def tensor_seed(base: int, *tags) -> int:
    """Deterministic 63-bit seed for one named tensor."""
    h = zlib.crc32(repr((int(base),) + tuple(tags)).encode())
    return (int(base) * 1_000_003 + h) & ((1 << 62) - 1)


def _gen(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def randn(shape, seed: int, device="cpu", std: float = 1.0, dtype=torch.float32):
    g = _gen(device, seed)
    t = torch.randn(tuple(shape), generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def uniform(shape, seed: int, device="cpu", lo: float = 0.0, hi: float = 1.0):
    g = _gen(device, seed)
    t = torch.rand(tuple(shape), generator=g, device=device, dtype=torch.float32)
    return t.mul_(hi - lo).add_(lo)


def layer_shapes(d: Dims) -> dict:
    h, f = d.hidden, d.mlp
    return {
        "W_qkv": (3 * h, h), "b_qkv": (3 * h,),
        "W_o": (h, h), "b_o": (h,),
        "W_xq": (h, h), "b_xq": (h,),
        "W_xkv": (2 * h, h), "b_xkv": (2 * h,),
        "W_xo": (h, h), "b_xo": (h,),
        "W_1": (f, h), "b_1": (f,),
        "W_2": (h, f), "b_2": (h,),
        "table": (6, h),
    }


def global_shapes(d: Dims) -> dict:
    h = d.hidden
    return {
        "W_e": (h, d.patch_dim), "b_e": (h,),
        "W_t1": (h, d.freq_dim), "b_t1": (h,),
        "W_t2": (h, h), "b_t2": (h,),
        "W_tb": (6 * h, h), "b_tb": (6 * h,),
        "table_f": (2, h),
        "W_f": (d.final_dim, h), "b_f": (d.final_dim,),
    }


@dataclass
class Weights:
    """Linear weights are [out][in] (y = x W^T + b), bf16; vectors fp32."""
    dims: Dims
    layers: list = field(default_factory=list)   # list of dict name -> tensor
    glob: dict = field(default_factory=dict)
    pos: torch.Tensor | None = None              # [N][hidden] fp32

    def to(self, device):
        return Weights(self.dims,
                       [{k: v.to(device) for k, v in L.items()} for L in self.layers],
                       {k: v.to(device) for k, v in self.glob.items()},
                       None if self.pos is None else self.pos.to(device))


def sincos_pos_table(d: Dims) -> torch.Tensor:
    """Fixed 2-D sin-cos positional table [N][hidden] (row-major grid y*W+x).

    Half of the channels encode the row coordinate, half the column; each half
    is [sin(p*w_k), cos(p*w_k)] with w_k = 10000^(-k/(hidden/4)).
    """
    quarter = d.hidden // 4
    omega = 1.0 / (10000.0 ** (np.arange(quarter, dtype=np.float64) / quarter))
    ys, xs = np.meshgrid(np.arange(d.grid_h, dtype=np.float64),
                         np.arange(d.grid_w, dtype=np.float64), indexing="ij")

    def enc(p):
        a = p.reshape(-1)[:, None] * omega[None, :]
        return np.concatenate([np.sin(a), np.cos(a)], axis=1)

    table = np.concatenate([enc(ys), enc(xs)], axis=1)
    return torch.from_numpy(table.astype(np.float32))


def make_weights(d: Dims, seed: int, device="cpu", std: float = 0.02) -> Weights:
    """Random-init weights of a PixArt-alpha-shaped DiT (Section 4.1 backbone).

    Matrices ~ N(0, std) rounded to bf16; biases ~ std * N(0, 1);
    modulation tables ~ N(0, std).
    """
    w = Weights(d)
    for l in range(d.layers):
        L = {}
        for name, shp in layer_shapes(d).items():
            dt = torch.bfloat16 if name.startswith("W_") else torch.float32
            L[name] = randn(shp, tensor_seed(seed, "layer", l, name), device, std, dt)
        w.layers.append(L)
    for name, shp in global_shapes(d).items():
        dt = torch.bfloat16 if name.startswith("W_") else torch.float32
        w.glob[name] = randn(shp, tensor_seed(seed, "global", name), device, std, dt)
    w.pos = sincos_pos_table(d).to(device)
    return w


def make_mod6(d: Dims, table: torch.Tensor, seed: int, noise: float = 0.1):
    """A 6 x hidden modulation vector: the layer table plus a random timestep
    embedding contribution (noise * N(0, 1))."""
    return table.float() + randn((6, d.hidden), tensor_seed(seed, "mod6"), table.device, noise)


def make_text(d: Dims, seed: int, device="cpu") -> torch.Tensor:
    """Text context [text_len][hidden] ~ N(0, 1), bf16."""
    return randn((d.text_len, d.hidden), tensor_seed(seed, "text"), device, 1.0, torch.bfloat16)


def make_latent(d: Dims, seed: int, device="cpu") -> torch.Tensor:
    return randn(d.latent_shape, tensor_seed(seed, "latent"), device)


def make_cache_slice(d: Dims, seed: int, session: int, layer: int, t: int, device="cpu",
                     dtype=torch.bfloat16):
    """Previous-turn cached (H, K, V) for one (layer, t): each [N][hidden] ~ N(0, 1)."""
    return tuple(randn((d.tokens, d.hidden), tensor_seed(seed, "cache", session, layer, t, k),
                       device, 1.0, dtype) for k in ("H", "K", "V"))


def make_hidden(d: Dims, seed: int, device="cpu", n: int | None = None) -> torch.Tensor:
    return randn((d.tokens if n is None else n, d.hidden), tensor_seed(seed, "hidden"), device)


# ----------------------------------------------------------------- schedules
def ddim_tables(T: int, train_steps: int = 1000, beta0: float = 1e-4, beta1: float = 0.02):
    """Timestep values (linear grid train_steps-1 .. 0 with T entries) and the
    matching cumulative alphas of a linear-beta schedule; alpha_bar[T] = 1."""
    betas = np.linspace(beta0, beta1, train_steps, dtype=np.float64)
    abar = np.cumprod(1.0 - betas)
    tv = np.round(np.linspace(train_steps - 1, 0, T)).astype(np.int64)
    ab = np.concatenate([abar[tv], [1.0]])
    return tv.astype(np.float32), ab.astype(np.float32)


# --------------------------------------------------------------------- masks
def rectangle_mask(d: Dims, seed: int, area=(35, 42)) -> np.ndarray:
    """One axis-aligned rectangle whose area lies in ``area`` (inclusive)."""
    rng = np.random.default_rng(tensor_seed(seed, "rect"))
    cands = [(h, w) for h in range(1, d.grid_h + 1) for w in range(1, d.grid_w + 1)
             if area[0] <= h * w <= area[1]]
    h, w = cands[rng.integers(len(cands))]
    y0 = rng.integers(0, d.grid_h - h + 1)
    x0 = rng.integers(0, d.grid_w - w + 1)
    m = np.zeros((d.grid_h, d.grid_w), np.uint8)
    m[y0:y0 + h, x0:x0 + w] = 1
    return m.reshape(-1)


def _ellipses(d: Dims, rng, k: int):
    out = []
    for _ in range(k):
        cy, cx = rng.uniform(0, d.grid_h), rng.uniform(0, d.grid_w)
        ratio = rng.uniform(0.5, 2.0)
        theta = rng.uniform(0, math.pi)
        out.append((cy, cx, ratio, theta))
    return out


def _raster(d: Dims, ell, scale: float) -> np.ndarray:
    ys, xs = np.meshgrid(np.arange(d.grid_h) + 0.5, np.arange(d.grid_w) + 0.5, indexing="ij")
    m = np.zeros((d.grid_h, d.grid_w), bool)
    for cy, cx, ratio, theta in ell:
        a, b = scale * math.sqrt(ratio), scale / math.sqrt(ratio)
        dy, dx = ys - cy, xs - cx
        u = dx * math.cos(theta) + dy * math.sin(theta)
        v = -dx * math.sin(theta) + dy * math.cos(theta)
        m |= (u / a) ** 2 + (v / b) ** 2 <= 1.0
    return m


def ellipse_blobs(d: Dims, seed: int, frac: float, n_blobs: int | None = None, tol=0.005):
    """Union of 1-3 seeded ellipses, scaled by bisection until the covered
    fraction is within ``tol`` of ``frac``.  Returns one boolean [N] map per
    ellipse (their union is the region)."""
    rng = np.random.default_rng(tensor_seed(seed, "ellipses", round(frac * 1e4)))
    k = int(rng.integers(1, 4)) if n_blobs is None else n_blobs
    ell = _ellipses(d, rng, k)
    lo, hi = 0.0, 2.0 * max(d.grid_h, d.grid_w)
    best = None
    for _ in range(80):
        mid = 0.5 * (lo + hi)
        f = _raster(d, ell, mid).mean()
        best = mid
        if abs(f - frac) <= tol:
            break
        if f < frac:
            lo = mid
        else:
            hi = mid
    return [_raster(d, [e], best).reshape(-1) for e in ell]


def indicator_scores(d: Dims, blobs, seed: int, M: int | None = None):
    """Cross-attention score map [1][N][M] fp32 in which delta column j_k is
    high (U(0.6, 1)) inside blob k and low (U(0, 0.4)) outside; every other
    column is U(0, 1).  Returns (scores, delta_ids)."""
    M = d.text_len if M is None else M
    rng = np.random.default_rng(tensor_seed(seed, "indicator"))
    N = d.tokens
    A = rng.uniform(0.0, 1.0, size=(N, M)).astype(np.float32)
    ids = rng.choice(M, size=len(blobs), replace=False).astype(np.int32)
    for j, b in zip(ids, blobs):
        col = rng.uniform(0.0, 0.4, size=N)
        col[b] = rng.uniform(0.6, 1.0, size=int(b.sum()))
        A[:, j] = col.astype(np.float32)
    return A[None], ids


def blob_scores(d: Dims, seed: int, n_delta=(3, 8), sigma=(1.2, 2.6), amp=6.0):
    """Random cross-attention map [1][N][M] (logits ~ N(0,1) plus a Gaussian
    bump of height ``amp`` per delta token at a uniform centre, then a row
    softmax over the M text tokens), and 3-8 distinct delta token ids."""
    rng = np.random.default_rng(tensor_seed(seed, "blobscores"))
    N, M = d.tokens, d.text_len
    logits = rng.standard_normal((N, M))
    k = int(rng.integers(n_delta[0], n_delta[1] + 1))
    ids = rng.choice(M, size=k, replace=False).astype(np.int32)
    ys, xs = np.meshgrid(np.arange(d.grid_h), np.arange(d.grid_w), indexing="ij")
    ys, xs = ys.reshape(-1), xs.reshape(-1)
    for j in ids:
        cy, cx = rng.uniform(0, d.grid_h), rng.uniform(0, d.grid_w)
        s = rng.uniform(*sigma)
        logits[:, j] += amp * np.exp(-((ys - cy) ** 2 + (xs - cx) ** 2) / (2 * s * s))
    e = np.exp(logits - logits.max(axis=1, keepdims=True))
    A = (e / e.sum(axis=1, keepdims=True)).astype(np.float32)
    return A[None], ids


def similarity(seed: int, turn: int) -> float:
    """Seeded prompt-similarity scalar s in [0, 1] for one editing turn."""
    rng = np.random.default_rng(tensor_seed(seed, "similarity", turn))
    return float(rng.uniform(0.0, 1.0))


def turn_dirty_fraction(seed: int, turn: int, lo: float = 0.05, hi: float = 0.20) -> float:
    """Seeded target dirty fraction of one editing turn's mask, U(lo, hi)."""
    rng = np.random.default_rng(tensor_seed(seed, "turn_fraction", turn))
    return float(rng.uniform(lo, hi))
