"""Oracle of RegionCache's region-sparse DiT denoising step, in float64 numpy.

TEST INFRASTRUCTURE ONLY: the product path never imports this module.  It is
the plain, slow statement of what the CUDA library computes, written from the
paper and checked by the pins under ``tests/test_oracle_*.py``.

What it follows:
  * Section 3.2, "Prompt-aligned Region Caching": the edit region is the set of
    image tokens i with a_j(i) >= theta_j for a new/modified text token j,
    where a_j aggregates that token's cross-attention column.  Readings: the
    aggregate over S score slices is their mean; theta_j is `threshold` after
    a per-token min-max normalisation; several delta tokens are united; the
    region is dilated on the token grid (Chebyshev radius `dilation`).  These
    decisions are taken in float32, the precision the CUDA kernel uses.
  * Section 3.2, "Hidden-State-Oriented Caching": a cache pool of hidden
    states per (layer, timestep) along the denoising trajectory.
  * Section 3.3, "Region-Level Sparse Attention": only active (dirty) tokens
    become queries; keys/values cover every token; inactive tokens' next
    hidden state is read from the cache and merged with the active outputs.
  * Section 3.4, "Kernel Fusing": keys/values are refreshed for active tokens
    only and the cached ones are reused for the rest.
  * Section 3.3, Eq. 1 and Eq. 2: similarity s = cos(e(tau-), e(tau+)) and the
    reuse cutoff T_reuse = T if s >= tau_s else floor(rho T).
  * Section 4.1 names PixArt-alpha as the backbone; the paper does not write
    out the block.  Reading: adaLN-single block = LayerNorm (no affine, eps
    1e-6) -> modulate x(1+scale)+shift -> self-attention (gate_msa) -> text
    cross-attention (no norm, no gate) -> LayerNorm -> modulate -> MLP with
    tanh-GELU (gate_mlp); a T2I final layer (norm, modulate with the timestep
    embedding, linear to p*p*out_ch) and a DDIM (eta = 0) update of the latent.

Linear layers use the [out][in] convention: y = x W^T + b.  Column block
h*dh .. h*dh+dh-1 of q, k and v is head h.
"""
from __future__ import annotations

import math

import numpy as np

LN_EPS = 1e-6
MODE_DENSE, MODE_SPARSE, MODE_REUSE = 0, 1, 2


def to64(x) -> np.ndarray:
    """float64 numpy copy of a numpy array or a (CPU) torch tensor."""
    if hasattr(x, "detach"):
        x = x.detach().to("cpu")
        if str(x.dtype) == "torch.bfloat16":
            x = x.float()
        x = x.numpy()
    return np.array(x, dtype=np.float64, copy=True)


# --------------------------------------------------------------- block pieces
def linear(x, W, b=None):
    """y = x W^T (+ b), W stored [out][in]."""
    y = x @ W.T
    return y if b is None else y + b


def layer_norm(x, eps=LN_EPS):
    """Row LayerNorm without affine parameters, biased variance."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def modulate(y, shift, scale):
    """adaLN modulation y * (1 + scale) + shift."""
    return y * (1.0 + scale) + shift


def gelu_tanh(z):
    """GELU with the tanh approximation."""
    return 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))


def silu(z):
    return z / (1.0 + np.exp(-z))


def softmax(s):
    """Softmax over the last axis."""
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def multihead_attention(q, k, v, heads):
    """softmax(q_h k_h^T / sqrt(dh)) v_h per head; q [Nq][h*dh], k,v [Nk][h*dh]."""
    dh = q.shape[1] // heads
    out = np.empty((q.shape[0], v.shape[1]))
    for h in range(heads):
        c = slice(h * dh, (h + 1) * dh)
        p = softmax((q[:, c] @ k[:, c].T) / math.sqrt(dh))
        out[:, c] = p @ v[:, c]
    return out


def split6(m6):
    """(shift_msa, scale_msa, gate_msa, shift_mlp, scale_mlp, gate_mlp)."""
    return tuple(m6[i] for i in range(6))


def text_kv(ctx, Lw):
    """Per-layer text keys/values of the cross-attention: ctx W_xkv^T + b,
    first `hidden` outputs are K, the next `hidden` are V."""
    kv = linear(ctx, Lw["W_xkv"], Lw["b_xkv"])
    d = kv.shape[1] // 2
    return kv[:, :d], kv[:, d:]


def cross_attention(x, tk, tv, Lw, heads):
    """Text cross-attention output (added to x by the caller)."""
    q = linear(x, Lw["W_xq"], Lw["b_xq"])
    return linear(multihead_attention(q, tk, tv, heads), Lw["W_xo"], Lw["b_xo"])


def cross_attention_maps(x, tk, Lw, heads):
    """The cross-attention matrices of one block, one per head (Section 3.2:
    A in R^{N x M} links image tokens to text tokens): softmax over the M text
    tokens of q'_h k_h^T / sqrt(dh), q' = x W_xq^T + b.  Returns [heads][N][M]."""
    q = linear(x, Lw["W_xq"], Lw["b_xq"])
    dh = q.shape[1] // heads
    out = np.empty((heads, q.shape[0], tk.shape[0]))
    for h in range(heads):
        c = slice(h * dh, (h + 1) * dh)
        out[h] = softmax((q[:, c] @ tk[:, c].T) / math.sqrt(dh))
    return out


def mlp_branch(x, Lw, shift, scale):
    a = modulate(layer_norm(x), shift, scale)
    return linear(gelu_tanh(linear(a, Lw["W_1"], Lw["b_1"])), Lw["W_2"], Lw["b_2"])


def qkv_rows(x, Lw, shift, scale):
    a = modulate(layer_norm(x), shift, scale)
    qkv = linear(a, Lw["W_qkv"], Lw["b_qkv"])
    d = x.shape[1]
    return qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]


# ---------------------------------------------------------------- the blocks
def dense_block(x, Lw, m6, tkv, heads, want_maps=False):
    """Full recompute of one DiT block over all N tokens (the backbone block,
    Section 4.1 reading).  Returns (x_out, K, V), K/V post-bias [N][hidden],
    and with want_maps also the block's cross-attention matrices [heads][N][M]."""
    sh1, sc1, g1, sh2, sc2, g2 = split6(m6)
    q, k, v = qkv_rows(x, Lw, sh1, sc1)
    o = multihead_attention(q, k, v, heads)
    x = x + g1 * linear(o, Lw["W_o"], Lw["b_o"])
    maps = cross_attention_maps(x, tkv[0], Lw, heads) if want_maps else None
    x = x + cross_attention(x, tkv[0], tkv[1], Lw, heads)
    x = x + g2 * mlp_branch(x, Lw, sh2, sc2)
    return (x, k, v, maps) if want_maps else (x, k, v)


def region_block(x_dirty, idx, cache, Lw, m6, tkv, heads):
    """Region-level sparse block (Section 3.3 Region-Level Sparse Attention,
    Section 3.4 Kernel Fusing).

    x_dirty  [D][hidden]: block inputs of the active tokens, row r is token idx[r].
    cache    dict H, K, V of [N][hidden]: the previous turn's block output,
             keys and values of this (layer, timestep).
    Returns (cache_new, x_dirty_out): the updated cache (active rows of K, V and
    H replaced by fresh values, every other row as cached) and the active
    tokens' block outputs.  H of cache_new is the merged H^{l+1}.
    """
    idx = np.asarray(idx, dtype=np.int64)
    sh1, sc1, g1, sh2, sc2, g2 = split6(m6)
    K = np.array(cache["K"], dtype=np.float64, copy=True)
    V = np.array(cache["V"], dtype=np.float64, copy=True)
    H = np.array(cache["H"], dtype=np.float64, copy=True)
    if idx.size == 0:
        return {"H": H, "K": K, "V": V}, np.zeros((0, H.shape[1]))
    q, k, v = qkv_rows(x_dirty, Lw, sh1, sc1)        # Q_active and fresh K, V rows
    K[idx] = k                                       # active keys/values written to
    V[idx] = v                                       # their target rows
    o = multihead_attention(q, K, V, heads)          # Q_active against all of K^l, V^l
    x = x_dirty + g1 * linear(o, Lw["W_o"], Lw["b_o"])
    x = x + cross_attention(x, tkv[0], tkv[1], Lw, heads)
    x = x + g2 * mlp_branch(x, Lw, sh2, sc2)
    H[idx] = x                                       # merge with the cached inactive rows
    return {"H": H, "K": K, "V": V}, x


# --------------------------------------------------------------- localization
def localize_mask(A, delta_ids, grid_h, grid_w, threshold=0.5, dilation=1):
    """Edit region R_edit of Section 3.2 as a token mask and its index list.

    A: cross-attention scores [S][N][M] (float32); delta_ids: the new/modified
    text tokens j.  a_j = mean over the S slices (summed in ascending s, then
    divided by S); theta_j: a_j is min-max normalised and compared (>=) with
    `threshold`; a constant column, or one whose averaged scores hold a
    non-finite value (NaN, +-Inf: the normalisation is undefined there),
    contributes no token; the regions of all
    delta tokens are united and dilated by a (2r+1)x(2r+1) square on the
    grid, ignoring neighbours outside it.  All arithmetic is float32.
    Returns (mask u8 [N], idx int32 ascending).
    """
    A = np.asarray(A, dtype=np.float32)
    S, N, M = A.shape
    if N != grid_h * grid_w:
        raise ValueError("N must equal grid_h * grid_w")
    acc = A[0].copy()
    for s in range(1, S):
        acc = (acc + A[s]).astype(np.float32)
    abar = (acc / np.float32(S)).astype(np.float32)
    tau = np.float32(threshold)
    union = np.zeros(N, dtype=bool)
    for j in delta_ids:
        a = abar[:, int(j)]
        if not np.all(np.isfinite(a)):
            continue
        mn = np.float32(a.min())
        mx = np.float32(a.max())
        rng = np.float32(mx - mn)
        if not rng > np.float32(0):
            continue
        nrm = ((a - mn).astype(np.float32) / rng).astype(np.float32)
        union |= nrm >= tau
    g = union.reshape(grid_h, grid_w)
    out = np.zeros_like(g)
    for dy in range(-dilation, dilation + 1):
        for dx in range(-dilation, dilation + 1):
            ys, ye = max(0, -dy), min(grid_h, grid_h - dy)
            xs, xe = max(0, -dx), min(grid_w, grid_w - dx)
            if ys < ye and xs < xe:
                out[ys:ye, xs:xe] |= g[ys + dy:ye + dy, xs + dx:xe + dx]
    mask = out.reshape(-1).astype(np.uint8)
    return mask, np.flatnonzero(mask).astype(np.int32)


# -------------------------------------------------- timestep, patches, final
def timestep_embedding(t_value, dim, max_period=10000.0):
    """Sinusoidal embedding: [cos(t w_k), sin(t w_k)], w_k = P^(-k/(dim/2))."""
    half = dim // 2
    w = np.exp(-math.log(max_period) * np.arange(half, dtype=np.float64) / half)
    a = float(t_value) * w
    return np.concatenate([np.cos(a), np.sin(a)])


def t_embed(t_value, G):
    """Timestep MLP: Linear(freq -> hidden), SiLU, Linear(hidden -> hidden)."""
    f = timestep_embedding(t_value, G["W_t1"].shape[1])
    return linear(silu(linear(f, G["W_t1"], G["b_t1"])), G["W_t2"], G["b_t2"])


def t_block(temb, G):
    """adaLN-single: SiLU then Linear(hidden -> 6 hidden), as [6][hidden]."""
    return linear(silu(temb), G["W_tb"], G["b_tb"]).reshape(6, -1)


def patchify(latent, p):
    """[C][p*gh][p*gw] -> [N][C*p*p], patch vector ordered (c, py, px)."""
    C, Hh, Ww = latent.shape
    gh, gw = Hh // p, Ww // p
    return latent.reshape(C, gh, p, gw, p).transpose(1, 3, 0, 2, 4).reshape(gh * gw, C * p * p)


def unpatchify(out, gh, gw, p):
    """[N][p*p*C] with channel fastest -> [C][p*gh][p*gw]."""
    C = out.shape[1] // (p * p)
    return out.reshape(gh, gw, p, p, C).transpose(4, 0, 2, 1, 3).reshape(C, gh * p, gw * p)


def patch_embed(latent, rows, G, pos, p):
    """x_i = W_e patch_i + b_e + pos_i for the given token rows."""
    P = patchify(latent, p)[rows]
    return linear(P, G["W_e"], G["b_e"]) + pos[rows]


def final_layer(H, temb, G, gh, gw, p, in_ch):
    """T2I final layer on all tokens; returns eps = the first in_ch channels."""
    shift = G["table_f"][0] + temb
    scale = G["table_f"][1] + temb
    out = linear(modulate(layer_norm(H), shift, scale), G["W_f"], G["b_f"])
    return unpatchify(out, gh, gw, p)[:in_ch]


def ddim_update(x, eps, ab_t, ab_next):
    """DDIM with eta = 0: x0 = (x - sqrt(1-ab_t) eps)/sqrt(ab_t);
    x_next = sqrt(ab_next) x0 + sqrt(1-ab_next) eps."""
    x0 = (x - math.sqrt(1.0 - ab_t) * eps) / math.sqrt(ab_t)
    return math.sqrt(ab_next) * x0 + math.sqrt(1.0 - ab_next) * eps


# ----------------------------------------------------------------------- step
def step(G, layers, pos, latent, t, mode, idx, cache_t, tkv_layers, t_values, alpha_bar,
         heads, grid_h, grid_w, patch, in_ch):
    """One denoising step of the region-sparse DiT.

    layers: per-layer weight dicts; cache_t: list over layers of dict H, K, V
    [N][hidden] at this timestep (not modified; updated copies are returned).
    mode: DENSE (every token recomputed, cache rows overwritten), SPARSE (the
    tokens in idx recomputed), REUSE (no block runs; H^L comes from the cache).
    Returns (latent_next, eps, cache_t_new).
    """
    N = grid_h * grid_w
    temb = t_embed(t_values[t], G)
    tb = t_block(temb, G)
    new_cache = []
    if mode == MODE_REUSE:
        new_cache = [{k: np.array(v, dtype=np.float64, copy=True) for k, v in c.items()}
                     for c in cache_t]
    else:
        rows = np.arange(N) if mode == MODE_DENSE else np.asarray(idx, dtype=np.int64)
        x = patch_embed(latent, rows, G, pos, patch)
        for l, Lw in enumerate(layers):
            m6 = Lw["table"] + tb
            if mode == MODE_DENSE:
                x, K, V = dense_block(x, Lw, m6, tkv_layers[l], heads)
                new_cache.append({"H": x.copy(), "K": K, "V": V})
            else:
                c, x = region_block(x, rows, cache_t[l], Lw, m6, tkv_layers[l], heads)
                new_cache.append(c)
    H_last = new_cache[-1]["H"]
    eps = final_layer(H_last, temb, G, grid_h, grid_w, patch, in_ch)
    x_next = ddim_update(latent, eps, float(alpha_bar[t]), float(alpha_bar[t + 1]))
    return x_next, eps, new_cache


def step_capture(G, layers, pos, latent, t, cache_t, tkv_layers, t_values, alpha_bar, heads,
                 grid_h, grid_w, patch, in_ch, delta_ids, M):
    """A DENSE step that also returns the localisation scores of Section 3.2:
    for each delta (new or modified) text token j, its cross-attention scores
    aggregated over heads and layers, a_j = mean_{l,h} A^{l,h}[:, j].
    Returns (latent_next, eps, cache_t_new, scores [N][M]) with the delta
    columns filled and every other column zero (the layout the localisation
    takes with S = 1)."""
    N = grid_h * grid_w
    temb = t_embed(t_values[t], G)
    tb = t_block(temb, G)
    new_cache = []
    scores = np.zeros((N, M))
    ids = np.asarray(delta_ids, dtype=np.int64)
    x = patch_embed(latent, np.arange(N), G, pos, patch)
    for l, Lw in enumerate(layers):
        x, K, V, maps = dense_block(x, Lw, Lw["table"] + tb, tkv_layers[l], heads, want_maps=True)
        new_cache.append({"H": x.copy(), "K": K, "V": V})
        scores[:, ids] += maps[:, :, ids].sum(axis=0)
    scores[:, ids] /= len(layers) * heads
    eps = final_layer(new_cache[-1]["H"], temb, G, grid_h, grid_w, patch, in_ch)
    x_next = ddim_update(latent, eps, float(alpha_bar[t]), float(alpha_bar[t + 1]))
    return x_next, eps, new_cache, scores


def cached_localization_scores(G, layers, pos, latent, cache_t, tkv_layers, heads, grid_h,
                               grid_w, patch, delta_ids, M):
    """Localisation scores of Section 3.2 for a new editing turn, taken from
    the cached diffusion states instead of a dense step (so that a turn
    scheduled by Eq. 2 -- REUSE, then SPARSE -- can localise its edit before
    anything is recomputed).

    For each delta (new or modified) text token j and image token i,
    a_j(i) = mean over blocks l and heads h of the cross-attention
    probability of j, softmax over all M text tokens of
    q'_{l,h}(i) . k_{l,h,j'} / sqrt(dh), where the text keys k are the new
    turn's (ctx W_xkv^T + b) and the image queries q' = H^l W_xq^T + b_xq are
    computed from the hidden state entering block l as the cache holds it at
    this step: H^0 is the patch embedding of `latent` (the state entering the
    first block; the cache starts at block outputs), H^l for l >= 1 is the
    cached output of block l - 1.  (Reading: the paper aggregates A_t over
    heads and layers without naming the operator, taken as the mean; the
    cached block input stands in for the cross-attention input, which the
    cache does not hold.)
    Returns scores [N][M] with the delta columns filled and every other
    column zero (the [S = 1][N][M] layout the localisation takes)."""
    N = grid_h * grid_w
    ids = np.asarray(delta_ids, dtype=np.int64)
    scores = np.zeros((N, M))
    for l, Lw in enumerate(layers):
        h_in = patch_embed(latent, np.arange(N), G, pos, patch) if l == 0 else cache_t[l - 1]["H"]
        maps = cross_attention_maps(h_in, tkv_layers[l][0], Lw, heads)
        scores[:, ids] += maps[:, :, ids].sum(axis=0)
    scores[:, ids] /= len(layers) * heads
    return scores


# ------------------------------------------------------------------ schedules
def cosine_similarity(e_minus, e_plus):
    """Eq. 1: s = cos(e(tau-), e(tau+))."""
    e_minus, e_plus = np.asarray(e_minus, float), np.asarray(e_plus, float)
    return float(e_minus @ e_plus / (np.linalg.norm(e_minus) * np.linalg.norm(e_plus)))


def reuse_cutoff(s, tau_s, T, rho=0.2):
    """Eq. 2: T_reuse = T if s >= tau_s else floor(rho T)."""
    return T if s >= tau_s else int(math.floor(rho * T))


def schedule_eq2(s, tau_s, T, rho=0.2):
    """Per-step modes for an edited region under Eq. 2: cached states are
    reused (REUSE) for steps t < T_reuse, the region is recomputed (SPARSE)
    from T_reuse on."""
    tr = reuse_cutoff(s, tau_s, T, rho)
    return np.array([MODE_REUSE if t < tr else MODE_SPARSE for t in range(T)], np.uint8)


def k_from_similarity(s):
    """Number of fully recomputed leading steps of a turn, k in {2, 4, 6, 8},
    from a similarity s in [0, 1]: k = 2 (1 + min(3, floor(4 (1 - s))))."""
    return 2 * (1 + min(3, int(math.floor(4.0 * (1.0 - s)))))


def schedule_first_k_dense(k, T):
    """First k steps DENSE, the rest SPARSE."""
    return np.array([MODE_DENSE if t < k else MODE_SPARSE for t in range(T)], np.uint8)
