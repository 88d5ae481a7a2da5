"""Shared set-up of the GPU parity tests: seeded problems loaded into the
library and into the oracle, and the tolerance checks."""
import numpy as np
import torch

import oracle as O
from paper_2608_29809_gb300 import synth
from tests.oracle_inputs import weights64

# Tolerances: per-block outputs max-abs <= 3e-2 x output RMS and cosine >=
# 0.999; end-of-step latent relative L2 <= 1e-2.
BLOCK_MAXABS_REL = 3e-2
BLOCK_COS = 0.999
LATENT_REL_L2 = 1e-2


def block_close(got, ref, what=""):
    got = np.asarray(got, np.float64).reshape(-1)
    ref = np.asarray(ref, np.float64).reshape(-1)
    rms = np.sqrt(np.mean(ref ** 2))
    maxabs = np.max(np.abs(got - ref)) if ref.size else 0.0
    cos = float(got @ ref / (np.linalg.norm(got) * np.linalg.norm(ref))) if ref.size else 1.0
    assert maxabs <= BLOCK_MAXABS_REL * rms, f"{what}: max|err| {maxabs:.3e} > 3e-2 x rms {rms:.3e}"
    assert cos >= BLOCK_COS, f"{what}: cosine {cos:.6f} < 0.999"
    return maxabs / rms, cos


def rel_l2(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.linalg.norm(got - ref) / np.linalg.norm(ref))


class Problem:
    """Weights, text and per-(layer, t) cache for one session, on both sides."""

    def __init__(self, R, d: "synth.Dims", seed: int, ts=(0,)):
        self.R, self.d, self.seed = R, d, seed
        w = synth.make_weights(d, seed)
        self.model = R.Model(d, w)
        self.layers64, self.G64, self.pos64 = weights64(w)
        self.text = synth.make_text(d, seed)
        R.rc_set_text(self.model.ctx, self.model.cache, 0, self.text.cuda())
        ctx64 = O.to64(self.text)
        self.tkv64 = [O.text_kv(ctx64, L) for L in self.layers64]
        tv, ab = synth.ddim_tables(d.timesteps)
        self.tv, self.ab = tv, ab
        R.rc_set_schedule(self.model.ctx, tv, ab)
        self.cache64 = {}
        for t in ts:
            for l in range(d.layers):
                H, K, V = synth.make_cache_slice(d, seed, 0, l, t)
                R.rc_cache_fill(self.model.cache, 0, l, t, H.cuda(), K.cuda(), V.cuda())
                self.cache64[(l, t)] = {"H": O.to64(H), "K": O.to64(K), "V": O.to64(V)}
        torch.cuda.synchronize()

    def read_slot(self, l, t):
        n, h = self.d.tokens, self.d.hidden
        H, K, V = (torch.empty(n, h, dtype=torch.bfloat16, device="cuda") for _ in range(3))
        self.R.rc_cache_read(self.model.cache, 0, l, t, H, K, V)
        torch.cuda.synchronize()
        return {"H": O.to64(H.cpu()), "K": O.to64(K.cpu()), "V": O.to64(V.cpu())}

    def oracle_step(self, latent64, t, mode, idx):
        cache_t = [self.cache64[(l, t)] for l in range(self.d.layers)]
        return O.step(self.G64, self.layers64, self.pos64, latent64, t, mode, idx, cache_t,
                      self.tkv64, self.tv.astype(np.float64), self.ab.astype(np.float64),
                      self.d.heads, self.d.grid_h, self.d.grid_w, self.d.patch, self.d.in_ch)

    def close(self):
        self.model.close()
