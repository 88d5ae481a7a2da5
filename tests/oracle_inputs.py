"""Helpers that turn seeded synthetic inputs into the oracle's float64 arrays."""
import numpy as np

import oracle as O
from paper_2608_29809_gb300 import synth


def weights64(w: "synth.Weights"):
    layers = [{k: O.to64(v) for k, v in L.items()} for L in w.layers]
    G = {k: O.to64(v) for k, v in w.glob.items()}
    return layers, G, O.to64(w.pos)


def small_problem(d: "synth.Dims", seed: int):
    """Weights, a text context, one cache slice and block inputs, all float64."""
    w = synth.make_weights(d, seed)
    layers, G, pos = weights64(w)
    ctx = O.to64(synth.make_text(d, seed))
    H, K, V = (O.to64(t) for t in synth.make_cache_slice(d, seed, 0, 0, 0))
    x = O.to64(synth.make_hidden(d, seed))
    m6 = O.to64(synth.make_mod6(d, w.layers[0]["table"], seed))
    return dict(w=w, layers=layers, G=G, pos=pos, ctx=ctx, cache={"H": H, "K": K, "V": V},
                x=x, m6=m6)


def rng(seed):
    return np.random.default_rng(seed)
