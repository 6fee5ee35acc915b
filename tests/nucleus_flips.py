"""When may a sampled target differ between the GPU and the oracle?

Both sides apply the same sampler (Sec. 2.1.2; the exact definition in oracle/sampling.py)
to their own logits, and the draw u = r / 2^64 is the same number on both sides (it depends
only on the seed, the produced position and the sequence).  The pick is the first kept id,
in ascending id order, whose cumulative weight fraction F exceeds u.  So when the logits
differ by at most e, the picks can differ only if u lies within the largest change of F
that an error e can cause of some boundary between the two picks:

  * every weight w_i = exp((l_i - max) / T) moves by a factor within exp(+-2e/T), so with
    eta = exp(2e/T) - 1 a cumulative fraction moves by at most 2 eta / (1 - eta);
  * ids that enter or leave the kept set (the top-p cut) move F by at most their mass;
  * the integer weights floor(w 2^24) add at most 2^-24 per kept id.

flip_explained() checks that condition for one row; a flip it cannot explain is a bug
(the logits tolerance alone would not catch an error that moves many samples).
"""
from __future__ import annotations

import math

import numpy as np

from oracle import sampling as OS


def _pick(W, kept, u):
    c = np.cumsum(W[kept].astype(np.float64))
    S = c[-1] if len(c) else 0.0
    if S <= 0:
        return int(kept[-1]), np.zeros(len(kept)), S
    F = c / S
    i = int(np.searchsorted(F, u, side="right"))
    return int(kept[min(i, len(kept) - 1)]), F, S


def flip_explained(l_ref, l_gpu, temperature, top_p, top_k, seed, position, seq, t_ref=None, t_gpu=None):
    """(explained, detail) for a row whose sampled targets differ: t_ref from the oracle's
    logits l_ref, t_gpu from the GPU's logits l_gpu (both default to the sampler's picks)."""
    l_ref = np.asarray(l_ref, dtype=np.float32)
    l_gpu = np.asarray(l_gpu, dtype=np.float32)
    W_ref, _ = OS.int_weights(l_ref, temperature)
    W_gpu, _ = OS.int_weights(l_gpu, temperature)
    k_ref = np.sort(OS.kept_set(W_ref, top_p, top_k))
    k_gpu = np.sort(OS.kept_set(W_gpu, top_p, top_k))
    u = OS.draw64(seed, position, seq) / 2.0 ** 64
    o, F, S = _pick(W_ref, k_ref, u)
    g, _, _ = _pick(W_gpu, k_gpu, u)
    o = o if t_ref is None else int(t_ref)
    g = g if t_gpu is None else int(t_gpu)
    if o not in set(k_ref.tolist()) or g not in set(k_gpu.tolist()):
        return False, dict(reason="a pick outside its kept set", o=o, g=g)
    e = float(np.max(np.abs(l_gpu.astype(np.float64) - l_ref.astype(np.float64))))
    eta = math.expm1(2.0 * e / temperature)
    changed = np.setxor1d(k_ref, k_gpu)
    delta = 2.0 * eta / max(1e-12, 1.0 - eta) + float(W_ref[changed].astype(np.float64).sum()) / max(S, 1.0)
    delta += len(k_ref) * 2.0 ** -24
    if g == o:
        return True, dict(u=u, delta=delta)
    if g > o:
        # the GPU passed every ref-kept id below g: F_gpu <= u there, F_ref > u from o on
        j = int(np.searchsorted(k_ref, g, side="left")) - 1         # the last ref-kept id < g
        boundary = F[j]
    else:
        # the GPU stopped at g: F_gpu(g) > u, while F_ref <= u up to the last ref-kept id <= g
        j = int(np.searchsorted(k_ref, g, side="right")) - 1
        boundary = F[j] if j >= 0 else 0.0
    return abs(boundary - u) <= delta, dict(u=u, boundary=boundary, delta=delta, e=e, o=o, g=g)
