"""The rule that decides which sampled-target differences the GPU parity tests accept."""
import numpy as np

from nucleus_flips import flip_explained
from oracle import sampling as OS


def _logits(seed, V=300):
    r = np.random.default_rng(seed)
    return (r.standard_normal(V) * 1.3).astype(np.float32)


def test_every_flip_from_a_small_perturbation_is_explained():
    """Perturb the logits by <= 2e-3 (the tiny model's error against the oracle): every
    pick that changes must be explained, and some do change (the rule is exercised)."""
    flips = 0
    for trial in range(400):
        l = _logits(trial)
        noise = np.random.default_rng(10_000 + trial).uniform(-2e-3, 2e-3, l.size).astype(np.float32)
        lg = (l + noise).astype(np.float32)
        for T, top_p, top_k in ((0.2, 0.95, 0), (1.0, 0.95, 10)):
            pos = 100 + trial
            o = OS.select(l, T, top_p, 77, pos, 0, top_k)[0]
            g = OS.select(lg, T, top_p, 77, pos, 0, top_k)[0]
            ok, info = flip_explained(l, lg, T, top_p, top_k, 77, pos, 0, o, g)
            assert ok, info
            flips += int(o != g)
    assert flips > 0


def test_a_flip_far_from_the_draw_is_not_explained():
    """Identical logits leave no room for a different pick; nor does a tiny error allow a
    pick several kept ids away from the draw."""
    l = _logits(3)
    T, p = 1.0, 0.95
    pos = 500
    o = OS.select(l, T, p, 5, pos, 0)[0]
    W, _ = OS.int_weights(l, T)
    kept = np.sort(OS.kept_set(W, p))
    assert kept.size > 3
    far = int(kept[(int(np.searchsorted(kept, o)) + kept.size // 2) % kept.size])
    ok, _ = flip_explained(l, l, T, p, 0, 5, pos, 0, o, far)
    assert not ok
    lg = (l + np.float32(1e-5)).astype(np.float32)
    ok, _ = flip_explained(l, lg, T, p, 0, 5, pos, 0, o, far)
    assert not ok
    # a pick outside the kept set is never explained
    outside = int(np.setdiff1d(np.arange(l.size), kept)[0])
    ok, _ = flip_explained(l, l, T, p, 0, 5, pos, 0, o, outside)
    assert not ok
