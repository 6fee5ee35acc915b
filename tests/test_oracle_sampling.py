"""Pins of the oracle's target selection (greedy and nucleus) to things other than itself."""
import itertools
import math
import os

import numpy as np
import pytest

from oracle import sampling as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_philox_known_answers():
    """Philox4x32-10 against the published known-answer vectors (Salmon et al., SC'11)."""
    n = 0
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            v = [int(x, 16) for x in line.split()]
            assert S.philox4x32_10(v[0:4], v[4:6]) == tuple(v[6:10])
            n += 1
    assert n == 3


def test_philox_uniformity():
    """Draws keyed by position look uniform: mean and a 16-bin chi^2 on the top bits."""
    r = np.array([S.draw64(1234, p, 0) for p in range(20000)], dtype=np.float64) / 2.0**64
    assert abs(r.mean() - 0.5) < 0.01
    counts = np.bincount((r * 16).astype(int), minlength=16)
    chi2 = ((counts - 1250.0) ** 2 / 1250.0).sum()
    assert chi2 < 40.0          # 15 dof: p ~ 5e-4


def test_exp_sd_accuracy():
    """exp_sd within 4 ulp of the exact e^s over the whole supported range."""
    s = np.concatenate([np.linspace(-87.0, 0.0, 400001, dtype=np.float32),
                        -np.logspace(-8, 1.9, 20000).astype(np.float32),
                        np.float32([0.0, -0.0, -1e-30, -math.log(2.0), -86.99])])
    got = S.exp_sd(s).astype(np.float64)
    ref = np.exp(s.astype(np.float64))
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    err = np.abs(got - ref) / ulp
    assert err.max() <= 4.0, err.max()
    assert S.exp_sd(np.float32([0.0]))[0] == np.float32(1.0)


def test_exp_sd_edges_and_monotone():
    s = np.float32([-87.5, -88.0, -np.inf, np.nan, -1000.0])
    assert np.all(S.exp_sd(s) == 0.0)
    g = np.sort(np.random.default_rng(0).uniform(-87, 0, 100000).astype(np.float32))
    e = S.exp_sd(g)
    assert np.all(np.diff(e.astype(np.float64)) >= 0.0)


def test_argmax_ties_and_nan():
    assert S.argmax_lowest(np.float32([1, 3, 3, 2]))[0] == 1
    idx, bad = S.argmax_lowest(np.float32([np.nan, 0.5, 0.7, np.nan]))
    assert idx == 2 and bad
    assert S.argmax_lowest(np.float32([-np.inf, -np.inf]))[0] == 0


def test_int_weights_top_is_2_24():
    l = np.random.default_rng(1).normal(0, 1.3, 500).astype(np.float32)
    W, _ = S.int_weights(l, 0.7)
    assert int(W.max()) == 1 << 24 and int(np.argmax(W)) == int(np.argmax(l))


def _brute_min_cardinality(W, p_fixed):
    """Smallest subset size whose weight C satisfies C * 2^24 >= P * S (exhaustive)."""
    V = len(W)
    S_tot = sum(int(w) for w in W)
    best = V
    for r in range(1, V + 1):
        for sub in itertools.combinations(range(V), r):
            if sum(int(W[i]) for i in sub) * (1 << 24) >= p_fixed * S_tot:
                return r
    return best


@pytest.mark.parametrize("seed", range(12))
def test_kept_set_is_smallest_top_p_set(seed):
    """Brute force over all subsets of a V <= 10 vocabulary: the kept set has the
    minimal size any subset reaching the top-p mass has, and it holds the heaviest ids."""
    rng = np.random.default_rng(seed)
    V = int(rng.integers(2, 11))
    l = rng.normal(0, 2.0, V).astype(np.float32)
    if seed % 3 == 0:
        l[rng.integers(0, V)] = l[0]          # force ties in weight
    T = float(rng.choice([0.2, 0.7, 1.0, 2.5]))
    top_p = float(rng.choice([0.5, 0.8, 0.95, 1.0]))
    W, _ = S.int_weights(l, T)
    kept = S.kept_set(W, top_p)
    assert len(kept) == _brute_min_cardinality(W, S.p_fixed(top_p))
    outside = sorted(set(range(V)) - set(int(i) for i in kept))
    if outside:
        assert min(int(W[i]) for i in kept) >= max(int(W[i]) for i in outside)


def test_top_k_prefilter():
    l = np.float32([5.0, 4.0, 3.9, 3.8, 1.0, 0.0])
    W, _ = S.int_weights(l, 1.0)
    assert sorted(S.kept_set(W, 1.0, top_k=2).tolist()) == [0, 1]
    assert sorted(S.kept_set(W, 1.0, top_k=0).tolist()) == [0, 1, 2, 3, 4, 5]


def test_inverse_cdf_draw_exact_counts():
    """Sweeping r over 2^64 in equal steps, each kept id is drawn in proportion to its weight."""
    l = np.float32([0.3, 2.0, -1.0, 1.5, 0.9])
    W, _ = S.int_weights(l, 1.0)
    kept = np.sort(S.kept_set(W, 0.9))
    Sk = sum(int(W[i]) for i in kept)
    N = 4096
    counts = {int(i): 0 for i in kept}
    for i in range(N):
        r = ((2 * i + 1) << 64) // (2 * N)
        tau = (r * Sk) >> 64
        C = 0
        for t in kept:
            C += int(W[t])
            if C > tau:
                counts[int(t)] += 1
                break
    for t in kept:
        assert abs(counts[int(t)] / N - int(W[t]) / Sk) <= 1.0 / N + 1e-12


def test_nucleus_frequencies_chi2():
    """Empirical frequencies over many positions match the renormalised kept weights."""
    rng = np.random.default_rng(7)
    l = rng.normal(0, 1.0, 12).astype(np.float32)
    T, top_p = 1.0, 0.95
    W, _ = S.int_weights(l, T)
    kept = np.sort(S.kept_set(W, top_p))
    Sk = sum(int(W[i]) for i in kept)
    n = 6000
    draws = [S.nucleus_sample(l, T, top_p, seed=99, position=p, seq=0)[0] for p in range(n)]
    assert set(draws) <= set(int(i) for i in kept)
    obs = np.array([draws.count(int(i)) for i in kept], dtype=np.float64)
    exp = np.array([n * int(W[i]) / Sk for i in kept])
    chi2 = ((obs - exp) ** 2 / exp).sum()
    assert chi2 < 3.0 * len(kept) + 20.0


def test_low_temperature_is_greedy():
    """Greedy is the temperature -> 0 special case of nucleus sampling (Fig. 1 caption)."""
    rng = np.random.default_rng(3)
    for i in range(50):
        l = rng.normal(0, 1.3, 300).astype(np.float32)
        g, _ = S.argmax_lowest(l)
        s, _ = S.nucleus_sample(l, 1e-4, 0.95, seed=i, position=i, seq=0)
        assert s == g


def test_weights_are_floor_of_scaled_exp():
    """W_i = floor(e^{(l_i - max)/T} * 2^24) to within the exp's few-ulp error: compare with
    the exact double-precision value (the floor can move by at most 1)."""
    rng = np.random.default_rng(5)
    l = rng.normal(0, 2.0, 4000).astype(np.float32)
    for T in (0.2, 1.0):
        W, _ = S.int_weights(l, T)
        s = ((l - l.max()) / np.float32(T)).astype(np.float32).astype(np.float64)
        exact = np.floor(np.exp(s) * 2.0**24)
        assert np.abs(W.astype(np.float64) - exact).max() <= 1.0


def test_degenerate_rows():
    l = np.float32([np.nan, np.nan, np.nan])
    t, bad = S.nucleus_sample(l, 0.5, 0.9, seed=1, position=3, seq=0)
    assert bad and t == 0
