"""Oracle: target-token selection (greedy argmax and nucleus sampling).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

Greedy search takes argmax P_theta at every block row (Eq. 1-3).  Nucleus
sampling (Sec. 2.1.2; settings top_p 0.95, temperatures 0.2 and 1, optional
top_k, Sec. 3.4.2) samples at every row instead; greedy is its temperature-0
special case (Fig. 1 caption).

The paper gives no arithmetic for the sampler, so it is defined here so that
a CPU and a GPU reach the same token from the same logits bit for bit:

  1. s_i = (l_i - max_j l_j) / T           one fp32 IEEE division
  2. w_i = exp_sd(s_i)                      fp32, every step a single
                                            correctly rounded operation
  3. W_i = floor(w_i * 2^24)                exact integer weights; the
                                            argmax has W = 2^24.  A token
                                            whose weight is below 2^-24 of
                                            the top one gets W = 0: it is
                                            below the resolution of an fp32
                                            normaliser that already holds 1
  4. candidates: all ids, or the top_k largest by (W desc, id asc)
  5. kept set: the shortest prefix of the candidates in (W desc, id asc)
     order whose cumulative weight C satisfies C * 2^24 >= P * S, where
     S = total candidate weight and P = round(top_p * 2^24)
  6. r = 64-bit Philox4x32-10 draw keyed by the seed, with counter
     (absolute position of the token being produced, sequence index, 0, 0)
  7. tau = floor(r * S_kept / 2^64); the sample is the first kept id in
     ascending id order whose inclusive cumulative weight exceeds tau.

Keying the draw by the position of the produced token makes speculative
nucleus decoding emit exactly the tokens of plain nucleus decoding with the
same seed.  NaN logits count as -inf (and raise the error flag).

exp_sd is Cody-Waite range reduction (Cody & Waite, "Software Manual for the
Elementary Functions", 1980) with a two-part ln 2, a degree-7 Taylor
polynomial of e^r on |r| <= ln2/2 evaluated by Horner's rule, and an exact
power-of-two scaling; arguments below -87 give 0.
"""
from __future__ import annotations

from typing import Optional, Sequence, Tuple

import numpy as np

f32 = np.float32

LOG2E = f32(1.4426950408889634)
LN2_HI = f32(0.693145751953125)          # 16 significant bits: n * LN2_HI is exact
LN2_LO = f32(0.6931471805599453 - 0.693145751953125)
EXP_COEF = [f32(1.0 / 5040.0), f32(1.0 / 720.0), f32(1.0 / 120.0), f32(1.0 / 24.0),
            f32(1.0 / 6.0), f32(0.5), f32(1.0), f32(1.0)]   # 1/7! ... 1/0!
EXP_MIN = f32(-87.0)
W_SHIFT = 24
P_SHIFT = 24

M32 = 0xFFFFFFFF


def argmax_lowest(logits: np.ndarray) -> Tuple[int, bool]:
    """Index of the maximum (lowest index on ties); NaN counts as -inf.

    Returns (index, saw_nan).
    """
    x = np.asarray(logits, dtype=np.float64)
    nan = np.isnan(x)
    if nan.any():
        x = np.where(nan, -np.inf, x)
    return int(np.argmax(x)), bool(nan.any())   # np.argmax returns the first maximum


def top2_gap(logits: np.ndarray) -> float:
    x = np.sort(np.asarray(logits, dtype=np.float64))
    return float(x[-1] - x[-2])


def exp_sd(s: np.ndarray) -> np.ndarray:
    """e^s for fp32 s <= 0 (see module docstring); fp32 result."""
    s = np.asarray(s, dtype=f32)
    ok = s >= EXP_MIN                        # false for NaN and -inf too
    s_ok = np.where(ok, s, f32(0.0)).astype(f32)
    n = np.rint(s_ok * LOG2E).astype(f32)
    r = ((s_ok - n * LN2_HI) - n * LN2_LO).astype(f32)
    p = EXP_COEF[0]
    for c in EXP_COEF[1:]:
        p = (p * r + c).astype(f32)
    out = np.ldexp(p, n.astype(np.int32)).astype(f32)
    return np.where(ok, out, f32(0.0)).astype(f32)


def int_weights(logits: np.ndarray, temperature: float) -> Tuple[np.ndarray, bool]:
    """Steps 1-3: exact uint64 weights W_i from fp32 logits.  Returns (W, saw_nan)."""
    l = np.asarray(logits, dtype=f32)
    nan = np.isnan(l)
    l = np.where(nan, f32(-np.inf), l).astype(f32)
    mx = l.max()
    s = ((l - mx) / f32(temperature)).astype(f32)
    w = exp_sd(s)
    W = np.floor(np.ldexp(w.astype(np.float64), W_SHIFT)).astype(np.uint64)
    return W, bool(nan.any())


def philox4x32_10(ctr: Sequence[int], key: Sequence[int]) -> Tuple[int, int, int, int]:
    """Philox4x32 with 10 rounds (Salmon, Moraes, Dror, Shaw, SC'11)."""
    M0, M1 = 0xD2511F53, 0xCD9E8D57
    W0, W1 = 0x9E3779B9, 0xBB67AE85
    c0, c1, c2, c3 = (int(c) & M32 for c in ctr)
    k0, k1 = (int(k) & M32 for k in key)
    for _ in range(10):
        p0 = M0 * c0
        p1 = M1 * c2
        c0, c1, c2, c3 = ((p1 >> 32) ^ c1 ^ k0), (p1 & M32), ((p0 >> 32) ^ c3 ^ k1), (p0 & M32)
        k0 = (k0 + W0) & M32
        k1 = (k1 + W1) & M32
    return c0, c1, c2, c3


def draw64(seed: int, position: int, seq: int) -> int:
    """64-bit uniform for the token produced at `position` of sequence `seq`."""
    x = philox4x32_10((position, seq, 0, 0), (seed & M32, (seed >> 32) & M32))
    return (x[0] << 32) | x[1]


def p_fixed(top_p: float) -> int:
    """P = round(top_p * 2^24), clamped to [0, 2^24]."""
    return int(min(max(round(top_p * (1 << P_SHIFT)), 0), 1 << P_SHIFT))


def kept_set(W: np.ndarray, top_p: float, top_k: int = 0) -> np.ndarray:
    """Steps 4-5: ids of the kept set (in W-desc, id-asc order)."""
    ids = np.arange(W.size, dtype=np.int64)
    order = np.lexsort((ids, -W.astype(np.int64)))      # primary: W desc; then id asc
    cand = order[:top_k] if top_k > 0 else order
    Wc = W[cand].astype(object)
    S = int(sum(Wc))
    P = p_fixed(top_p)
    C = 0
    for i, w in enumerate(Wc):
        C += int(w)
        if C * (1 << P_SHIFT) >= P * S:
            return cand[:i + 1]
    return cand


def nucleus_sample(logits: np.ndarray, temperature: float, top_p: float, seed: int,
                   position: int, seq: int, top_k: int = 0) -> Tuple[int, bool]:
    """The sampled token id for one row (temperature > 0).  Returns (id, saw_nan)."""
    W, nan = int_weights(logits, temperature)
    kept = np.sort(kept_set(W, top_p, top_k))           # ascending id
    S_kept = int(sum(int(W[i]) for i in kept))
    r = draw64(seed, position, seq)
    tau = (r * S_kept) >> 64
    C = 0
    for i in kept:
        C += int(W[i])
        if C > tau:
            return int(i), nan
    return int(kept[-1]), nan       # only when S_kept == 0 (an all-NaN row): its single kept id


def select(logits: np.ndarray, temperature: float = 0.0, top_p: float = 1.0, seed: int = 0,
           position: int = 0, seq: int = 0, top_k: int = 0) -> Tuple[int, bool]:
    """Target token of one block row: argmax for temperature 0, else a nucleus sample."""
    if temperature <= 0.0:
        return argmax_lowest(logits)
    return nucleus_sample(logits, temperature, top_p, seed, position, seq, top_k)
