"""Oracle: two-step-draft-then-verify decoding (Sec. 2.1) and plain decoding.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

One loop (Sec. 2.1.1, Eq. 1-3), with len = committed KV length and `last`
the newest emitted token (not yet in the cache):

  draft step 1 (Eq. 1)  block [last, a_1 .. a_k] at slots len .. len+k.
                        Row 0's target is y_{n+1} (emitted); rows 1..k give
                        the drafts y'_{n+2} .. y'_{n+k+1}.  Commit len += 1
                        (the adaptive positions are rolled back).
  draft step 2 (Eq. 2)  block [y_{n+1}, d_1 .. d_k] at slots len .. len+k.
                        Row j's target t_j is y_{n+2} (j = 0) or y''_{n+2+j}.
  verification (Eq. 3)  accept t_0; accept t_i while d_i == t_{i-1} for all
                        i' <= i (y''_{n+2} is y_{n+2}); stop at the first
                        mismatch.  With m matches, t_0 .. t_m are emitted and
                        len += 1 + m; t_m becomes `last`.

So each loop emits 2 + m tokens, 0 <= m <= k (Sec. 2.1.1).  The nucleus form
(Sec. 2.1.2) is the same chain with sampled targets; the chain is the
width-1 case of the paper's draft tree, and its "longest accepted branch" is
the accepted prefix.  Drafts may be overridden by a per-position table (the
harness's draft stub); the method accepts whatever drafts it is given.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence

import numpy as np

from . import model as M
from . import sampling as S


def verify(targets: Sequence[int], block_tokens: Sequence[int], n_verify: int) -> int:
    """Eq. 3: the number m of accepted drafts (0 <= m <= n_verify).

    Draft i (block row i, 1 <= i <= n_verify) is accepted while it equals the
    target of row i-1 and every earlier draft was accepted.
    """
    m = 0
    for i in range(1, n_verify + 1):
        if int(block_tokens[i]) != int(targets[i - 1]):
            break
        m = i
    return m


@dataclass
class SamplingParams:
    temperature: float = 0.0      # 0 => greedy
    top_p: float = 1.0
    top_k: int = 0
    seed: int = 0


def row_targets(logits: np.ndarray, sp: SamplingParams, first_position: int, seq: int):
    """Target of every block row; row j produces the token at first_position + j."""
    out, nan = [], False
    for j in range(logits.shape[0]):
        t, bad = S.select(logits[j].astype(np.float32), sp.temperature, sp.top_p, sp.seed,
                          first_position + j, seq, sp.top_k)
        out.append(t)
        nan |= bad
    return out, nan


@dataclass
class StepLog:
    """Everything one block step consumed and produced (for teacher-forced parity)."""
    mode: str                     # "draft" (step 1) or "verify" (step 2)
    len_before: int
    tokens: List[int]
    logits: np.ndarray
    targets: List[int]
    accepted: int                 # emitted tokens this step (1 + m)


@dataclass
class DecodeResult:
    tokens: List[int]
    steps: List[StepLog] = field(default_factory=list)
    loops: int = 0
    per_loop: List[int] = field(default_factory=list)


def sdsat_decode(W: M.Weights, kv: M.KVCache, seq: int, last: int, n_new: int, k: int,
                 adaptive_ids: Sequence[int], sp: SamplingParams = SamplingParams(),
                 draft_table: Optional[np.ndarray] = None, log: bool = False) -> DecodeResult:
    """Two-step-draft-then-verify decoding of n_new tokens after a prefilled cache.

    adaptive_ids: one id (repeated k times) or a list of k ids (diverse tokens,
    App. B).  draft_table[p], when given, replaces the draft for position p.
    """
    ids = list(adaptive_ids)
    a = ids * k if len(ids) == 1 else ids[:k]
    if len(a) != k:
        raise ValueError("need k adaptive ids")
    res = DecodeResult(tokens=[])
    while len(res.tokens) < n_new:
        # draft step 1 (Eq. 1)
        L0 = kv.len[seq]
        blk = [last] + a
        logits = M.block_forward(W, kv, seq, blk)
        t, _ = row_targets(logits, sp, L0 + 1, seq)
        kv.len[seq] += 1
        res.tokens.append(t[0])
        drafts = t[1:]
        if log:
            res.steps.append(StepLog("draft", L0, blk, logits, t, 1))
        L1 = kv.len[seq]
        if draft_table is not None:
            drafts = [int(draft_table[L1 + j]) for j in range(1, k + 1)]
        # draft step 2 (Eq. 2)
        blk = [t[0]] + drafts
        logits = M.block_forward(W, kv, seq, blk)
        t2, _ = row_targets(logits, sp, L1 + 1, seq)
        m = verify(t2, blk, k)                                   # Eq. 3
        kv.len[seq] += 1 + m
        res.tokens.extend(t2[:m + 1])
        last = t2[m]
        if log:
            res.steps.append(StepLog("verify", L1, blk, logits, t2, 1 + m))
        res.loops += 1
        res.per_loop.append(2 + m)
    res.tokens = res.tokens[:n_new]
    return res


def plain_decode(W: M.Weights, kv: M.KVCache, seq: int, last: int, n_new: int,
                 sp: SamplingParams = SamplingParams()) -> List[int]:
    """Ordinary one-token-per-step decoding (the paper's baseline)."""
    out = []
    for _ in range(n_new):
        L0 = kv.len[seq]
        logits = M.block_forward(W, kv, seq, [last])
        t, _ = row_targets(logits, sp, L0 + 1, seq)
        kv.len[seq] += 1
        out.append(t[0])
        last = t[0]
    return out
