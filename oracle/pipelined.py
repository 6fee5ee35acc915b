"""Oracle: the pipelined variant of two-step-draft-then-verify decoding.

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

Not a step the paper describes: in Sec. 2.1.1 draft step 2's block holds y_{n+1} and the k
drafts only, and the next loop starts with its own draft step 1.  The pipelined variant
appends the k adaptive tokens to the verification block, so that when every draft is
accepted the same forward also yields the next loop's drafts and that loop's draft step 1
is skipped.  Every block has q = 2k + 1 rows [x_0, r_1 .. r_k, a_1 .. a_k]:

  * mode A (drafts known): r_i = d_i; Eq. 3 verifies the k drafts; t_0 .. t_m are emitted
    and len advances by 1 + m.  If m = k, the adaptive rows' targets t_{k+1} .. t_{2k} are
    the drafts for the positions after t_k and the next block is again mode A
    (x_0 = t_k); otherwise the next block is mode S (x_0 = t_m).
  * mode S (no drafts): r_i = a_i, nothing is verified (m = 0): the block is draft step 1
    (Eq. 1) with k extra adaptive rows; t_0 is emitted, len advances by 1, and t_1 .. t_k
    are the next block's drafts (mode A, x_0 = t_0).

Row j sits at position len + j and its target is the token at position len + j + 1 (the
same selection as the chain step), so, as for the chain, the emitted sequence is the plain
decoding sequence: a draft is emitted only as the target that verified it.  With a draft
table (the harness's stub), a mode-A block takes its drafts from the table at positions
len + 1 .. len + k instead, exactly as draft step 2 does in oracle/decode.py.
"""
from __future__ import annotations

from typing import Optional, Sequence

import numpy as np

from . import model as M
from .decode import DecodeResult, SamplingParams, StepLog, row_targets, verify

MODE_S = 0
MODE_A = 1


def block_tokens(x0: int, drafts: Optional[Sequence[int]], a: Sequence[int]):
    """The q = 2k + 1 block and its number of verified drafts: mode A with drafts, else S."""
    k = len(a)
    if drafts is None:
        return [int(x0)] + list(a) + list(a), 0
    return [int(x0)] + [int(d) for d in drafts] + list(a), k


def next_state(mode: int, m: int, k: int, targets: Sequence[int]):
    """(next mode, next x_0, next drafts or None) after a block of `mode` accepted m drafts."""
    if mode == MODE_S:
        return MODE_A, targets[0], list(targets[1:k + 1])
    if m == k:
        return MODE_A, targets[k], list(targets[k + 1:2 * k + 1])
    return MODE_S, targets[m], None


def pipelined_decode(W: M.Weights, kv: M.KVCache, seq: int, last: int, n_new: int, k: int,
                     adaptive_ids: Sequence[int], sp: SamplingParams = SamplingParams(),
                     draft_table: Optional[np.ndarray] = None, log: bool = False) -> DecodeResult:
    """Pipelined decoding of n_new tokens after a prefilled cache (one forward per step).

    res.per_loop holds the tokens each step (each forward) emitted; res.loops the steps.
    """
    ids = list(adaptive_ids)
    a = ids * k if len(ids) == 1 else ids[:k]
    if len(a) != k:
        raise ValueError("need k adaptive ids")
    res = DecodeResult(tokens=[])
    mode, x0, drafts = MODE_S, int(last), None
    while len(res.tokens) < n_new:
        L0 = kv.len[seq]
        if mode == MODE_A and draft_table is not None:
            drafts = [int(draft_table[L0 + i]) for i in range(1, k + 1)]
        blk, n_verify = block_tokens(x0, drafts if mode == MODE_A else None, a)
        logits = M.block_forward(W, kv, seq, blk)
        t, _ = row_targets(logits, sp, L0 + 1, seq)
        m = verify(t, blk, n_verify)
        kv.len[seq] += 1 + m
        res.tokens.extend(t[:m + 1])
        if log:
            res.steps.append(StepLog("verify" if mode == MODE_A else "draft", L0, blk, logits, t, 1 + m))
        res.loops += 1
        res.per_loop.append(1 + m)
        mode, x0, drafts = next_state(mode, m, k, t)
    res.tokens = res.tokens[:n_new]
    return res
