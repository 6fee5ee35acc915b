"""Oracle: tree-structured draft step 2 and its verification (Sec. 2.1.2).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

With nucleus sampling, draft step 1 offers several possible draft tokens per
position; draft step 2 arranges them as a tree whose branches are alternative
continuations, evaluates the whole tree in one pass with a tree attention mask,
and verification keeps the longest branch that is verified and accepted
(Sec. 2.1.2; Fig. 1, right).  The paper does not spell out the tree layout or
the acceptance test along a branch; the readings used here:

  * The block rows are the tree's nodes in topological order: row 0 is the
    root y_{n+1} (the token draft step 1 emitted) and parent[j] < j for every
    other row.
  * Row j occupies cache slot len + j, sits at position len + depth(j) (RoPE
    and the sampler's position key), and attends to the committed slots
    [0, len) plus the slots of its ancestors and itself.
  * Targets: t_j is selected from row j's logits as in the chain step -- argmax,
    or the position-keyed nucleus sampler producing position len + depth(j) + 1.
  * Acceptance: the root is accepted; a child c is accepted iff its parent is
    accepted and token(c) == t_{parent(c)} -- the chain's Eq. 3 test applied
    along every branch.  The deepest accepted node (the lowest row index among
    equally deep ones) ends the accepted path n_0 = 0, n_1, ..., n_m; the
    emitted tokens are t_{n_0} .. t_{n_m}, so a loop still emits 2 + m tokens.
  * Commit: the path's K and V rows move to contiguous slots (slot len + i
    receives row n_i's rows; they were rotated at position len + i already)
    and len advances by 1 + m.

A tree whose rows form one chain (parent[j] = j - 1) is exactly the chain step
of oracle/decode.py.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

from . import model as M


def check_parent(parent: Sequence[int]) -> None:
    """Raise unless parent describes a tree in topological order rooted at row 0."""
    if len(parent) == 0 or int(parent[0]) != -1:
        raise ValueError("row 0 must be the root (parent -1)")
    for j in range(1, len(parent)):
        if not 0 <= int(parent[j]) < j:
            raise ValueError("parent[%d] = %d is not an earlier row" % (j, int(parent[j])))


def depths(parent: Sequence[int]) -> List[int]:
    check_parent(parent)
    d = [0] * len(parent)
    for j in range(1, len(parent)):
        d[j] = d[int(parent[j])] + 1
    return d


def ancestors(parent: Sequence[int]) -> List[List[int]]:
    """Row j's root path (ascending rows: root first, j last)."""
    check_parent(parent)
    out = []
    for j in range(len(parent)):
        path, i = [], j
        while i >= 0:
            path.append(i)
            i = int(parent[i])
        out.append(sorted(path))
    return out


def positions(parent: Sequence[int], L0: int) -> List[int]:
    return [L0 + d for d in depths(parent)]


def tree_forward(W: M.Weights, kv: M.KVCache, seq: int, tokens: Sequence[int], parent: Sequence[int],
                 final: bool = True):
    """Logits of every tree node (rows at slots len + j, positions len + depth(j))."""
    L0 = kv.len[seq]
    return M.block_forward(W, kv, seq, tokens, positions=positions(parent, L0), final=final,
                           visible=ancestors(parent))


def tree_verify(targets: Sequence[int], tokens: Sequence[int], parent: Sequence[int]) -> List[int]:
    """The accepted path [n_0 = 0, n_1, ..., n_m] (rows, root first)."""
    d = depths(parent)
    acc = [False] * len(parent)
    acc[0] = True
    best = 0
    for j in range(1, len(parent)):
        pj = int(parent[j])
        acc[j] = acc[pj] and int(tokens[j]) == int(targets[pj])
        if acc[j] and d[j] > d[best]:
            best = j
    path, i = [], best
    while i >= 0:
        path.append(i)
        i = int(parent[i])
    return path[::-1]


def tree_commit(kv: M.KVCache, seq: int, path: Sequence[int]) -> None:
    """Move the accepted path's K / V rows to contiguous slots and commit them."""
    L0 = kv.len[seq]
    for l in range(len(kv.K)):
        for i, n in enumerate(path):
            if n != i:
                kv.K[l][seq][:, L0 + i] = kv.K[l][seq][:, L0 + n]
                kv.V[l][seq][:, L0 + i] = kv.V[l][seq][:, L0 + n]
    kv.len[seq] += len(path)


def chains_parent(width: int, k: int) -> List[int]:
    """The tree of `width` chains of k drafts below the root (row 1 + w*k + i is draft i + 1 of
    branch w); width 1 is the chain step."""
    parent = [-1]
    for w in range(width):
        for i in range(k):
            parent.append(0 if i == 0 else 1 + w * k + i - 1)
    return parent


def tree_targets(logits, sp, parent: Sequence[int], L0: int, seq: int) -> List[int]:
    """t_j for every node: the selection of oracle/sampling.py, producing position L0 + depth(j) + 1."""
    import numpy as np
    from . import sampling as S
    d = depths(parent)
    return [S.select(np.asarray(logits[j], dtype=np.float32), sp.temperature, sp.top_p, sp.seed,
                     L0 + d[j] + 1, seq, sp.top_k)[0] for j in range(len(parent))]


def tree_decode(W: M.Weights, kv: M.KVCache, seq: int, last: int, n_new: int, k: int, width: int,
                adaptive_ids: Sequence[int], sp, draft_tables, log: bool = False):
    """Two-step-draft-then-verify decoding with a tree draft step 2 (Sec. 2.1.2).

    Draft step 1 is the chain step of oracle/decode.py.  Draft step 2 evaluates the tree
    chains_parent(width, k) whose branch w holds draft_tables[w][position] at depths
    1..k (the harness's stand-in for draft step 1's alternative candidates), and the
    longest accepted branch is emitted and committed.
    """
    from .decode import DecodeResult, StepLog, row_targets
    ids = list(adaptive_ids)
    a = ids * k if len(ids) == 1 else ids[:k]
    parent = chains_parent(width, k)
    res = DecodeResult(tokens=[])
    while len(res.tokens) < n_new:
        L0 = kv.len[seq]
        blk = [last] + a
        logits = M.block_forward(W, kv, seq, blk)
        t, _ = row_targets(logits, sp, L0 + 1, seq)
        kv.len[seq] += 1
        res.tokens.append(t[0])
        if log:
            res.steps.append(StepLog("draft", L0, blk, logits, t, 1))
        L1 = kv.len[seq]
        blk = [t[0]] + [int(draft_tables[w][L1 + i]) for w in range(width) for i in range(1, k + 1)]
        logits = tree_forward(W, kv, seq, blk, parent)
        t2 = tree_targets(logits, sp, parent, L1, seq)
        path = tree_verify(t2, blk, parent)
        tree_commit(kv, seq, path)
        emitted = [t2[n] for n in path]
        res.tokens.extend(emitted)
        last = emitted[-1]
        if log:
            res.steps.append(StepLog("verify", L1, blk, logits, t2, len(path)))
        res.loops += 1
        res.per_loop.append(1 + len(path))
    res.tokens = res.tokens[:n_new]
    return res
