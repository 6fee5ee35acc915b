"""Pins of the oracle's tree draft step 2 (Sec. 2.1.2: tree attention, longest accepted branch)."""
import itertools
import os
import random

import numpy as np
import pytest

import synth
from oracle import decode as D
from oracle import model as M
from oracle import tree as T

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
K = 4
PROMPT = 24
N_NEW = 24


def _ints(s):
    return [int(x) for x in s.split()]


def test_tree_verify_hand_worked_cases():
    n = 0
    with open(os.path.join(GOLDEN, "tree_verify_cases.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parent, tokens, targets, path, emitted = [_ints(p) for p in line.split(";")]
            got = T.tree_verify(targets, tokens, parent)
            assert got == path, line
            assert [targets[i] for i in got] == emitted
            n += 1
    assert n == 7


def _brute_force_path(targets, tokens, parent):
    """Every root path, accepted iff each edge's token matches the parent's target; the
    longest wins, then the one ending at the lowest row."""
    best = [0]
    for j in range(len(parent)):
        path, i = [], j
        while i >= 0:
            path.append(i)
            i = parent[i]
        path = path[::-1]
        if all(tokens[path[e]] == targets[path[e - 1]] for e in range(1, len(path))):
            if len(path) > len(best) or (len(path) == len(best) and path[-1] < best[-1]):
                best = path
    return best


def test_tree_verify_against_brute_force():
    rng = random.Random(3)
    for _ in range(3000):
        n = rng.randint(1, 12)
        parent = [-1] + [rng.randrange(j) for j in range(1, n)]
        targets = [rng.randrange(3) for _ in range(n)]
        tokens = [rng.randrange(3) for _ in range(n)]
        assert T.tree_verify(targets, tokens, parent) == _brute_force_path(targets, tokens, parent)


def test_tree_shapes():
    p = T.chains_parent(2, 3)
    assert p == [-1, 0, 1, 2, 0, 4, 5]
    assert T.depths(p) == [0, 1, 2, 3, 1, 2, 3]
    assert T.ancestors(p)[6] == [0, 4, 5, 6]
    assert T.chains_parent(1, 4) == [-1, 0, 1, 2, 3]
    with pytest.raises(ValueError):
        T.check_parent([-1, 1])
    with pytest.raises(ValueError):
        T.check_parent([0, -1])


@pytest.fixture(scope="module")
def setup(tiny_shape, tiny_model_cpu):
    W = M.Weights(tiny_shape, tensors=tiny_model_cpu)
    prompt = synth.prompt_ids(0, 1, PROMPT, 4096).tolist()
    kv = M.KVCache(tiny_shape, 1, PROMPT + N_NEW + 8 * 16)
    M.prefill(W, kv, 0, prompt[:-1])
    return W, kv, prompt


def test_chain_tree_equals_chain_step(setup, tiny_shape):
    """A tree whose rows form one chain is the chain step: same logits and cache, bit for bit."""
    W, kv, prompt = setup
    blk = [7, 300, 4096, 12, 99]
    a, b = kv.copy(), kv.copy()
    la = M.block_forward(W, a, 0, blk)
    lb = T.tree_forward(W, b, 0, blk, T.chains_parent(1, len(blk) - 1))
    assert np.array_equal(la, lb)
    for l in range(tiny_shape.n_layers):
        assert np.array_equal(a.K[l], b.K[l]) and np.array_equal(a.V[l], b.V[l])


def test_tree_node_equals_its_root_path(setup, tiny_shape):
    """Tree attention: every node's logits are those of a chain forward of its root path
    (same positions, same visible slots in the same order)."""
    W, kv, prompt = setup
    parent = [-1, 0, 1, 0, 3, 3, 2]
    blk = [11, 22, 33, 44, 55, 66, 77]
    lt = T.tree_forward(W, kv.copy(), 0, blk, parent)
    for j, path in enumerate(T.ancestors(parent)):
        lc = M.block_forward(W, kv.copy(), 0, [blk[i] for i in path])
        assert np.array_equal(lt[j], lc[-1]), j


def test_tree_commit_equals_chain_of_accepted_path(setup, tiny_shape):
    """After the commit the cache holds the accepted path's rows contiguously, exactly as a
    chain forward of the path's tokens would have written them."""
    W, kv, prompt = setup
    parent = T.chains_parent(2, 3)
    blk = [5, 17, 18, 19, 27, 28, 29]
    a = kv.copy()
    T.tree_forward(W, a, 0, blk, parent)
    path = [0, 4, 5]
    L0 = a.len[0]
    T.tree_commit(a, 0, path)
    assert a.len[0] == L0 + 3
    b = kv.copy()
    M.block_forward(W, b, 0, [blk[i] for i in path])
    for l in range(tiny_shape.n_layers):
        assert np.array_equal(a.K[l][0][:, L0:L0 + 3], b.K[l][0][:, L0:L0 + 3])
        assert np.array_equal(a.V[l][0][:, L0:L0 + 3], b.V[l][0][:, L0:L0 + 3])


def _tables(ref, match, vocab, width):
    full = np.zeros(PROMPT + len(ref) + 64, dtype=np.int64)
    full[PROMPT:PROMPT + len(ref)] = ref
    import torch
    return [synth.stub_table(w, 0, torch.tensor(full), match, vocab).numpy() for w in range(width)]


@pytest.mark.parametrize("width,match", [(1, 0.7), (2, 0.5), (3, 0.4)])
def test_tree_greedy_equals_plain_greedy(setup, tiny_shape, width, match):
    """Greedy with a draft tree still emits exactly the plain greedy tokens (Sec. 2.1.1's
    invariant holds along the accepted branch)."""
    W, kv, prompt = setup
    ref = D.plain_decode(W, kv.copy(), 0, prompt[-1], N_NEW + K + 2)
    res = T.tree_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, width, [tiny_shape.adaptive_id],
                        D.SamplingParams(), _tables(ref, match, tiny_shape.vocab, width))
    assert res.tokens == ref[:N_NEW]
    assert all(2 <= n <= K + 2 for n in res.per_loop)


def test_tree_nucleus_equals_plain_nucleus(setup, tiny_shape):
    """Position-keyed sampling: tree SDSAT nucleus decoding emits the plain nucleus tokens."""
    W, kv, prompt = setup
    sp = D.SamplingParams(temperature=0.7, top_p=0.95, top_k=10, seed=99)
    ref = D.plain_decode(W, kv.copy(), 0, prompt[-1], N_NEW + K + 2, sp)
    res = T.tree_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, 2, [tiny_shape.adaptive_id], sp,
                        _tables(ref, 0.5, tiny_shape.vocab, 2))
    assert res.tokens == ref[:N_NEW]


def test_wider_tree_accepts_at_least_as_much(setup, tiny_shape):
    """Adding branches never shortens the accepted path (the width-1 chain is a subtree)."""
    W, kv, prompt = setup
    ref = D.plain_decode(W, kv.copy(), 0, prompt[-1], N_NEW + K + 2)
    tabs = _tables(ref, 0.5, tiny_shape.vocab, 2)
    one = T.tree_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, 1, [tiny_shape.adaptive_id], D.SamplingParams(),
                        tabs[:1], log=True)
    two = T.tree_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, 2, [tiny_shape.adaptive_id], D.SamplingParams(),
                        tabs, log=True)
    # compare the first loop, where both start from the same state
    assert two.per_loop[0] >= one.per_loop[0]
