"""Pins of the oracle's pipelined variant (step 2 also carries the k adaptive tokens)."""
import numpy as np
import pytest
import torch

import synth
from oracle import decode as D
from oracle import model as M
from oracle import pipelined as P

K = 3
PROMPT = 40
N_NEW = 30


@pytest.fixture(scope="module")
def setup(tiny_shape, tiny_model_cpu):
    W = M.Weights(tiny_shape, tensors=tiny_model_cpu)
    prompt = synth.prompt_ids(0, 3, PROMPT, 4096).tolist()
    kv = M.KVCache(tiny_shape, 1, PROMPT + 2 * N_NEW + 8 * K)
    M.prefill(W, kv, 0, prompt[:-1])
    return W, kv, prompt


def _plain(setup, sp=D.SamplingParams()):
    W, kv, prompt = setup
    return D.plain_decode(W, kv.copy(), 0, prompt[-1], N_NEW + 2 * K + 2, sp)


def _table(ref, match, vocab, seed=0):
    full = np.zeros(PROMPT + len(ref) + 64, dtype=np.int64)
    full[PROMPT:PROMPT + len(ref)] = ref
    return synth.stub_table(seed, 0, torch.tensor(full), match, vocab).numpy()


def test_block_layout_and_transitions_hand_worked():
    a = [9, 9]
    assert P.block_tokens(5, None, a) == ([5, 9, 9, 9, 9], 0)
    assert P.block_tokens(5, [7, 8], a) == ([5, 7, 8, 9, 9], 2)
    t = [11, 12, 13, 14, 15]
    assert P.next_state(P.MODE_S, 0, 2, t) == (P.MODE_A, 11, [12, 13])     # step 1's drafts
    assert P.next_state(P.MODE_A, 2, 2, t) == (P.MODE_A, 13, [14, 15])     # all accepted: no step 1
    assert P.next_state(P.MODE_A, 1, 2, t) == (P.MODE_S, 12, None)         # a rejection: step 1 next
    assert P.next_state(P.MODE_A, 0, 2, t) == (P.MODE_S, 11, None)


@pytest.mark.parametrize("match", [None, 0.0, 0.5, 0.9])
def test_pipelined_greedy_equals_plain_greedy(setup, tiny_shape, match):
    W, kv, prompt = setup
    ref = _plain(setup)
    table = None if match is None else _table(ref, match, tiny_shape.vocab)
    res = P.pipelined_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id], draft_table=table)
    assert res.tokens == ref[:N_NEW]
    assert all(1 <= n <= K + 1 for n in res.per_loop)


def test_pipelined_nucleus_equals_plain_nucleus(setup, tiny_shape):
    W, kv, prompt = setup
    sp = D.SamplingParams(0.8, 0.9, 0, seed=17)
    ref = _plain(setup, sp)
    table = _table(ref, 0.7, tiny_shape.vocab)
    res = P.pipelined_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id], sp, draft_table=table)
    assert res.tokens == ref[:N_NEW]


def test_perfect_drafts_skip_draft_step_1(setup, tiny_shape):
    """Every draft right: one S block, then every block verifies all k drafts and emits k + 1."""
    W, kv, prompt = setup
    ref = _plain(setup)
    res = P.pipelined_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id],
                             draft_table=_table(ref, 1.0, tiny_shape.vocab), log=True)
    assert res.per_loop[0] == 1 and all(n == K + 1 for n in res.per_loop[1:])
    assert [s.mode for s in res.steps] == ["draft"] + ["verify"] * (len(res.steps) - 1)


def test_wrong_drafts_alternate_like_the_two_step_loop(setup, tiny_shape):
    """Every draft wrong: S and A blocks alternate, one token each, as draft steps 1 and 2 do."""
    W, kv, prompt = setup
    ref = _plain(setup)
    full = np.zeros(PROMPT + len(ref) + 64, dtype=np.int64)
    full[PROMPT:PROMPT + len(ref)] = (np.asarray(ref) + 1) % tiny_shape.vocab
    res = P.pipelined_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id], draft_table=full,
                             log=True)
    assert res.per_loop == [1] * len(res.per_loop)
    assert [s.mode for s in res.steps] == ["draft", "verify"] * (len(res.steps) // 2) + ["draft"] * (len(res.steps) % 2)
    # the KV after n steps equals the two-step loop's: same committed length per emitted token
    assert res.tokens == ref[:N_NEW]
