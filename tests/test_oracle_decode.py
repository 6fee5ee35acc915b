"""Pins of the oracle's two-step-draft-then-verify loops (Sec. 2.1, Eq. 1-3)."""
import os

import numpy as np
import pytest

import synth
from oracle import decode as D
from oracle import model as M

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
K = 5
PROMPT = 40
N_NEW = 32


def test_verify_hand_worked_cases():
    n = 0
    with open(os.path.join(GOLDEN, "eq3_verify_cases.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            k, t, b, m = [p.split() for p in line.split("|")]
            assert D.verify([int(x) for x in t], [int(x) for x in b], int(k[0])) == int(m[0])
            n += 1
    assert n == 6


@pytest.fixture(scope="module")
def setup(tiny_shape, tiny_model_cpu):
    W = M.Weights(tiny_shape, tensors=tiny_model_cpu)
    prompt = synth.prompt_ids(0, 0, PROMPT, 4096).tolist()
    kv = M.KVCache(tiny_shape, 1, PROMPT + N_NEW + 4 * K)
    M.prefill(W, kv, 0, prompt[:-1])
    return W, kv, prompt


def _plain(setup, sp=D.SamplingParams()):
    W, kv, prompt = setup
    return D.plain_decode(W, kv.copy(), 0, prompt[-1], N_NEW + K + 2, sp)


def _table(ref, prompt_len, match, vocab, seed=0, n=None):
    """Per-position draft table: position prompt_len + i holds ref[i] with prob `match`."""
    full = np.zeros(prompt_len + len(ref) + 64, dtype=np.int64)
    full[prompt_len:prompt_len + len(ref)] = ref
    t = synth.stub_table(seed, 0, __import__("torch").tensor(full), match, vocab).numpy()
    return t


@pytest.mark.parametrize("match", [None, 0.0, 0.7, 1.0])
def test_greedy_sdsat_equals_plain_greedy(setup, tiny_shape, match):
    """Sec. 2.1.1: greedy SDSAT output is token-for-token the plain greedy output,
    whatever the drafts are (the model's own, a perfect stub, a useless stub)."""
    W, kv, prompt = setup
    ref = _plain(setup)
    table = None if match is None else _table(ref, PROMPT, match, tiny_shape.vocab)
    res = D.sdsat_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id],
                         draft_table=table)
    assert res.tokens == ref[:N_NEW]
    assert all(2 <= n <= K + 2 for n in res.per_loop)          # Sec. 2.1.1 bound
    if match == 1.0:
        assert all(n == K + 2 for n in res.per_loop[:-1])
    if match == 0.0:
        # a useless draft can still coincide with the target only by chance (1 / V)
        assert sum(n > 2 for n in res.per_loop) <= 1


def test_wrong_drafts_give_two_tokens_per_loop(setup, tiny_shape):
    W, kv, prompt = setup
    ref = _plain(setup)
    full = np.zeros(PROMPT + len(ref) + 64, dtype=np.int64)
    full[PROMPT:PROMPT + len(ref)] = (np.array(ref) + 1) % tiny_shape.vocab
    res = D.sdsat_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id],
                         draft_table=full)
    assert all(n == 2 for n in res.per_loop[:-1])
    assert res.tokens == ref[:N_NEW]


@pytest.mark.parametrize("T,top_p,top_k", [(0.2, 0.95, 0), (1.0, 0.95, 10), (1.0, 0.5, 0)])
def test_nucleus_sdsat_equals_plain_nucleus(setup, tiny_shape, T, top_p, top_k):
    """With the draw keyed by the produced token's position, the chain nucleus loop
    (Sec. 2.1.2) emits exactly what plain nucleus decoding emits with the same seed."""
    W, kv, prompt = setup
    sp = D.SamplingParams(T, top_p, top_k, seed=2024)
    ref = _plain(setup, sp)
    for table in (None, _table(ref, PROMPT, 0.6, tiny_shape.vocab)):
        res = D.sdsat_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, [tiny_shape.adaptive_id],
                             sp, draft_table=table)
        assert res.tokens == ref[:N_NEW]


def test_diverse_adaptive_ids(setup, tiny_shape):
    """App. B: a list of distinct adaptive ids is accepted and leaves greedy output unchanged."""
    W, kv, prompt = setup
    ref = _plain(setup)
    ids = [4096, 4097, 4098, 4099, 4100]
    res = D.sdsat_decode(W, kv.copy(), 0, prompt[-1], N_NEW, K, ids)
    assert res.tokens == ref[:N_NEW]


def test_step_log_shapes(setup, tiny_shape):
    W, kv, prompt = setup
    res = D.sdsat_decode(W, kv.copy(), 0, prompt[-1], 8, K, [tiny_shape.adaptive_id], log=True)
    assert [s.mode for s in res.steps[:4]] == ["draft", "verify", "draft", "verify"]
    for s in res.steps:
        assert s.logits.shape == (K + 1, tiny_shape.vocab)
        assert s.tokens[1:] == [tiny_shape.adaptive_id] * K if s.mode == "draft" else True
