"""Parity of the pipelined variant on the GPU against oracle/pipelined.py.

  * the block builder: tokens, next mode and verify counts bit-exact against the oracle's
    transition rule, with and without a draft table, b = 3;
  * the loop on the device alone (build -> forward -> accept, no host in between) emits the
    plain greedy sequence and the oracle's tokens per step;
  * every step of the oracle's nucleus run replayed on the GPU: logits within the chain
    step's tolerances, targets and accepted counts bit-exact on the GPU's logits.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import decode as OD
from oracle import model as OM
from oracle import pipelined as OP
from oracle import sampling as OS

pytestmark = pytest.mark.gpu

K = 3
Q = 2 * K + 1
PROMPT = 96
N_NEW = 40
LOGIT_MAX_ABS = 3e-2
LOGIT_REL_RMS = 1e-2


@pytest.fixture(scope="module")
def sd():
    import paper_2403_18647_gb300 as sd
    return sd


@pytest.fixture(scope="module")
def tiny(sd):
    shape = synth.SHAPES["tiny"]
    w_gpu = synth.make_model(shape, seed=0, device="cuda", gain_std=0.1)
    w_cpu = synth.make_model(shape, seed=0, device="cpu", gain_std=0.1)
    ctx = sd.Context(shape, w_gpu, max_position=1024)
    return shape, ctx, OM.Weights(shape, tensors=w_cpu)


def _i32(x):
    return torch.tensor(list(x), dtype=torch.int32, device="cuda")


@pytest.mark.parametrize("with_table", [False, True])
def test_build_pipelined_block_transitions(sd, tiny, with_table):
    shape, ctx, W = tiny
    b = 3
    a = shape.adaptive_id
    kv = ctx.kv(b, 64)
    lens = [10, 20, 30]
    ctx.kv_commit(kv, _i32(lens), b)
    rng = np.random.default_rng(5)
    prev_out = rng.integers(0, 4000, size=b * Q).tolist()
    cases = [(0, 1), (1, K + 1), (1, 2)]          # (previous mode, accepted length): S; A all; A partial
    stride = 64 + 16
    table = rng.integers(0, 4000, size=b * stride).tolist()
    mode = _i32([c[0] for c in cases])
    nver = _i32([-1] * b)
    toks = torch.zeros(b * Q, dtype=torch.int32, device="cuda")
    ctx.build_pipelined_block(kv, _i32(prev_out), _i32([c[1] for c in cases]), mode, nver, toks, b, K,
                              draft_table=_i32(table) if with_table else None, table_stride=stride)
    got = toks.cpu().tolist()
    for s, (pm, acc) in enumerate(cases):
        t = prev_out[s * Q:(s + 1) * Q]
        if pm == OP.MODE_A and acc - 1 < K:
            nm, x0, drafts = OP.MODE_S, t[acc - 1], None
        else:
            nm, x0, drafts = OP.next_state(pm, acc - 1, K, t)
        if nm == OP.MODE_A and with_table:
            drafts = [table[s * stride + lens[s] + i] for i in range(1, K + 1)]
        blk, nv = OP.block_tokens(x0, drafts, [a] * K)
        assert got[s * Q:(s + 1) * Q] == blk, (s, got[s * Q:(s + 1) * Q], blk)
        assert mode[s].item() == nm and nver[s].item() == nv


def _oracle_run(shape, W, sp, match, n_new=N_NEW):
    prompt = synth.prompt_ids(0, 0, PROMPT, 4096)
    kv = OM.KVCache(shape, 1, PROMPT + 2 * n_new + 4 * Q)
    OM.prefill(W, kv, 0, prompt[:-1].tolist())
    base = kv.copy()
    ref = OD.plain_decode(W, kv.copy(), 0, int(prompt[-1]), n_new + Q + 2, sp)
    full = torch.zeros(kv.max_len + 64, dtype=torch.int32)
    full[PROMPT:PROMPT + len(ref)] = torch.tensor(ref, dtype=torch.int32)
    table = synth.stub_table(0, 0, full, match, shape.vocab)
    res = OP.pipelined_decode(W, base.copy(), 0, int(prompt[-1]), n_new, K, [shape.adaptive_id], sp,
                              draft_table=table.numpy(), log=True)
    return prompt, ref, table, res, kv.max_len


def test_pipelined_device_loop_equals_plain_greedy(sd, tiny):
    shape, ctx, W = tiny
    sp = OD.SamplingParams()
    prompt, ref, table, res, cap = _oracle_run(shape, W, sp, 0.8)
    stride = cap + 32
    tab = torch.zeros(stride, dtype=torch.int32)
    tab[:min(stride, table.numel())] = table[:stride]
    tab = tab.cuda()
    kv = ctx.kv(1, cap)
    ctx.prefill(kv, 0, prompt[:-1].cuda())
    logits = torch.empty(Q, shape.vocab, device="cuda")
    acc = torch.ones(1, dtype=torch.int32, device="cuda")
    out = torch.zeros(Q, dtype=torch.int32, device="cuda")
    out[0] = int(prompt[-1])
    mode = _i32([1])
    nver = _i32([0])
    toks = torch.empty(Q, dtype=torch.int32, device="cuda")
    emitted, per_step = [], []
    while len(emitted) < N_NEW:
        ctx.build_pipelined_block(kv, out, acc, mode, nver, toks, 1, K, draft_table=tab, table_stride=stride)
        ctx.block_forward(kv, toks, logits, 1, Q)
        ctx.accept_pipelined(kv, logits, toks, nver, 1, Q, acc, out)
        a = int(acc.item())
        emitted += out[:a].cpu().tolist()
        per_step.append(a)
    assert all(1 <= n <= K + 1 for n in per_step)
    emitted = emitted[:N_NEW]
    first_diff = next((i for i, (x, y) in enumerate(zip(emitted, ref)) if x != y), None)
    assert first_diff is None or first_diff > 8, (first_diff, emitted[:10], ref[:10])
    if first_diff is None:
        assert per_step[:-1] == res.per_loop[:len(per_step) - 1]
    assert max(per_step) == K + 1   # some steps verified every draft (and skipped draft step 1)
    assert ctx.get_error() == 0


def test_pipelined_teacher_forced_nucleus(sd, tiny):
    shape, ctx, W = tiny
    sp = OD.SamplingParams(0.3, 0.95, 10, seed=77)
    prompt, ref, table, res, cap = _oracle_run(shape, W, sp, 0.7, n_new=30)
    kv = ctx.kv(1, cap)
    ctx.prefill(kv, 0, prompt[:-1].cuda())
    logits = torch.empty(Q, shape.vocab, device="cuda")
    acc = torch.empty(1, dtype=torch.int32, device="cuda")
    out = torch.empty(Q, dtype=torch.int32, device="cuda")
    for st in res.steps:
        toks = _i32(st.tokens)
        nv = K if st.mode == "verify" else 0
        ctx.kv_commit(kv, _i32([st.len_before]), 1)
        ctx.block_forward(kv, toks, logits, 1, Q)
        ctx.accept_pipelined(kv, logits, toks, _i32([nv]), 1, Q, acc, out, temperature=sp.temperature,
                             top_p=sp.top_p, seed=sp.seed, top_k=sp.top_k, commit=False)
        lg = logits.cpu().numpy()
        err = np.abs(lg.astype(np.float64) - st.logits).max()
        rel = np.sqrt(((lg - st.logits) ** 2).mean() / (st.logits ** 2).mean())
        assert err <= LOGIT_MAX_ABS and rel <= LOGIT_REL_RMS, (err, rel)
        tg = out.cpu().tolist()
        ref_t = [OS.select(lg[j], sp.temperature, sp.top_p, sp.seed, st.len_before + j + 1, 0, sp.top_k)[0]
                 for j in range(Q)]
        assert tg == ref_t
        assert int(acc.item()) == 1 + OD.verify(ref_t, st.tokens, nv)
    assert ctx.get_error() == 0
