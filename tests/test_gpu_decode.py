"""End-to-end parity of the block decode step (block forward + acceptance + KV commit).

Protocol (teacher forcing): the oracle runs the two-step-draft-then-verify loop and
logs every step's inputs; the GPU replays each step from the same committed state
and is compared step by step:
  * logits: max-abs <= 3e-2 and relative RMS <= 1e-2 against the oracle;
  * targets and accepted counts: bit-exact, except rows whose oracle top-2 gap is
    below 1e-2 (a near-tie may legitimately flip);
then the oracle's committed length is imposed before the next step.
"""
import numpy as np
import pytest
import torch

import synth
from nucleus_flips import flip_explained
from oracle import decode as OD
from oracle import model as OM
from oracle import sampling as OS

pytestmark = pytest.mark.gpu

K = 5
Q = K + 1
PROMPT = 128
N_NEW = 64
LOGIT_MAX_ABS = 3e-2
LOGIT_REL_RMS = 1e-2
TIE_GAP = 1e-2


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


def _oracle_run(shape, W, sp, match=0.7, n_new=N_NEW, k=K):
    q = k + 1
    prompt = synth.prompt_ids(0, 0, PROMPT, 4096)
    kv = OM.KVCache(shape, 1, PROMPT + n_new + 4 * q)
    OM.prefill(W, kv, 0, prompt[:-1].tolist())
    base = kv.copy()
    ref = OD.plain_decode(W, kv.copy(), 0, int(prompt[-1]), n_new + q + 2, sp)
    full = torch.zeros(kv.max_len + 64, dtype=torch.int32)
    full[PROMPT:PROMPT + len(ref)] = torch.tensor(ref, dtype=torch.int32)
    table = synth.stub_table(0, 0, full, match, shape.vocab)
    res = OD.sdsat_decode(W, base.copy(), 0, int(prompt[-1]), n_new, k, [shape.adaptive_id], sp,
                          draft_table=table.numpy(), log=True)
    return prompt, ref, table, res


def _compare_logits(got, ref):
    err = np.abs(got - ref).max()
    rel = np.sqrt(((got - ref) ** 2).mean() / (ref ** 2).mean())
    assert err <= LOGIT_MAX_ABS and rel <= LOGIT_REL_RMS, (err, rel)
    return err, rel


def _teacher_forced(sd, shape, ctx, res, prompt, sp, k=K):
    """Replays the oracle's logged steps on the GPU.  Returns the worst logit error and the
    number of rows whose target differs from the oracle's (greedy: only near-ties may)."""
    Q = k + 1
    kv = ctx.kv(1, PROMPT + N_NEW + 4 * Q)
    ctx.prefill(kv, 0, prompt[:-1].cuda())
    logits = torch.empty(Q, shape.vocab, device="cuda")
    acc = torch.empty(1, dtype=torch.int32, device="cuda")
    out = torch.empty(Q, dtype=torch.int32, device="cuda")
    worst = 0.0
    flips = 0
    for st in res.steps:
        toks = torch.tensor(st.tokens, dtype=torch.int32, device="cuda")
        ctx.kv_commit(kv, torch.tensor([st.len_before], dtype=torch.int32, device="cuda"), 1)
        ctx.block_forward(kv, toks, logits, 1, Q)
        nv = 0 if st.mode == "draft" else k
        if sp.temperature > 0:
            ctx.accept_nucleus(kv, logits, toks, 1, Q, nv, sp.top_p, sp.temperature, sp.seed, acc, out,
                               top_k=sp.top_k, commit=False)
        else:
            ctx.accept_greedy(kv, logits, toks, 1, Q, nv, acc, out, commit=False)
        lg = logits.cpu().numpy()
        err, _ = _compare_logits(lg.astype(np.float64), st.logits)
        worst = max(worst, err)
        tg = out.cpu().tolist()
        # targets: exact except near-ties of the oracle
        step_flips = 0
        for j in range(Q):
            if tg[j] != st.targets[j]:
                # greedy: only a near-tie of the oracle may flip; a sampled target only where this
                # row's logit error can move a sampling boundary across the shared draw
                if sp.temperature > 0:
                    ok, info = flip_explained(st.logits[j], lg[j], sp.temperature, sp.top_p, sp.top_k, sp.seed,
                                              st.len_before + j + 1, 0)
                    assert ok, (j, info)
                else:
                    assert OS.top2_gap(st.logits[j]) < TIE_GAP, (j, tg[j], st.targets[j])
                step_flips += 1
        flips += step_flips
        if step_flips == 0:
            assert int(acc.item()) == st.accepted
        # the acceptance kernel itself is bit-exact on the logits it was given
        for j in range(Q):
            ref_t = OS.select(lg[j], sp.temperature, sp.top_p, sp.seed, st.len_before + j + 1, 0, sp.top_k)[0]
            assert tg[j] == ref_t
    assert ctx.get_error() == 0
    return worst, flips


def test_tiny_greedy_teacher_forced(sd, tiny):
    shape, ctx, W = tiny
    sp = OD.SamplingParams()
    prompt, ref, table, res = _oracle_run(shape, W, sp)
    worst, flips = _teacher_forced(sd, shape, ctx, res, prompt, sp)
    assert flips <= 1


def test_tiny_nucleus_teacher_forced(sd, tiny):
    shape, ctx, W = tiny
    sp = OD.SamplingParams(0.2, 0.95, 0, seed=1234)
    prompt, ref, table, res = _oracle_run(shape, W, sp, match=0.6, n_new=32)
    worst, flips = _teacher_forced(sd, shape, ctx, res, prompt, sp)
    # every flip was explained by its row's logit error; the rows still agree mostly
    assert flips <= len(res.steps) * (K + 1) // 4, (flips, len(res.steps))


def test_tiny_greedy_teacher_forced_k13(sd, tiny):
    """The largest block of the k-sweep (k = 13, q = 14; Sec. 3.4.1, Fig. 3)."""
    shape, ctx, W = tiny
    sp = OD.SamplingParams()
    prompt, ref, table, res = _oracle_run(shape, W, sp, n_new=48, k=13)
    assert any(st.mode == "verify" and st.accepted > 3 for st in res.steps)
    worst, flips = _teacher_forced(sd, shape, ctx, res, prompt, sp, k=13)
    assert flips <= 1


def test_tiny_nucleus_teacher_forced_k13(sd, tiny):
    shape, ctx, W = tiny
    sp = OD.SamplingParams(1.0, 0.95, 10, seed=99)
    prompt, ref, table, res = _oracle_run(shape, W, sp, match=0.6, n_new=32, k=13)
    worst, flips = _teacher_forced(sd, shape, ctx, res, prompt, sp, k=13)
    assert flips <= len(res.steps) * 14 // 4, (flips, len(res.steps))


def test_tiny_kv_append_matches_oracle(sd, tiny):
    """The QKV epilogue writes RoPE'd K and V rows into the cache at slots len .. len+q-1."""
    shape, ctx, W = tiny
    prompt = synth.prompt_ids(0, 0, 40, 4096)
    kvo = OM.KVCache(shape, 1, 64)
    OM.prefill(W, kvo, 0, prompt.tolist())
    kv = ctx.kv(1, 64)
    ctx.prefill(kv, 0, prompt.cuda())
    for l in range(shape.n_layers):
        k, v = ctx.kv_read(kv, l, 0, 0, 40)
        ek = np.abs(k.float().cpu().numpy() - kvo.K[l][0][:, :40]).max()
        ev = np.abs(v.float().cpu().numpy() - kvo.V[l][0][:, :40]).max()
        scale = max(np.abs(kvo.K[l][0][:, :40]).max(), np.abs(kvo.V[l][0][:, :40]).max())
        assert ek <= 2e-2 * scale and ev <= 2e-2 * scale, (l, ek, ev, scale)
    assert ctx.kv_lengths(kv).item() == 40


def test_tiny_device_loop_equals_plain_greedy(sd, tiny):
    """The whole loop on the device (build_block -> block_forward -> accept, no host in between)
    emits the plain-greedy sequence of the oracle (Sec. 2.1.1), up to near-tie flips."""
    shape, ctx, W = tiny
    sp = OD.SamplingParams()
    prompt, ref, table, res = _oracle_run(shape, W, sp)
    kv = ctx.kv(1, PROMPT + N_NEW + 4 * Q)
    ctx.prefill(kv, 0, prompt[:-1].cuda())
    cap = PROMPT + N_NEW + 4 * Q
    tab = torch.zeros(cap + 16, dtype=torch.int32)
    tab[:min(cap + 16, table.numel())] = table[:cap + 16]
    tab = tab.cuda()
    logits = torch.empty(Q, shape.vocab, device="cuda")
    acc = torch.ones(1, dtype=torch.int32, device="cuda")
    out = torch.zeros(Q, dtype=torch.int32, device="cuda")
    out[0] = int(prompt[-1])
    toks = torch.empty(Q, dtype=torch.int32, device="cuda")
    emitted = []
    per_loop = []
    while len(emitted) < N_NEW:
        n_loop = 0
        for mode in (1, 2):
            ctx.build_block(kv, mode, out, acc, toks, 1, Q, draft_table=tab if mode == 2 else None,
                            table_stride=tab.numel())
            ctx.block_forward(kv, toks, logits, 1, Q)
            ctx.accept_greedy(kv, logits, toks, 1, Q, 0 if mode == 1 else K, acc, out)
            a = int(acc.item())
            emitted += out[:a].cpu().tolist()
            n_loop += a
        per_loop.append(n_loop)
    # the stub drafts the true token with probability 0.7, so loops accept drafts (Sec. 2.1.1: 2..k+2 per loop)
    assert all(2 <= n <= K + 2 for n in per_loop)
    assert np.mean(per_loop) > 3.0, per_loop
    emitted = emitted[:N_NEW]
    same = sum(int(a == b) for a, b in zip(emitted, ref[:N_NEW]))
    first_diff = next((i for i, (a, b) in enumerate(zip(emitted, ref)) if a != b), None)
    assert same == N_NEW or first_diff is not None and first_diff > 8, (first_diff, emitted[:10], ref[:10])
    assert ctx.get_error() == 0


def test_block_equals_sequential_on_gpu(sd, tiny):
    """A q-row block forward equals q single-row forwards (within the logit tolerance)."""
    shape, ctx, W = tiny
    prompt = synth.prompt_ids(0, 5, 30, 4096)
    blk = torch.tensor([5, 17, 4096, 4096, 900, 3], dtype=torch.int32, device="cuda")
    kv = ctx.kv(1, 64)
    ctx.prefill(kv, 0, prompt.cuda())
    lb = torch.empty(Q, shape.vocab, device="cuda")
    ctx.block_forward(kv, blk, lb, 1, Q)
    kv2 = ctx.kv(1, 64)
    ctx.prefill(kv2, 0, prompt.cuda())
    l1 = torch.empty(1, shape.vocab, device="cuda")
    for j in range(Q):
        ctx.block_forward(kv2, blk[j:j + 1].contiguous(), l1, 1, 1)
        ctx.kv_commit(kv2, torch.tensor([30 + j + 1], dtype=torch.int32, device="cuda"), 1)
        assert (l1[0] - lb[j]).abs().max().item() <= 1e-3


def test_batched_rows_are_independent(sd, tiny):
    """b = 4 sequences with different contexts in one block forward equal four b = 1 passes."""
    shape, ctx, W = tiny
    b = 4
    kv = ctx.kv(b, 128)
    kv1 = ctx.kv(1, 128)
    toks = synth.uniform_ids(0, 55, b * Q, 4104).cuda()
    lens = [10, 33, 64, 100]
    for s in range(b):
        p = synth.prompt_ids(0, 10 + s, lens[s], 4096).cuda()
        ctx.prefill(kv, s, p)
    lg = torch.empty(b * Q, shape.vocab, device="cuda")
    ctx.block_forward(kv, toks, lg, b, Q)
    for s in range(b):
        kv1 = ctx.kv(1, 128)
        ctx.prefill(kv1, 0, synth.prompt_ids(0, 10 + s, lens[s], 4096).cuda())
        l1 = torch.empty(Q, shape.vocab, device="cuda")
        ctx.block_forward(kv1, toks[s * Q:(s + 1) * Q].contiguous(), l1, 1, Q)
        assert (l1 - lg[s * Q:(s + 1) * Q]).abs().max().item() <= 1e-3
