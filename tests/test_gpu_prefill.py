"""Parity of the prefill path (the step before the decode loop) against the oracle.

Prefill runs chunks of up to 64 positions through one block forward each, attended as causal
groups of 16 rows that share the sequence's cache; a tail shorter than a group runs as one
block.  Checked:
  * tiny model, prompt lengths that exercise full chunks, partial chunks and the tail: every
    layer's K / V rows against the oracle's prefill, then the logits of a decode block on top;
  * grouped prefill equals the same prompt fed as 16-row blocks (the decode path) on the GPU;
  * 7B shape at the bench's prompt length (2047): layer 0's K / V rows of every position
    against the oracle's arithmetic for that layer, and the last layer against 16-row blocks.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import model as OM

pytestmark = pytest.mark.gpu

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


def _kv_close(got, ref, rel=2e-2):
    scale = np.abs(ref).max()
    err = np.abs(got - ref).max()
    assert err <= rel * scale, (err, scale)


@pytest.mark.parametrize("n", [5, 16, 40, 64, 131, 200])
def test_prefill_matches_oracle(sd, tiny, n):
    shape, ctx, W = tiny
    prompt = synth.prompt_ids(0, 60 + n, n, 4096)
    cap = n + 16
    kvo = OM.KVCache(shape, 1, cap)
    OM.prefill(W, kvo, 0, prompt.tolist())
    kv = ctx.kv(1, cap)
    ctx.prefill(kv, 0, prompt.cuda())
    assert ctx.kv_lengths(kv).item() == n
    for l in range(shape.n_layers):
        k, v = ctx.kv_read(kv, l, 0, 0, n)
        _kv_close(k.float().cpu().numpy(), kvo.K[l][0][:, :n])
        _kv_close(v.float().cpu().numpy(), kvo.V[l][0][:, :n])
    # a decode block on top of the prefilled cache
    blk = synth.uniform_ids(0, 61, 6, shape.vocab)
    lg = torch.empty(6, shape.vocab, device="cuda")
    ctx.block_forward(kv, blk.cuda(), lg, 1, 6)
    ref = OM.block_forward(W, kvo, 0, blk.tolist())
    got = lg.cpu().numpy().astype(np.float64)
    err = np.abs(got - ref).max()
    rel = np.sqrt(((got - ref) ** 2).mean() / (ref ** 2).mean())
    assert err <= LOGIT_MAX_ABS and rel <= LOGIT_REL_RMS, (err, rel)
    assert ctx.get_error() == 0


def test_prefill_equals_blocks_on_gpu(sd, tiny):
    """Grouped chunks and 16-row decode blocks write the same cache (up to rounding order)."""
    shape, ctx, W = tiny
    n = 150
    prompt = synth.prompt_ids(0, 70, n, 4096).cuda()
    kv1 = ctx.kv(1, n + 8)
    ctx.prefill(kv1, 0, prompt)
    kv2 = ctx.kv(1, n + 8)
    lg = torch.empty(16, shape.vocab, device="cuda")
    for i in range(0, n, 16):
        blk = prompt[i:i + 16].contiguous()
        ctx.block_forward(kv2, blk, lg[:blk.numel()], 1, blk.numel())
        ctx.kv_commit(kv2, torch.tensor([i + blk.numel()], dtype=torch.int32, device="cuda"), 1)
    for l in range(shape.n_layers):
        a = ctx.kv_read(kv1, l, 0, 0, n)
        b = ctx.kv_read(kv2, l, 0, 0, n)
        for x, y in zip(a, b):
            x, y = x.float(), y.float()
            assert (x - y).abs().max().item() <= 1e-2 * y.abs().max().item()
    assert ctx.get_error() == 0


def test_prefill_full_size_7b(sd):
    """7B shape, the bench's prompt (2047 positions): layer 0's K / V of every position against
    the oracle's arithmetic for that layer (RMSNorm, projections, RoPE); the last layer against
    the same prompt fed as 16-row blocks."""
    shape = synth.SHAPES["7b"]
    P = 2047
    w = synth.make_model(shape, seed=0, device="cuda")
    ctx = sd.Context(shape, w, max_position=P + 64)
    prompt = synth.prompt_ids(0, 0, P, shape.adaptive_id)
    kv = ctx.kv(1, P + 16)
    ctx.prefill(kv, 0, prompt.cuda())
    assert ctx.kv_lengths(kv).item() == P
    # layer 0 in the oracle's arithmetic (fp64), every position
    l0 = w["layers"][0]
    x = OM.rmsnorm(OM.to64(w["embed"][prompt.long().cuda()].cpu()), OM.to64(l0["attn_norm"].cpu()), shape.rms_eps)
    H, hd = shape.n_heads, shape.head_dim
    kref = OM.rope(OM.linear(x, OM.to64(l0["wk"].cpu())).reshape(P, H, hd), list(range(P)), shape.rope_theta)
    vref = OM.linear(x, OM.to64(l0["wv"].cpu())).reshape(P, H, hd)
    k, v = ctx.kv_read(kv, 0, 0, 0, P)
    _kv_close(k.float().cpu().numpy(), kref.transpose(1, 0, 2))
    _kv_close(v.float().cpu().numpy(), vref.transpose(1, 0, 2))
    # the last layer: grouped chunks against 16-row blocks
    kv2 = ctx.kv(1, P + 16)
    pc = prompt.cuda()
    lg = torch.empty(16, shape.vocab, device="cuda")
    for i in range(0, P, 16):
        blk = pc[i:i + 16].contiguous()
        ctx.block_forward(kv2, blk, lg[:blk.numel()], 1, blk.numel())
        ctx.kv_commit(kv2, torch.tensor([i + blk.numel()], dtype=torch.int32, device="cuda"), 1)
    last = shape.n_layers - 1
    for x1, x2 in zip(ctx.kv_read(kv, last, 0, 0, P), ctx.kv_read(kv2, last, 0, 0, P)):
        x1, x2 = x1.float(), x2.float()
        assert (x1 - x2).abs().max().item() <= 2e-2 * x2.abs().max().item()
    assert ctx.get_error() == 0
