"""Pins of the oracle's whole decoder forward (oracle/model.py block_forward) on weight
settings where it reduces to something with a plain definition, computed here with
torch's library routines (rms_norm, linear, silu, scaled_dot_product_attention) and the
complex-number form of RoPE -- none of which the oracle uses.

A Llama decoder layer adds two branches to the residual stream: attention (ending in the
O projection) and the SwiGLU MLP (ending in the down projection).  Zeroing the last
projection of a branch removes it exactly, so:
  * both branches off in every layer: logits = LM head (final RMSNorm (embedding));
  * MLP only: each layer adds W_down (silu(W_gate x) * W_up x), x = RMSNorm_ffn(h);
  * attention only, one key: softmax over a single slot is 1, so the branch adds
    W_o W_v RMSNorm_attn(h) whatever Q, K and RoPE are; equal tokens have equal values,
    so the same holds for every row of a block of one repeated token;
  * attention only, one layer: causal attention over the block, the library's SDPA.
A dropped branch, a swapped gate / up, a norm applied in the wrong place, values taken
from K, or a RoPE sign error each fails one of these.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

import synth
from oracle import model as M


def _t64(x):
    return x.detach().to(torch.float64)


@pytest.fixture(scope="module")
def shape():
    return synth.SHAPES["tiny"]


def _weights(shape, zero_o=(), zero_down=()):
    w = synth.make_model(shape, seed=3, device="cpu", gain_std=0.1)
    for l in zero_o:
        w["layers"][l]["wo"].zero_()
    for l in zero_down:
        w["layers"][l]["w_down"].zero_()
    return w


def _rms(h, g, eps):
    return F.rms_norm(h, (h.shape[-1],), weight=g, eps=eps)


def _head(w, h, eps):
    return F.linear(_rms(h, _t64(w["final_norm"]), eps), _t64(w["lm_head"]))


def _mlp(w, l, h, eps):
    x = _rms(h, _t64(w["layers"][l]["ffn_norm"]), eps)
    a = F.silu(F.linear(x, _t64(w["layers"][l]["w_gate"]))) * F.linear(x, _t64(w["layers"][l]["w_up"]))
    return F.linear(a, _t64(w["layers"][l]["w_down"]))


def _rope_complex(x, pos, theta):
    """x: [n, H, hd] rotated by e^{i pos theta_j} on the pairs (x_j, x_{j + hd/2})."""
    n, H, hd = x.shape
    half = hd // 2
    z = torch.complex(x[..., :half], x[..., half:])
    freq = theta ** (-2.0 * torch.arange(half, dtype=torch.float64) / hd)
    rot = torch.polar(torch.ones(n, half, dtype=torch.float64), torch.tensor(pos, dtype=torch.float64)[:, None] * freq)
    z = z * rot[:, None, :]
    return torch.cat([z.real, z.imag], dim=-1)


def _forward(shape, w, tokens, L0=0, prefix=None):
    W = M.Weights(shape, tensors=w)
    kv = M.KVCache(shape, 1, 64)
    if prefix:
        M.prefill(W, kv, 0, prefix)
    assert kv.len[0] == L0
    return torch.from_numpy(M.block_forward(W, kv, 0, tokens))


def test_both_branches_off_is_norm_and_head(shape):
    L = shape.n_layers
    w = _weights(shape, zero_o=range(L), zero_down=range(L))
    toks = [5, 17, shape.vocab - 1, 0, 17]
    got = _forward(shape, w, toks)
    E = _t64(w["embed"])[toks]
    torch.testing.assert_close(got, _head(w, E, shape.rms_eps), rtol=1e-12, atol=1e-12)


def test_mlp_only_layers_compose_in_order(shape):
    """wo = 0 everywhere: h_{l+1} = h_l + MLP_l(h_l), whatever the cache holds."""
    L = shape.n_layers
    w = _weights(shape, zero_o=range(L))
    toks = [9, 4000, 9, 123]
    prefix = [7, 8, 9, 10, 11, 12]
    got = _forward(shape, w, toks, L0=len(prefix), prefix=prefix)
    h = _t64(w["embed"])[toks]
    for l in range(L):
        h = h + _mlp(w, l, h, shape.rms_eps)
    torch.testing.assert_close(got, _head(w, h, shape.rms_eps), rtol=1e-10, atol=1e-10)
    # the layer order matters: applying the two MLPs the other way round differs
    h2 = _t64(w["embed"])[toks]
    for l in reversed(range(L)):
        h2 = h2 + _mlp(w, l, h2, shape.rms_eps)
    assert (got - _head(w, h2, shape.rms_eps)).abs().max() > 1e-3


def test_single_key_attention_adds_wo_wv(shape):
    """Attention only in layer 0: a one-token block at slot 0 attends to itself alone."""
    L = shape.n_layers
    w = _weights(shape, zero_o=range(1, L), zero_down=range(L))
    lw = w["layers"][0]
    eps = shape.rms_eps
    for tok in (3, 2048):
        e = _t64(w["embed"])[[tok]]
        v = F.linear(_rms(e, _t64(lw["attn_norm"]), eps), _t64(lw["wv"]))
        h = e + F.linear(v, _t64(lw["wo"]))
        expect = _head(w, h, eps)
        torch.testing.assert_close(_forward(shape, w, [tok]), expect, rtol=1e-10, atol=1e-10)
        # a block of the same token: every key carries the same value, so every row is the same
        got = _forward(shape, w, [tok] * 5)
        torch.testing.assert_close(got, expect.expand(5, -1), rtol=1e-10, atol=1e-10)


def test_one_attention_layer_is_causal_sdpa(shape):
    """Attention only in layer 0, distinct tokens: q, k through RoPE (complex form), then
    the library's causal scaled-dot-product attention over the block."""
    L = shape.n_layers
    w = _weights(shape, zero_o=range(1, L), zero_down=range(L))
    lw = w["layers"][0]
    eps, H, hd = shape.rms_eps, shape.n_heads, shape.head_dim
    toks = [11, 250, 3999, 42, 7, 1000]
    n = len(toks)
    e = _t64(w["embed"])[toks]
    x = _rms(e, _t64(lw["attn_norm"]), eps)
    pos = list(range(n))
    q = _rope_complex(F.linear(x, _t64(lw["wq"])).reshape(n, H, hd), pos, shape.rope_theta)
    k = _rope_complex(F.linear(x, _t64(lw["wk"])).reshape(n, H, hd), pos, shape.rope_theta)
    v = F.linear(x, _t64(lw["wv"])).reshape(n, H, hd)
    o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1), is_causal=True)
    h = e + F.linear(o.transpose(0, 1).reshape(n, H * hd), _t64(lw["wo"]))
    torch.testing.assert_close(_forward(shape, w, toks), _head(w, h, eps), rtol=1e-9, atol=1e-9)
    # RoPE with the opposite sign gives other logits (the pin sees the rotation's direction)
    qm = _rope_complex(F.linear(x, _t64(lw["wq"])).reshape(n, H, hd), [-p for p in pos], shape.rope_theta)
    km = _rope_complex(F.linear(x, _t64(lw["wk"])).reshape(n, H, hd), pos, shape.rope_theta)
    om = F.scaled_dot_product_attention(qm.transpose(0, 1), km.transpose(0, 1), v.transpose(0, 1), is_causal=True)
    hm = e + F.linear(om.transpose(0, 1).reshape(n, H * hd), _t64(lw["wo"]))
    assert (_forward(shape, w, toks) - _head(w, hm, eps)).abs().max() > 1e-6
