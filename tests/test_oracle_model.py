"""Pins of the oracle's decoder block forward to closed forms, invariants and library routines."""
import math

import numpy as np
import pytest
import torch

import synth
from oracle import model as M


def test_rmsnorm_closed_form():
    """A constant row c gives c / sqrt(c^2 + eps) * g for every element."""
    g = np.array([0.5, 1.0, 2.0, -1.0])
    for c in (3.0, -0.25, 1e-3):
        out = M.rmsnorm(np.full((1, 4), c), g, 1e-5)
        np.testing.assert_allclose(out[0], c / math.sqrt(c * c + 1e-5) * g, rtol=1e-14)


def test_rmsnorm_unit_rms():
    h = np.random.default_rng(0).normal(0, 7.0, (3, 512))
    out = M.rmsnorm(h, np.ones(512), 0.0)
    np.testing.assert_allclose(np.sqrt((out ** 2).mean(-1)), 1.0, rtol=1e-12)


def test_rope_complex_formulation():
    """Rotate-half RoPE equals multiplying z_i = x_i + i x_{i+hd/2} by e^{i pos theta_i},
    theta_i = base^(-2i/hd) (RoFormer's complex form), a different computation path."""
    rng = np.random.default_rng(1)
    n, H, hd, base = 5, 3, 16, 1e4
    x = rng.normal(size=(n, H, hd))
    pos = [0, 1, 7, 100, 4095]
    got = M.rope(x, pos, base)
    half = hd // 2
    z = x[..., :half] + 1j * x[..., half:]
    freq = np.array([base ** (-2.0 * i / hd) for i in range(half)])
    rot = z * np.exp(1j * np.outer(pos, freq))[:, None, :]
    np.testing.assert_allclose(got[..., :half], rot.real, atol=1e-12)
    np.testing.assert_allclose(got[..., half:], rot.imag, atol=1e-12)


def test_rope_identity_norm_relative():
    rng = np.random.default_rng(2)
    q = rng.normal(size=(1, 1, 64))
    k = rng.normal(size=(1, 1, 64))
    np.testing.assert_array_equal(M.rope(q, [0], 1e4), q)
    np.testing.assert_allclose(np.linalg.norm(M.rope(q, [33], 1e4)), np.linalg.norm(q), rtol=1e-13)
    # <R_m q, R_n k> depends only on m - n
    a = (M.rope(q, [10], 1e4) * M.rope(k, [3], 1e4)).sum()
    b = (M.rope(q, [107], 1e4) * M.rope(k, [100], 1e4)).sum()
    assert abs(a - b) < 1e-10


def test_attend_special_cases():
    rng = np.random.default_rng(3)
    H, hd, slots = 2, 8, 6
    K = rng.normal(size=(H, slots, hd))
    V = rng.normal(size=(H, slots, hd))
    q = rng.normal(size=(1, H, hd))
    # one visible key: the output is that key's value
    np.testing.assert_allclose(M.attend(q, K, V, [1])[0], V[:, 0], atol=1e-14)
    # q = 0: uniform weights, the mean of the visible values
    np.testing.assert_allclose(M.attend(np.zeros((1, H, hd)), K, V, [4])[0], V[:, :4].mean(1), atol=1e-14)


def test_attend_matches_library_sdpa():
    """Block-causal rows against torch's scaled_dot_product_attention with an explicit mask."""
    rng = np.random.default_rng(4)
    H, hd, L0, n = 3, 16, 9, 5
    K = rng.normal(size=(H, L0 + n, hd))
    V = rng.normal(size=(H, L0 + n, hd))
    q = rng.normal(size=(n, H, hd))
    got = M.attend(q, K, V, [L0 + j + 1 for j in range(n)])
    mask = torch.zeros(n, L0 + n, dtype=torch.bool)
    for j in range(n):
        mask[j, :L0 + j + 1] = True
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.tensor(q).permute(1, 0, 2), torch.tensor(K), torch.tensor(V), attn_mask=mask)
    np.testing.assert_allclose(got, ref.permute(1, 0, 2).numpy(), atol=1e-12)


def _weights(shape, tensors):
    return M.Weights(shape, tensors=tensors)


def test_block_equals_sequential_steps(tiny_shape, tiny_model_cpu):
    """A q-row block forward equals q single-token steps, bit for bit (Eq. 1-2 evaluate
    every appended position in one pass of the unchanged model)."""
    W = _weights(tiny_shape, tiny_model_cpu)
    prompt = synth.prompt_ids(0, 0, 20, 4096).tolist()
    kv = M.KVCache(tiny_shape, 1, 64)
    M.prefill(W, kv, 0, prompt)
    blk = [5, 17, 4096, 4096, 900, 3]
    kv_a = kv.copy()
    blk_logits = M.block_forward(W, kv_a, 0, blk)
    kv_b = kv.copy()
    for j, t in enumerate(blk):
        lj = M.block_forward(W, kv_b, 0, [t])
        kv_b.len[0] += 1
        np.testing.assert_array_equal(lj[0], blk_logits[j])
    for l in range(tiny_shape.n_layers):
        np.testing.assert_array_equal(kv_a.K[l][0][:, :26], kv_b.K[l][0][:, :26])


def test_cached_decode_matches_full_causal_recompute(tiny_shape, tiny_model_cpu):
    """The incremental (KV-cache, block-causal) forward equals a cache-free causal forward
    of the whole sequence that uses torch's causal SDPA for attention."""
    sh = tiny_shape
    W = _weights(sh, tiny_model_cpu)
    seqtoks = synth.prompt_ids(0, 3, 23, 4096).tolist()
    kv = M.KVCache(sh, 1, 64)
    M.prefill(W, kv, 0, seqtoks[:17])
    got = M.block_forward(W, kv, 0, seqtoks[17:])
    # cache-free reference
    T = len(seqtoks)
    H, hd = sh.n_heads, sh.head_dim
    t64 = lambda a: torch.tensor(a, dtype=torch.float64)
    h = t64(W.get("embed")[seqtoks])
    pos = torch.arange(T, dtype=torch.float64)
    inv = sh.rope_theta ** (-2.0 * torch.arange(hd // 2, dtype=torch.float64) / hd)
    ang = pos[:, None] * inv[None]
    cos, sin = torch.cos(ang)[:, None], torch.sin(ang)[:, None]

    def rot(x):
        x1, x2 = x[..., :hd // 2], x[..., hd // 2:]
        return torch.cat([x1 * cos - x2 * sin, x2 * cos + x1 * sin], -1)

    def rms(x, g):
        return x * torch.rsqrt((x * x).mean(-1, keepdim=True) + sh.rms_eps) * t64(g)

    for l in range(sh.n_layers):
        x = rms(h, W.get("attn_norm", l))
        q = rot((x @ t64(W.get("wq", l)).T).view(T, H, hd))
        k = rot((x @ t64(W.get("wk", l)).T).view(T, H, hd))
        v = (x @ t64(W.get("wv", l)).T).view(T, H, hd)
        o = torch.nn.functional.scaled_dot_product_attention(
            q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1), is_causal=True)
        h = h + o.transpose(0, 1).reshape(T, H * hd) @ t64(W.get("wo", l)).T
        x = rms(h, W.get("ffn_norm", l))
        g = x @ t64(W.get("w_gate", l)).T
        h = h + (torch.nn.functional.silu(g) * (x @ t64(W.get("w_up", l)).T)) @ t64(W.get("w_down", l)).T
    ref = rms(h, W.get("final_norm")) @ t64(W.get("lm_head")).T
    np.testing.assert_allclose(got, ref[17:].numpy(), atol=1e-10, rtol=1e-10)


def test_explicit_positions_equal_implicit(tiny_shape, tiny_model_cpu):
    W = _weights(tiny_shape, tiny_model_cpu)
    kv = M.KVCache(tiny_shape, 1, 32)
    M.prefill(W, kv, 0, [1, 2, 3, 4])
    a = M.block_forward(W, kv.copy(), 0, [9, 8, 7])
    b = M.block_forward(W, kv.copy(), 0, [9, 8, 7], positions=[4, 5, 6])
    np.testing.assert_array_equal(a, b)


def test_norm_gain_matters(tiny_shape, tiny_model_cpu, tiny_model_cpu_unit_gain):
    """The test model's gains differ from 1, so a dropped gain changes the logits."""
    a = M.block_forward(_weights(tiny_shape, tiny_model_cpu), M.KVCache(tiny_shape, 1, 8), 0, [3])
    b = M.block_forward(_weights(tiny_shape, tiny_model_cpu_unit_gain), M.KVCache(tiny_shape, 1, 8), 0, [3])
    assert np.abs(a - b).max() > 1e-3


def test_round_bf16_ties_to_even():
    """bf16 keeps 8 significant bits: the spacing just above 1 is 2^-7."""
    x = np.array([1.0, 1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, 1 + 2.0 ** -8 + 2.0 ** -20, -(1 + 2.0 ** -8),
                  3.0 * 2.0 ** -130, 1.0 + 2.0 ** -7])
    want = np.array([1.0, 1.0, 1 + 2.0 ** -6, 1 + 2.0 ** -7, -1.0, 3.0 * 2.0 ** -130, 1.0 + 2.0 ** -7])
    np.testing.assert_array_equal(M.round_bf16(x), want)


def test_bf16_cache_mode(tiny_shape, tiny_model_cpu):
    """Diagnostic mode: cached K / V rows are bf16 values, a block still equals the
    sequential steps bit for bit, and the logits move by the cache's rounding only."""
    W = _weights(tiny_shape, tiny_model_cpu)
    prompt = synth.prompt_ids(0, 5, 30, 4096).tolist()
    blk = [7, 4096, 11, 2000, 4096, 8]
    exact, rounded = M.KVCache(tiny_shape, 1, 64), M.KVCache(tiny_shape, 1, 64, kv_bf16=True)
    M.prefill(W, exact, 0, prompt)
    M.prefill(W, rounded, 0, prompt)
    assert rounded.copy().kv_bf16
    kv_a = rounded.copy()
    la = M.block_forward(W, kv_a, 0, blk)
    for l in range(tiny_shape.n_layers):
        K = kv_a.K[l][0][:, :36]
        np.testing.assert_array_equal(M.round_bf16(K), K)
        assert not np.array_equal(M.round_bf16(exact.K[l][0][:, :30]), exact.K[l][0][:, :30])
    kv_b = rounded.copy()
    for j, t in enumerate(blk):
        lj = M.block_forward(W, kv_b, 0, [t])
        kv_b.len[0] += 1
        np.testing.assert_array_equal(lj[0], la[j])
    le = M.block_forward(W, exact.copy(), 0, blk)
    d = np.abs(la - le).max()
    assert 0 < d < 0.05 * np.abs(le).max(), d
