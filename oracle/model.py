"""Oracle: Llama-architecture block forward of q new positions (fp64, CPU).

TEST INFRASTRUCTURE ONLY (see oracle/__init__.py).

The paper runs an unmodified decoder-only LLM (CodeLlama); the semantic
adaptive tokens are ordinary vocabulary ids, so the model structure is
untouched (Abstract; Sec. 1; Fig. 2 caption; Sec. 3.2).  Draft step 1
(Eq. 1) and draft step 2 (Eq. 2) each evaluate P_theta at every position of
a block of q = k + 1 appended tokens in one pass; this module computes the
logits of that pass.

The decoder is the standard Llama block (the paper names no variant):

    h   = E[t]
    per layer:  x = RMSNorm(h; g_attn)
                q, k, v = x Wq^T, x Wk^T, x Wv^T ; q, k <- RoPE(position)
                append k, v to the cache at slots len .. len+q-1
                o = softmax(q K^T / sqrt(hd) + mask) V      (block-causal)
                h = h + o Wo^T
                x = RMSNorm(h; g_ffn)
                h = h + (silu(x Wgate^T) * (x Wup^T)) Wdown^T
    logits = RMSNorm(h; g_final) Whead^T

Readings where the paper is silent (all configurable):
  * RoPE pairs dimension i with i + hd/2 ("rotate half"), frequency
    theta_i = base^(-2i/hd), angle = position * theta_i.
  * Row j of a block sees cache slots [0, len) and block rows 0..j.
  * Every linear map is computed row by row, so a row's result never
    depends on how many rows share the block (a q-row block is bit-identical
    to q single-token steps, the invariant the method relies on).

All arithmetic is fp64; weights are the bf16 values widened exactly.

Diagnostic mode (KVCache(kv_bf16=True)): the K and V rows are rounded to bf16
(round to nearest even) when written, as a cache stored in bf16 holds them; every
other step stays fp64.  Comparing a bf16-cache implementation with this mode
separates its arithmetic errors from the cache's storage precision.
"""
from __future__ import annotations

import math
from typing import Callable, Dict, List, Optional, Sequence

import numpy as np
import torch


def to64(t) -> np.ndarray:
    """Widen a (bf16) torch tensor or array to an fp64 numpy array, exactly."""
    if isinstance(t, torch.Tensor):
        return t.detach().to("cpu").to(torch.float64).numpy()
    return np.asarray(t, dtype=np.float64)


def rmsnorm(h: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """x = h / sqrt(mean(h^2) + eps) * g over the last axis."""
    ms = np.mean(h * h, axis=-1, keepdims=True)
    return h / np.sqrt(ms + eps) * g


def rope(x: np.ndarray, pos: Sequence[int], theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing.  x: [n, H, hd]; pos: [n]."""
    n, H, hd = x.shape
    half = hd // 2
    i = np.arange(half, dtype=np.float64)
    inv_freq = theta ** (-2.0 * i / hd)                          # theta_i
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def linear(x: np.ndarray, W: np.ndarray) -> np.ndarray:
    """y = x W^T, one row at a time (rows never interact)."""
    out = np.empty((x.shape[0], W.shape[0]), dtype=np.float64)
    for r in range(x.shape[0]):
        out[r] = W @ x[r]
    return out


def attend(q: np.ndarray, K: np.ndarray, V: np.ndarray, n_visible: Sequence[int]) -> np.ndarray:
    """softmax(q k^T / sqrt(hd)) v per row and head over the first n_visible[j] slots.

    q: [n, H, hd]; K, V: [H, slots, hd].  Returns [n, H, hd].
    """
    n, H, hd = q.shape
    out = np.empty_like(q)
    scale = 1.0 / math.sqrt(hd)
    for j in range(n):
        nv = int(n_visible[j])
        for h in range(H):
            s = (K[h, :nv] @ q[j, h]) * scale
            e = np.exp(s - s.max())
            p = e / e.sum()
            out[j, h] = p @ V[h, :nv]
    return out


def attend_rows(q: np.ndarray, K: np.ndarray, V: np.ndarray, L0: int,
                visible: Sequence[Sequence[int]]) -> np.ndarray:
    """softmax(q k^T / sqrt(hd)) v per row and head over the committed slots [0, L0) and the
    block slots L0 + i for i in visible[j] (ascending), the tree-attention mask of Sec. 2.1.2.

    With visible[j] = 0..j this is attend() with n_visible[j] = L0 + j + 1, in the same
    slot order, so the two agree bit for bit.
    """
    n, H, hd = q.shape
    out = np.empty_like(q)
    scale = 1.0 / math.sqrt(hd)
    for j in range(n):
        slots = list(range(L0)) + [L0 + int(i) for i in sorted(visible[j])]
        for h in range(H):
            s = (K[h, slots] @ q[j, h]) * scale
            e = np.exp(s - s.max())
            p = e / e.sum()
            out[j, h] = p @ V[h, slots]
    return out


class Weights:
    """fp64 view of a synth-style weight dict, widened lazily (optionally cached)."""

    def __init__(self, shape, tensors: Optional[dict] = None,
                 provider: Optional[Callable[[str, int], "torch.Tensor"]] = None,
                 cache: bool = True):
        self.shape = shape
        self._tensors = tensors
        self._provider = provider
        self._cache: Dict[tuple, np.ndarray] = {}
        self._use_cache = cache

    def get(self, name: str, layer: int = -1) -> np.ndarray:
        key = (name, layer)
        if key in self._cache:
            return self._cache[key]
        if self._tensors is not None:
            t = self._tensors[name] if layer < 0 else self._tensors["layers"][layer][name]
        else:
            t = self._provider(name, layer)
        a = to64(t)
        if self._use_cache:
            self._cache[key] = a
        return a


def round_bf16(x: np.ndarray) -> np.ndarray:
    """x rounded to the nearest bf16 value (ties to even), returned in fp64."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float64)).to(torch.bfloat16).to(torch.float64).numpy()


class KVCache:
    """Per-layer K and V (fp64) for b sequences: [L][b][H][max_len][hd], plus len[b].
    kv_bf16: store the rows rounded to bf16 (the diagnostic mode of the module docstring)."""

    def __init__(self, shape, batch: int, max_len: int, kv_bf16: bool = False):
        L, H, hd = shape.n_layers, shape.n_heads, shape.head_dim
        self.K = [np.zeros((batch, H, max_len, hd)) for _ in range(L)]
        self.V = [np.zeros((batch, H, max_len, hd)) for _ in range(L)]
        self.len = [0] * batch
        self.max_len = max_len
        self.kv_bf16 = kv_bf16

    def copy(self) -> "KVCache":
        c = KVCache.__new__(KVCache)
        c.K = [k.copy() for k in self.K]
        c.V = [v.copy() for v in self.V]
        c.len = list(self.len)
        c.max_len = self.max_len
        c.kv_bf16 = self.kv_bf16
        return c


def block_forward(W: Weights, kv: KVCache, seq: int, tokens: Sequence[int],
                  positions: Optional[Sequence[int]] = None,
                  layers: Optional[Sequence[int]] = None,
                  final: bool = True,
                  visible: Optional[Sequence[Sequence[int]]] = None) -> np.ndarray:
    """Logits [n, V] of the n = q block rows of sequence `seq`.

    Block rows occupy cache slots len .. len+n-1 (written here; `kv.len` is
    not advanced -- committing is the acceptance step's job).  RoPE uses
    `positions` when given, else the slot index.  `layers` restricts the
    pass to a subset (used only to time a bounded sample).  `visible[j]`,
    when given, lists the block rows row j attends to (a tree mask, see
    oracle/tree.py); the default is block-causal (rows 0..j).
    """
    shape = W.shape
    n = len(tokens)
    L0 = kv.len[seq]
    if L0 + n > kv.max_len:
        raise ValueError("KV capacity exceeded")
    pos = list(positions) if positions is not None else [L0 + j for j in range(n)]
    H, hd, eps = shape.n_heads, shape.head_dim, shape.rms_eps
    E = W.get("embed")
    h = np.stack([E[int(t)] for t in tokens]).astype(np.float64)
    n_visible = [L0 + j + 1 for j in range(n)]
    for l in (range(shape.n_layers) if layers is None else layers):
        x = rmsnorm(h, W.get("attn_norm", l), eps)
        q = linear(x, W.get("wq", l)).reshape(n, H, hd)
        k = linear(x, W.get("wk", l)).reshape(n, H, hd)
        v = linear(x, W.get("wv", l)).reshape(n, H, hd)
        q = rope(q, pos, shape.rope_theta)
        k = rope(k, pos, shape.rope_theta)
        if kv.kv_bf16:
            k, v = round_bf16(k), round_bf16(v)
        kv.K[l][seq][:, L0:L0 + n] = k.transpose(1, 0, 2)
        kv.V[l][seq][:, L0:L0 + n] = v.transpose(1, 0, 2)
        if visible is None:
            o = attend(q, kv.K[l][seq], kv.V[l][seq], n_visible)
        else:
            o = attend_rows(q, kv.K[l][seq], kv.V[l][seq], L0, visible)
        h = h + linear(o.reshape(n, H * hd), W.get("wo", l))
        x = rmsnorm(h, W.get("ffn_norm", l), eps)
        a = silu(linear(x, W.get("w_gate", l))) * linear(x, W.get("w_up", l))
        h = h + linear(a, W.get("w_down", l))
    if not final:
        return h
    x = rmsnorm(h, W.get("final_norm"), eps)
    return linear(x, W.get("lm_head"))


def prefill(W: Weights, kv: KVCache, seq: int, tokens: Sequence[int], chunk: int = 16) -> None:
    """Run `tokens` through the model in blocks of `chunk` rows and commit them."""
    for i in range(0, len(tokens), chunk):
        blk = list(tokens[i:i + chunk])
        block_forward(W, kv, seq, blk, final=False)
        kv.len[seq] += len(blk)
