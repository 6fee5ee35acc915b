"""Seeded synthetic inputs for the SDSAT block decode step.

This module is shared by the CPU oracle side (tests, bench's CPU baseline)
and the CUDA side (tests, bench).  It holds none of the method's arithmetic:
it only turns (seed, stream, element index) into model weights, prompt token
ids, KV-cache contents and draft-stub tables, and it names the model shapes
the workloads use.

Generator.  Every value comes from a counter-based hash, so any element (or
any subset of rows) of any tensor can be produced independently, on the CPU
or on a CUDA device, with bit-identical results:

    key1 = fmix32(seed * 0x9E3779B1 + stream)        (mod 2^32)
    key2 = fmix32(key1 ^ 0x5BD1E995)
    u32(i) = fmix32(fmix32(i ^ key1) + key2)          (mod 2^32)

where fmix32 is the 32-bit finaliser of MurmurHash3 (Appleby, 2008; public
domain): x ^= x>>16; x *= 0x85EBCA6B; x ^= x>>13; x *= 0xC2B2AE35; x ^= x>>16.
Only integer operations are used (each 32x32-bit multiply is split into
16-bit halves so that int64 tensors never overflow), and the single
float step is an exact int->fp32 conversion followed by one correctly
rounded fp32 multiply and a round-to-nearest-even cast to bf16, which are
the same on every IEEE device.

"N(0, std)" weights are the standardised sum of four 16-bit uniforms
(Irwin-Hall with n = 4): mean 0, standard deviation exactly `std` (up to the
bf16 rounding), support +-3.46 std.  Token ids are uniform through the
multiply-shift map (u32 * n) >> 32.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Sequence

import torch

M32 = 0xFFFFFFFF

# ---------------------------------------------------------------------------
# model shapes of the workloads (Llama-architecture decoders)
# ---------------------------------------------------------------------------


@dataclasses.dataclass(frozen=True)
class ModelShape:
    name: str
    n_layers: int
    d_model: int
    n_heads: int
    head_dim: int
    ffn_dim: int
    vocab: int            # includes the adaptive-token ids
    adaptive_id: int      # the semantic adaptive token (the same id repeated)
    rms_eps: float = 1e-5
    rope_theta: float = 1e4


SHAPES = {
    # 2 layers, d 256, 4 heads x 64, FFN 688, vocab 4096 + 8 adaptive ids
    "tiny": ModelShape("tiny", 2, 256, 4, 64, 688, 4096 + 8, 4096),
    # CodeLlama-7B shape; the adaptive id lives inside the 32016-entry vocab
    "7b": ModelShape("7b", 32, 4096, 32, 128, 11008, 32016, 32011),
    # CodeLlama-13B shape
    "13b": ModelShape("13b", 40, 5120, 40, 128, 13824, 32016, 32011),
}

# per-layer matrix names and their stream offsets
LAYER_MATS = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down", "attn_norm", "ffn_norm")


def weight_shape(shape: ModelShape, name: str):
    d, F, H, hd = shape.d_model, shape.ffn_dim, shape.n_heads, shape.head_dim
    return {
        "wq": (H * hd, d), "wk": (H * hd, d), "wv": (H * hd, d), "wo": (d, H * hd),
        "w_gate": (F, d), "w_up": (F, d), "w_down": (d, F),
        "attn_norm": (d,), "ffn_norm": (d,),
        "embed": (shape.vocab, d), "lm_head": (shape.vocab, d), "final_norm": (d,),
    }[name]


def stream_id(name: str, layer: int = -1) -> int:
    if layer < 0:
        return {"embed": 1, "lm_head": 2, "final_norm": 3}[name]
    return 100 + 16 * layer + LAYER_MATS.index(name)


# ---------------------------------------------------------------------------
# the hash
# ---------------------------------------------------------------------------


def _fmix32_int(x: int) -> int:
    x &= M32
    x ^= x >> 16
    x = (x * 0x85EBCA6B) & M32
    x ^= x >> 13
    x = (x * 0xC2B2AE35) & M32
    x ^= x >> 16
    return x


def _mul32(x: torch.Tensor, c: int) -> torch.Tensor:
    lo, hi = c & 0xFFFF, c >> 16
    return (x * lo + (((x * hi) & 0xFFFF) << 16)) & M32


def _fmix32(x: torch.Tensor) -> torch.Tensor:
    x = x ^ (x >> 16)
    x = _mul32(x, 0x85EBCA6B)
    x = x ^ (x >> 13)
    x = _mul32(x, 0xC2B2AE35)
    x = x ^ (x >> 16)
    return x


def _keys(seed: int, stream: int):
    k1 = _fmix32_int((seed * 0x9E3779B1 + stream) & M32)
    k2 = _fmix32_int(k1 ^ 0x5BD1E995)
    return k1, k2


def u32(seed: int, stream: int, idx: torch.Tensor) -> torch.Tensor:
    """32-bit hash of int64 element indices idx (0 <= idx < 2^32); int64 result."""
    k1, k2 = _keys(seed, stream)
    return _fmix32((_fmix32(idx ^ k1) + k2) & M32)


def u32_int(seed: int, stream: int, i: int) -> int:
    k1, k2 = _keys(seed, stream)
    return _fmix32_int((_fmix32_int(i ^ k1) + k2) & M32)


# ---------------------------------------------------------------------------
# tensors
# ---------------------------------------------------------------------------


def normal_bf16(seed: int, stream: int, shape: Sequence[int], std: float,
                device="cpu", rows: Optional[torch.Tensor] = None,
                chunk_elems: int = 1 << 25) -> torch.Tensor:
    """bf16 tensor of `shape` (rows x cols, or a vector) with values ~ N(0, std).

    Element (r, c) is a function of (seed, stream, r * cols + c) only.  With
    `rows` given, only those rows are produced (shape [len(rows), cols]).
    """
    shape = tuple(int(s) for s in shape)
    cols = shape[-1]
    nrows = 1 if len(shape) == 1 else shape[0]
    if rows is None:
        rows = torch.arange(nrows, dtype=torch.int64, device=device)
    else:
        rows = rows.to(device=device, dtype=torch.int64)
    out = torch.empty((rows.numel(), cols), dtype=torch.bfloat16, device=device)
    scale = torch.tensor(std * math.sqrt(3.0) / 65536.0, dtype=torch.float32, device=device)
    col = torch.arange(cols, dtype=torch.int64, device=device)
    step = max(1, chunk_elems // cols)
    for r0 in range(0, rows.numel(), step):
        r = rows[r0:r0 + step]
        idx = r[:, None] * cols + col[None, :]
        a = u32(seed, stream, 2 * idx)
        b = u32(seed, stream, 2 * idx + 1)
        s = (a & 0xFFFF) + (a >> 16) + (b & 0xFFFF) + (b >> 16) - 131070
        out[r0:r0 + step] = (s.to(torch.float32) * scale).to(torch.bfloat16)
    if len(shape) == 1 and rows.numel() == 1:
        return out[0]
    return out


def normal_f32(seed: int, stream: int, shape: Sequence[int], std: float = 1.0, device="cpu") -> torch.Tensor:
    """fp32 tensor ~ N(0, std) (same Irwin-Hall construction, not rounded to bf16)."""
    shape = tuple(int(s) for s in shape)
    n = int(math.prod(shape))
    idx = torch.arange(n, dtype=torch.int64, device=device)
    a = u32(seed, stream, 2 * idx)
    b = u32(seed, stream, 2 * idx + 1)
    s = (a & 0xFFFF) + (a >> 16) + (b & 0xFFFF) + (b >> 16) - 131070
    scale = torch.tensor(std * math.sqrt(3.0) / 65536.0, dtype=torch.float32, device=device)
    return (s.to(torch.float32) * scale).reshape(shape)


def ones_bf16(n: int, device="cpu") -> torch.Tensor:
    return torch.ones(n, dtype=torch.bfloat16, device=device)


def uniform_ids(seed: int, stream: int, n: int, upper: int, device="cpu") -> torch.Tensor:
    """n token ids uniform in [0, upper), int32."""
    idx = torch.arange(n, dtype=torch.int64, device=device)
    return ((u32(seed, stream, idx) * upper) >> 32).to(torch.int32)


def uniform01(seed: int, stream: int, n: int, device="cpu") -> torch.Tensor:
    """n floats in [0, 1) (fp64), 2^-32 resolution."""
    idx = torch.arange(n, dtype=torch.int64, device=device)
    return u32(seed, stream, idx).to(torch.float64) / 4294967296.0


# ---------------------------------------------------------------------------
# whole models
# ---------------------------------------------------------------------------

WEIGHT_STD = 0.02
PROMPT_STREAM = 1_000_000
STUB_COIN_STREAM = 2_000_000
STUB_ID_STREAM = 3_000_000
KV_STREAM = 4_000_000


def make_weight(shape: ModelShape, name: str, layer: int = -1, seed: int = 0,
                device="cpu", gain_std: float = 0.0) -> torch.Tensor:
    """One weight tensor of the synthetic model, bf16, row-major [out, in].

    Norm gains are 1.0 unless gain_std > 0, in which case they are
    1 + N(0, gain_std) (used by tests so that a dropped gain is visible).
    """
    shp = weight_shape(shape, name)
    if name.endswith("norm"):
        if gain_std <= 0.0:
            return ones_bf16(shp[0], device)
        g = normal_bf16(seed, stream_id(name, layer), (1, shp[0]), gain_std, device)[0]
        return (g.float() + 1.0).to(torch.bfloat16)
    return normal_bf16(seed, stream_id(name, layer), shp, WEIGHT_STD, device)


def make_model(shape: ModelShape, seed: int = 0, device="cpu", gain_std: float = 0.0) -> dict:
    """All weights of the synthetic model as a dict of bf16 tensors.

    Keys: "embed", "lm_head", "final_norm" and "layers" (a list of dicts with
    the LAYER_MATS keys).
    """
    m = {n: make_weight(shape, n, -1, seed, device, gain_std) for n in ("embed", "lm_head", "final_norm")}
    m["layers"] = [{n: make_weight(shape, n, l, seed, device, gain_std) for n in LAYER_MATS}
                   for l in range(shape.n_layers)]
    return m


def prompt_ids(seed: int, seq: int, n: int, upper: int, device="cpu") -> torch.Tensor:
    """Prompt of n ids uniform in [0, upper) for sequence `seq`."""
    return uniform_ids(seed, PROMPT_STREAM + seq, n, upper, device)


def kv_values(seed: int, layer: int, which: int, shape: Sequence[int], std: float = 1.0,
              device="cpu") -> torch.Tensor:
    """Synthetic KV-cache contents (bf16), e.g. [H, len, hd]; which: 0 = K, 1 = V."""
    n = int(math.prod(shape))
    flat = normal_bf16(seed, KV_STREAM + 2 * layer + which, (1, n), std, device)[0]
    return flat.reshape(tuple(shape))


def stub_table(seed: int, seq: int, ref_tokens: torch.Tensor, match_rate: float,
               vocab: int) -> torch.Tensor:
    """Draft-stub table indexed by absolute position.

    Entry p is ref_tokens[p] with probability match_rate (a per-position coin)
    and otherwise an id uniform in [0, vocab).  The stub stands in for the
    drafts a fine-tuned model would propose; it is harness, not method.
    """
    n = ref_tokens.numel()
    dev = ref_tokens.device
    coin = uniform01(seed, STUB_COIN_STREAM + seq, n, dev)
    other = uniform_ids(seed, STUB_ID_STREAM + seq, n, vocab, dev)
    return torch.where(coin < match_rate, ref_tokens.to(torch.int32), other)
