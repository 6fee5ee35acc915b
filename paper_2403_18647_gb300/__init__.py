"""GB300-native SDSAT block decode step: Python binding of libsdsat.

Argument marshalling only: every step of the decode path runs in the CUDA
kernels of libsdsat.so (built in-tree from csrc/ for sm_103a).  PyTorch is
used for device memory and streams.  There is no CPU fallback: if the
library cannot be loaded, importing the binding raises.

    ctx = Context(shape, weights)            # weights: synth-style dict of CUDA bf16 tensors
    kv = ctx.kv(batch, max_len)
    ctx.prefill(kv, seq, prompt_ids)
    ctx.block_forward(kv, tokens, logits, b, q)
    ctx.accept_greedy(kv, logits, tokens, b, q, n_verify, acc, out)
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

from . import build as _build

MAX_Q = 16
MAX_ROWS = 64
MAX_ADAPTIVE = 16
TRACE_WORDS = 8        # words per device trace record

DEV_NAN_LOGITS = 0x1
DEV_TIMEOUT = 0x2
DEV_CAPACITY = 0x4
DEV_TOKEN = 0x8
DEV_POSITION = 0x10


class SdsatError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__("%s: %s (status %d)" % (what, _lib().sdsat_status_string(status).decode(), status))


class Config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("max_position", ctypes.c_int32), ("n_adaptive", ctypes.c_int32),
                ("adaptive_ids", ctypes.c_int32 * MAX_ADAPTIVE)]


class KernelStat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int64), ("total_ms", ctypes.c_double)]


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")]


class Weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p), ("lm_head", ctypes.c_void_p),
                ("layers", ctypes.POINTER(LayerWeights))]


_LIB = None


def _lib():
    global _LIB
    if _LIB is None:
        if _build.is_stale():
            _build.build()
        lib = ctypes.CDLL(_build.LIB)
        P, I, F, U64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_uint64
        sig = {
            "sdsat_create": [ctypes.POINTER(Config), ctypes.POINTER(Weights), P, ctypes.POINTER(P)],
            "sdsat_set_stream": [P, P],
            "sdsat_kv_create": [P, I, I, ctypes.POINTER(P)],
            "sdsat_kv_info": [P, ctypes.POINTER(P), ctypes.POINTER(P), ctypes.POINTER(P),
                              ctypes.POINTER(I), ctypes.POINTER(I)],
            "sdsat_block_forward": [P, P, P, P, I, I, P],
            "sdsat_kv_write": [P, P, I, I, I, I, P, P],
            "sdsat_kv_read": [P, P, I, I, I, I, P, P],
            "sdsat_accept_greedy": [P, P, P, P, I, I, I, P, P, I],
            "sdsat_accept_nucleus": [P, P, P, P, I, I, I, F, F, U64, I, P, P, I],
            "sdsat_kv_commit": [P, P, P, I],
            "sdsat_kv_lengths": [P, P, P, I],
            "sdsat_kv_emitted": [P, P, P, I, I],
            "sdsat_profile_begin": [P, I],
            "sdsat_trace_begin": [P, I],
            "sdsat_trace_end": [P, P, I, ctypes.POINTER(I)],
            "sdsat_profile_end": [P, ctypes.POINTER(KernelStat), I, ctypes.POINTER(I)],
            "sdsat_build_block": [P, P, I, P, P, P, I, I, I, P],
            "sdsat_block_forward_tree": [P, P, P, P, I, I, P],
            "sdsat_accept_tree": [P, P, P, P, P, I, I, F, F, U64, I, P, P, P, I],
            "sdsat_build_tree_block": [P, P, I, P, I, P, P, I, I, I, I, P],
            "sdsat_build_pipelined_block": [P, P, P, P, P, P, P, I, I, I, P],
            "sdsat_accept_pipelined": [P, P, P, P, P, I, I, F, F, U64, I, P, P, I],
            "sdsat_prefill": [P, P, I, P, I],
            "sdsat_get_error": [P, ctypes.POINTER(ctypes.c_uint32)],
            "sdsat_op_gemm": [P, P, I, I, P, I, P],
            "sdsat_op_attention": [P, P, P, P, P, I, I, I, I, I, P],
            "sdsat_op_exp": [P, P, P, I],
            "sdsat_debug_workspace": [P, I, I, P],
            "sdsat_debug_wait_timeout": [P],
            "sdsat_attention_grid": [I, P, I, I, ctypes.POINTER(I), ctypes.POINTER(I)],
        }
        for name, args in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = ctypes.c_int
        lib.sdsat_destroy.argtypes = [P]
        lib.sdsat_destroy.restype = None
        lib.sdsat_kv_destroy.argtypes = [P]
        lib.sdsat_kv_destroy.restype = None
        lib.sdsat_kernel_class_name.argtypes = [ctypes.c_int]
        lib.sdsat_kernel_class_name.restype = ctypes.c_char_p
        lib.sdsat_status_string.argtypes = [ctypes.c_int]
        lib.sdsat_status_string.restype = ctypes.c_char_p
        _LIB = lib
    return _LIB


def lib():
    """The loaded libsdsat (raises if it cannot be built or loaded)."""
    return _lib()


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _check(status: int, what: str):
    if status != 0:
        raise SdsatError(status, what)


def attention_grid(pairs: int, max_clusters, cs_cap: int = 16, num_sms: int = 152):
    """(cluster size, clusters) the attention launches for `pairs` (sequence, head) pairs,
    given max_clusters[c] = the most clusters of c CTAs resident at once (c = 1..16)."""
    arr = (ctypes.c_int32 * 17)(0, *[int(v) for v in list(max_clusters)[1:17]])
    cs, nc = ctypes.c_int(0), ctypes.c_int(0)
    _check(_lib().sdsat_attention_grid(pairs, ctypes.cast(arr, ctypes.c_void_p), cs_cap, num_sms,
                                       ctypes.byref(cs), ctypes.byref(nc)), "sdsat_attention_grid")
    return cs.value, nc.value


def _stream():
    import torch
    return torch.cuda.current_stream().cuda_stream


def make_config(shape, max_position: int = 8192, adaptive_ids=None) -> Config:
    c = Config()
    c.n_layers, c.d_model, c.n_heads = shape.n_layers, shape.d_model, shape.n_heads
    c.n_kv_heads, c.head_dim, c.ffn_dim, c.vocab = shape.n_heads, shape.head_dim, shape.ffn_dim, shape.vocab
    c.rms_eps, c.rope_theta, c.max_position = shape.rms_eps, shape.rope_theta, max_position
    ids = list(adaptive_ids) if adaptive_ids is not None else [shape.adaptive_id]
    c.n_adaptive = len(ids)
    for i, a in enumerate(ids):
        c.adaptive_ids[i] = a
    return c


class KV:
    """A library-owned KV cache of `batch` sequences and `max_len` slots."""

    def __init__(self, ctx: "Context", batch: int, max_len: int):
        self.ctx = ctx
        h = ctypes.c_void_p()
        _check(_lib().sdsat_kv_create(ctx.handle, batch, max_len, ctypes.byref(h)), "sdsat_kv_create")
        self.handle = h
        self.batch, self.max_len = batch, max_len

    def info(self):
        k, v, ln = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
        b, m = ctypes.c_int(), ctypes.c_int()
        _check(_lib().sdsat_kv_info(self.handle, ctypes.byref(k), ctypes.byref(v), ctypes.byref(ln),
                                    ctypes.byref(b), ctypes.byref(m)), "sdsat_kv_info")
        return k.value, v.value, ln.value, b.value, m.value

    def close(self):
        if getattr(self, "handle", None):
            _lib().sdsat_kv_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class Context:
    """Borrowed weights + TMA descriptors + workspaces for one model shape."""

    def __init__(self, shape, weights: Optional[dict] = None, max_position: int = 8192, adaptive_ids=None,
                 stream=None):
        import torch
        self.shape = shape
        self.cfg = make_config(shape, max_position, adaptive_ids)
        self._keep = weights
        w = None
        if weights is not None:
            L = shape.n_layers
            self._layers = (LayerWeights * L)()
            for l in range(L):
                for n in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
                    setattr(self._layers[l], n, _ptr(weights["layers"][l][n]))
            w = Weights(_ptr(weights["embed"]), _ptr(weights["final_norm"]), _ptr(weights["lm_head"]),
                        ctypes.cast(self._layers, ctypes.POINTER(LayerWeights)))
            self._w = w
        h = ctypes.c_void_p()
        st = stream if stream is not None else torch.cuda.current_stream().cuda_stream
        _check(_lib().sdsat_create(ctypes.byref(self.cfg), ctypes.byref(w) if w is not None else None, st,
                                   ctypes.byref(h)), "sdsat_create")
        self.handle = h

    def _bind_stream(self):
        _lib().sdsat_set_stream(self.handle, _stream())

    def kv(self, batch: int, max_len: int) -> KV:
        return KV(self, batch, max_len)

    def kv_write(self, kv: KV, layer: int, seq: int, slot0: int, k, v):
        """k, v: bf16 CUDA tensors [n_heads, n, head_dim] written to slots slot0 .. slot0+n-1."""
        self._bind_stream()
        _check(_lib().sdsat_kv_write(self.handle, kv.handle, layer, seq, slot0, k.shape[1], _ptr(k), _ptr(v)),
               "sdsat_kv_write")

    def kv_read(self, kv: KV, layer: int, seq: int, slot0: int, n: int):
        import torch
        self._bind_stream()
        H, hd = self.shape.n_heads, self.shape.head_dim
        k = torch.empty(H, n, hd, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        _check(_lib().sdsat_kv_read(self.handle, kv.handle, layer, seq, slot0, n, _ptr(k), _ptr(v)), "sdsat_kv_read")
        return k, v

    # ---- the block decode step ----
    def block_forward(self, kv: KV, tokens, logits, b: int, q: int, positions=None):
        self._bind_stream()
        _check(_lib().sdsat_block_forward(self.handle, kv.handle, _ptr(tokens), _ptr(positions), b, q,
                                          _ptr(logits)), "sdsat_block_forward")

    def accept_greedy(self, kv: KV, logits, drafts, b: int, q: int, n_verify: int, accepted_len, out_tokens,
                      commit: bool = True):
        self._bind_stream()
        _check(_lib().sdsat_accept_greedy(self.handle, kv.handle, _ptr(logits), _ptr(drafts), b, q, n_verify,
                                          _ptr(accepted_len), _ptr(out_tokens), int(commit)), "sdsat_accept_greedy")

    def accept_nucleus(self, kv: KV, logits, drafts, b: int, q: int, n_verify: int, top_p: float,
                       temperature: float, seed: int, accepted_len, out_tokens, top_k: int = 0,
                       commit: bool = True):
        self._bind_stream()
        _check(_lib().sdsat_accept_nucleus(self.handle, kv.handle, _ptr(logits), _ptr(drafts), b, q, n_verify,
                                           top_p, temperature, seed, top_k, _ptr(accepted_len), _ptr(out_tokens),
                                           int(commit)), "sdsat_accept_nucleus")

    def kv_commit(self, kv: KV, new_len, b: int):
        self._bind_stream()
        _check(_lib().sdsat_kv_commit(self.handle, kv.handle, _ptr(new_len), b), "sdsat_kv_commit")

    def kv_lengths(self, kv: KV, b: int = None):
        """The committed lengths as an int32 CUDA tensor [b] (queued on the current stream)."""
        import torch
        b = kv.batch if b is None else b
        out = torch.empty(b, dtype=torch.int32, device="cuda")
        self._bind_stream()
        _check(_lib().sdsat_kv_lengths(self.handle, kv.handle, _ptr(out), b), "sdsat_kv_lengths")
        return out

    def kv_emitted(self, kv: KV, reset: bool = False):
        """Tokens emitted per sequence so far (int64 CUDA tensor [batch])."""
        import torch
        out = torch.empty(kv.batch, dtype=torch.int64, device="cuda")
        self._bind_stream()
        _check(_lib().sdsat_kv_emitted(self.handle, kv.handle, _ptr(out), kv.batch, int(reset)), "sdsat_kv_emitted")
        return out

    def profile_begin(self, max_launches: int):
        _check(_lib().sdsat_profile_begin(self.handle, max_launches), "sdsat_profile_begin")

    def profile_end(self) -> dict:
        """{kernel class: (launches, total_ms)} of the launches since profile_begin."""
        self._bind_stream()
        buf = (KernelStat * 32)()
        n = ctypes.c_int(0)
        _check(_lib().sdsat_profile_end(self.handle, buf, 32, ctypes.byref(n)), "sdsat_profile_end")
        return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].total_ms)) for i in range(n.value)}

    def trace_begin(self, max_records: int):
        _check(_lib().sdsat_trace_begin(self.handle, max_records), "sdsat_trace_begin")

    def trace_end(self, max_records: int):
        """Device timeline records: list of dicts with the kernel class name, launch seq, block,
        smid, flags and the %globaltimer stamps entry / wait / marks (3) / exit."""
        import numpy as np
        buf = np.zeros((max_records, TRACE_WORDS), dtype=np.uint64)
        n = ctypes.c_int(0)
        self._bind_stream()
        _check(_lib().sdsat_trace_end(self.handle, buf.ctypes.data, max_records, ctypes.byref(n)), "sdsat_trace_end")
        out = []
        for r in buf[:n.value]:
            tag, blk = int(r[0]) >> 32, int(r[0]) & 0xFFFFFFFF
            out.append(dict(kernel=_lib().sdsat_kernel_class_name(tag >> 24).decode(), seq=tag & 0xFFFFFF,
                            block=blk, smid=int(r[1]) & 0xFFFFFFFF, flags=int(r[1]) >> 32, entry=int(r[2]),
                            wait=int(r[3]), marks=(int(r[4]), int(r[5]), int(r[6])), exit=int(r[7])))
        return out

    def build_block(self, kv: KV, mode: int, prev_out, prev_acc, tokens_out, b: int, q: int,
                    draft_table=None, table_stride: int = 0):
        self._bind_stream()
        _check(_lib().sdsat_build_block(self.handle, kv.handle, mode, _ptr(prev_out), _ptr(prev_acc),
                                        _ptr(draft_table), table_stride, b, q, _ptr(tokens_out)),
               "sdsat_build_block")

    # ---- tree-structured draft step 2 (Sec. 2.1.2) ----
    def block_forward_tree(self, kv: KV, tokens, parent, logits, b: int, q: int):
        self._bind_stream()
        _check(_lib().sdsat_block_forward_tree(self.handle, kv.handle, _ptr(tokens), _ptr(parent), b, q,
                                               _ptr(logits)), "sdsat_block_forward_tree")

    def accept_tree(self, kv: KV, logits, tokens, parent, b: int, q: int, accepted_len, out_tokens, path=None,
                    temperature: float = 0.0, top_p: float = 1.0, seed: int = 0, top_k: int = 0,
                    commit: bool = True):
        self._bind_stream()
        _check(_lib().sdsat_accept_tree(self.handle, kv.handle, _ptr(logits), _ptr(tokens), _ptr(parent), b, q,
                                        temperature, top_p, seed, top_k, _ptr(accepted_len), _ptr(out_tokens),
                                        _ptr(path), int(commit)), "sdsat_accept_tree")

    def build_tree_block(self, kv: KV, mode: int, prev_out, prev_q: int, prev_acc, tokens_out, b: int, k: int,
                         draft_tables=None, width: int = 1, table_stride: int = 0):
        self._bind_stream()
        _check(_lib().sdsat_build_tree_block(self.handle, kv.handle, mode, _ptr(prev_out), prev_q, _ptr(prev_acc),
                                             _ptr(draft_tables), width, table_stride, b, k, _ptr(tokens_out)),
               "sdsat_build_tree_block")

    # ---- pipelined variant ----
    def build_pipelined_block(self, kv: KV, prev_out, prev_acc, mode, n_verify, tokens_out, b: int, k: int,
                              draft_table=None, table_stride: int = 0):
        self._bind_stream()
        _check(_lib().sdsat_build_pipelined_block(self.handle, kv.handle, _ptr(prev_out), _ptr(prev_acc), _ptr(mode),
                                                  _ptr(n_verify), _ptr(draft_table), table_stride, b, k,
                                                  _ptr(tokens_out)), "sdsat_build_pipelined_block")

    def accept_pipelined(self, kv: KV, logits, tokens, n_verify, b: int, q: int, accepted_len, out_tokens,
                         temperature: float = 0.0, top_p: float = 1.0, seed: int = 0, top_k: int = 0,
                         commit: bool = True):
        self._bind_stream()
        _check(_lib().sdsat_accept_pipelined(self.handle, kv.handle, _ptr(logits), _ptr(tokens), _ptr(n_verify), b, q,
                                             temperature, top_p, seed, top_k, _ptr(accepted_len), _ptr(out_tokens),
                                             int(commit)), "sdsat_accept_pipelined")

    def prefill(self, kv: KV, seq: int, tokens):
        self._bind_stream()
        _check(_lib().sdsat_prefill(self.handle, kv.handle, seq, _ptr(tokens), tokens.numel()), "sdsat_prefill")

    def get_error(self) -> int:
        """Synchronise; return and clear the device error bits."""
        self._bind_stream()
        f = ctypes.c_uint32(0)
        st = _lib().sdsat_get_error(self.handle, ctypes.byref(f))
        if st not in (0, 5):
            raise SdsatError(st, "sdsat_get_error")
        return f.value

    # ---- single kernels ----
    def op_gemm(self, x, w, y):
        self._bind_stream()
        M, K = x.shape
        N = w.shape[0]
        _check(_lib().sdsat_op_gemm(self.handle, _ptr(x), M, K, _ptr(w), N, _ptr(y)), "sdsat_op_gemm")

    def op_attention(self, q, k, v, lens, b: int, qn: int, H: int, hd: int, cap: int, out):
        self._bind_stream()
        _check(_lib().sdsat_op_attention(self.handle, _ptr(q), _ptr(k), _ptr(v), _ptr(lens), b, qn, H, hd, cap,
                                         _ptr(out)), "sdsat_op_attention")

    def debug_workspace(self, which: int, rows: int):
        """Last-layer workspace of the last forward: 0 h, 1 q, 2 attention out, 3 SwiGLU act."""
        import torch
        s = self.shape
        cols = [s.d_model, s.n_heads * s.head_dim, s.n_heads * s.head_dim, s.ffn_dim][which]
        out = torch.empty(rows, cols, device="cuda")
        self._bind_stream()
        _check(_lib().sdsat_debug_workspace(self.handle, which, rows, _ptr(out)), "sdsat_debug_workspace")
        return out

    def debug_wait_timeout(self):
        """Queue a kernel whose bounded wait runs out (device bit TIMEOUT after ~2 s)."""
        self._bind_stream()
        _check(_lib().sdsat_debug_wait_timeout(self.handle), "sdsat_debug_wait_timeout")

    def op_exp(self, x, y):
        self._bind_stream()
        _check(_lib().sdsat_op_exp(self.handle, _ptr(x), _ptr(y), x.numel()), "sdsat_op_exp")

    def close(self):
        if getattr(self, "handle", None):
            _lib().sdsat_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
