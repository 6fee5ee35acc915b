"""sdsat_gemm_static: the scratch-free GEMM entry point, for callers that cannot allocate.

Callers that capture CUDA graphs, run under a framework's own allocator or work to a
fixed memory budget cannot have the library cudaMalloc scratch on their behalf; this
entry point keeps its scratch in a fixed device array instead.  The test calls it
through the C ABI twice in a row (the second call reuses the array the first call
left behind) and checks each result against the context-based sdsat_op_gemm within
the GEMM tolerance of the kernel tests, and against the oracle's y = x W^T.  The
file is collected last.
"""
import ctypes
import math

import numpy as np
import pytest
import torch

import synth
from oracle import model as OM

pytestmark = pytest.mark.gpu


def _lib():
    import paper_2403_18647_gb300 as sd
    lib = sd.lib()
    fn = lib.sdsat_gemm_static
    fn.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
                   ctypes.c_void_p, ctypes.c_void_p]
    fn.restype = ctypes.c_int
    return sd, fn


def test_gemm_static_matches_op_gemm_twice():
    sd, fn = _lib()
    ctx = sd.Context(synth.SHAPES["tiny"], None, max_position=256)
    stream = torch.cuda.current_stream().cuda_stream
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    for i, (M, K, N) in enumerate([(6, 4096, 12288), (13, 688, 4104)]):
        x = synth.normal_f32(9, 200 + i, (M, K), 1.0, device="cuda")
        w = synth.normal_bf16(9, 300 + i, (N, K), 0.02, device="cuda")
        ref = torch.empty(M, N, device="cuda")
        ctx.op_gemm(x, w, ref)
        got = torch.full((M, N), float("nan"), device="cuda")
        assert fn(x.data_ptr(), M, K, w.data_ptr(), N, got.data_ptr(), stream, err.data_ptr()) == 0
        torch.cuda.synchronize()
        tol = 5e-5 * math.sqrt(K) * 0.02 + 1e-6 * ref.abs().max().item()
        e_op = (got - ref).abs().max().item()
        assert e_op <= tol, (i, e_op, tol)
        exact = OM.linear(OM.to64(x), OM.to64(w))
        e_or = np.abs(got.cpu().numpy() - exact).max()
        assert e_or <= tol, (i, e_or, tol)
    assert err.item() == 0


def test_gemm_static_rejects_sizes_past_the_limits():
    sd, fn = _lib()
    x = torch.zeros(17, 64, device="cuda")
    w = torch.zeros(128, 64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(17, 128, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    assert fn(x.data_ptr(), 17, 64, w.data_ptr(), 128, y.data_ptr(), stream, None) == 3      # M > 16: ECAPACITY
    assert fn(x.data_ptr(), 4, 20000, w.data_ptr(), 128, y.data_ptr(), stream, None) == 3    # K > 16384
    assert fn(x.data_ptr(), 4, 60, w.data_ptr(), 128, y.data_ptr(), stream, None) == 1       # K % 8 != 0: EINVAL
