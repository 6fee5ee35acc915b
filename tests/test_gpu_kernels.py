"""Single-kernel parity: each CUDA kernel (through the C ABI) against the oracle on seeded inputs.

Tolerances are derived from the arithmetic:
  * GEMM: X is split into bf16 hi + lo parts (|x - hi - lo| <= 2^-16 |x|), products
    accumulate in fp32, so |err| <~ 2^-16 sum|w x| + K 2^-24 max|y|: we allow
    5e-5 * sqrt(K) * std(w) * rms(x) + 1e-6 max|y|.
  * attention: fp32 scores and softmax over bf16 K/V that both sides read exactly;
    allow 2e-5 absolute on outputs of O(1).
  * exp and the acceptance kernel: bit-exact (their arithmetic is defined exactly).
"""
import math

import numpy as np
import pytest
import torch

import synth
from oracle import model as OM
from oracle import sampling as OS
from oracle import decode as OD

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sd():
    import paper_2403_18647_gb300 as sd
    return sd


@pytest.fixture(scope="module")
def tiny_ctx(sd):
    return sd.Context(synth.SHAPES["tiny"], None, max_position=4096)


@pytest.fixture(scope="module")
def big_ctx(sd):
    # weights-free context with 7B-shaped attention workspaces (kernel entry points only)
    return sd.Context(synth.SHAPES["7b"], None, max_position=16384 + 64)


# ---------------------------------------------------------------- exp
def test_exp_bit_exact(tiny_ctx):
    """The sampler's exp: GPU bits == oracle bits on 2^22 arguments across [-90, 0] and edges."""
    x = -torch.rand(1 << 22, generator=torch.Generator().manual_seed(0), dtype=torch.float64) * 90.0
    x = torch.cat([x.float(), torch.tensor([0.0, -0.0, -87.0, -86.99999, -87.00001, -1e-30, -float("inf"),
                                            float("nan"), -0.34657359, -0.34657362])])
    y = torch.empty_like(x, device="cuda")
    tiny_ctx.op_exp(x.cuda(), y)
    got = y.cpu().numpy().view(np.uint32)
    ref = OS.exp_sd(x.numpy()).view(np.uint32)
    bad = np.nonzero(got != ref)[0]
    assert bad.size == 0, (x[bad[:5]], got[bad[:5]], ref[bad[:5]])


# ---------------------------------------------------------------- GEMM
GEMM_CASES = [
    # (M, K, N): tiles, ragged N tail, ragged K tail (688 = 10.75 chunks), split-K sharing
    (1, 256, 256), (6, 256, 768), (6, 688, 256), (16, 256, 4104), (17, 512, 300), (24, 256, 1376),
    (33, 128, 130), (64, 256, 512), (6, 4096, 384), (2, 11008, 256),
    # the tiled prefill GEMM: partial position blocks, ragged N and K, several waves of tiles
    (65, 256, 256), (128, 688, 300), (200, 1024, 1000), (512, 4096, 384), (300, 512, 5000),
]


@pytest.mark.parametrize("M,K,N", GEMM_CASES)
def test_gemm_parity(tiny_ctx, M, K, N):
    x = synth.normal_f32(1, 10 + M, (M, K), 1.0, device="cuda")
    w = synth.normal_bf16(1, 20 + N, (N, K), 0.02, device="cuda")
    y = torch.full((M, N), float("nan"), device="cuda")
    tiny_ctx.op_gemm(x, w, y)
    torch.cuda.synchronize()
    ref = OM.linear(x.cpu().double().numpy(), w.cpu().double().numpy())
    tol = 5e-5 * math.sqrt(K) * 0.02 + 1e-6 * np.abs(ref).max()
    err = np.abs(y.cpu().double().numpy() - ref).max()
    assert err <= tol, (err, tol)


@pytest.mark.parametrize("N,K", [(12288, 4096), (22016, 4096), (4096, 11008), (32016, 4096)])
@pytest.mark.parametrize("M", [6, 16])
def test_gemm_full_size_sampled(tiny_ctx, M, N, K):
    """The kernel-sweep shapes of the 7B model at full size; the oracle checks 512 sampled
    output columns (row-wise fp64 dot products)."""
    x = synth.normal_f32(2, M, (M, K), 1.0, device="cuda")
    w = synth.normal_bf16(2, N + K, (N, K), 0.02, device="cuda")
    y = torch.empty((M, N), device="cuda")
    tiny_ctx.op_gemm(x, w, y)
    torch.cuda.synchronize()
    cols = torch.cat([torch.arange(0, 128), torch.randint(0, N, (256,), generator=torch.Generator().manual_seed(N)),
                      torch.arange(N - 128, N)])
    ref = OM.linear(x.cpu().double().numpy(), w[cols.cuda()].cpu().double().numpy())
    err = np.abs(y[:, cols.cuda()].cpu().double().numpy() - ref).max()
    assert err <= 5e-5 * math.sqrt(K) * 0.02 + 1e-6 * np.abs(ref).max(), err


def test_gemm_deterministic(tiny_ctx):
    x = synth.normal_f32(3, 1, (6, 4096), 1.0, device="cuda")
    w = synth.normal_bf16(3, 2, (4096, 4096), 0.02, device="cuda")
    a = torch.empty((6, 4096), device="cuda")
    b = torch.empty_like(a)
    tiny_ctx.op_gemm(x, w, a)
    tiny_ctx.op_gemm(x, w, b)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


# ---------------------------------------------------------------- attention
ATT_CASES = [
    # (b, q, H, hd, lens, cap)
    (1, 1, 4, 64, [0], 64), (1, 6, 4, 64, [5], 64), (1, 6, 4, 64, [122], 256), (1, 6, 4, 64, [123], 256),
    (1, 16, 2, 128, [300], 512), (3, 6, 4, 128, [0, 127, 250], 300), (2, 11, 4, 64, [129, 1000], 1100),
    (4, 6, 32, 128, [1024, 1100, 1200, 1270], 1290),
    # more (sequence, head) pairs than fit as clusters: single CTAs, some taking two pairs
    # (q <= 8: 512 pairs; q = 9: 448 pairs), or one pair each (256 pairs)
    (16, 4, 32, 128, [0, 1, 63, 64, 65, 100, 127, 128, 200, 257, 300, 383, 450, 511, 600, 630], 640),
    (7, 9, 64, 64, [0, 5, 64, 130, 200, 255, 310], 320),
    (8, 8, 32, 128, [700, 10, 333, 64, 512, 1, 600, 129], 710),
]


def _att_ref(qm, K, V, lens, b, q, H, hd):
    out = np.empty((b * q, H * hd))
    for s in range(b):
        qs = qm[s * q:(s + 1) * q].reshape(q, H, hd)
        o = OM.attend(qs, K[s], V[s], [lens[s] + j + 1 for j in range(q)])
        out[s * q:(s + 1) * q] = o.reshape(q, H * hd)
    return out


@pytest.mark.parametrize("b,q,H,hd,lens,cap", ATT_CASES)
def test_attention_parity(big_ctx, b, q, H, hd, lens, cap):
    K = synth.normal_bf16(4, 1, (b * H * cap, hd), 1.0, device="cuda").reshape(b, H, cap, hd)
    V = synth.normal_bf16(4, 2, (b * H * cap, hd), 1.0, device="cuda").reshape(b, H, cap, hd)
    qm = synth.normal_f32(4, 3, (b * q, H * hd), 1.0, device="cuda")
    ln = torch.tensor(lens, dtype=torch.int32, device="cuda")
    out = torch.full((b * q, H * hd), float("nan"), device="cuda")
    big_ctx.op_attention(qm, K, V, ln, b, q, H, hd, cap, out)
    torch.cuda.synchronize()
    ref = _att_ref(qm.cpu().double().numpy(), K.cpu().double().numpy(), V.cpu().double().numpy(), lens, b, q, H, hd)
    err = np.abs(out.cpu().double().numpy() - ref).max()
    assert err <= 2e-5, err


@pytest.mark.parametrize("ctxlen", [2048, 16384])
def test_attention_full_size_sampled(big_ctx, ctxlen):
    """7B shape (32 heads x 128) at full context; the oracle checks 3 sampled heads."""
    b, q, H, hd = 1, 6, 32, 128
    cap = ctxlen + q
    K = synth.normal_bf16(5, 1, (H * cap, hd), 1.0, device="cuda").reshape(1, H, cap, hd)
    V = synth.normal_bf16(5, 2, (H * cap, hd), 1.0, device="cuda").reshape(1, H, cap, hd)
    qm = synth.normal_f32(5, 3, (q, H * hd), 1.0, device="cuda")
    ln = torch.tensor([ctxlen], dtype=torch.int32, device="cuda")
    out = torch.empty((q, H * hd), device="cuda")
    big_ctx.op_attention(qm, K, V, ln, b, q, H, hd, cap, out)
    torch.cuda.synchronize()
    for h in (0, 17, 31):
        qs = qm.cpu().double().numpy().reshape(q, H, hd)[:, h:h + 1]
        o = OM.attend(qs, K[0, h:h + 1].cpu().double().numpy(), V[0, h:h + 1].cpu().double().numpy(),
                      [ctxlen + j + 1 for j in range(q)])
        err = np.abs(out.cpu().double().numpy().reshape(q, H, hd)[:, h] - o[:, 0]).max()
        assert err <= 2e-5, (h, err)


# ---------------------------------------------------------------- acceptance
def _logits(seed, rows, V, device="cuda", std=1.3):
    return synth.normal_f32(seed, 77, (rows, V), std, device=device)


@pytest.fixture(scope="module")
def accept_env(sd):
    shape = synth.SHAPES["tiny"]
    w = synth.make_model(shape, seed=0, device="cuda")
    ctx = sd.Context(shape, w, max_position=4096)
    return ctx


def _run_accept(ctx, logits, drafts, b, q, n_verify, lens, temperature=0.0, top_p=1.0, seed=0, top_k=0):
    kv = ctx.kv(b, 4000)
    ln = torch.tensor(lens, dtype=torch.int32, device="cuda")
    ctx.kv_commit(kv, ln, b)
    acc = torch.empty(b, dtype=torch.int32, device="cuda")
    out = torch.empty(b * q, dtype=torch.int32, device="cuda")
    if temperature > 0:
        ctx.accept_nucleus(kv, logits, drafts, b, q, n_verify, top_p, temperature, seed, acc, out, top_k=top_k)
    else:
        ctx.accept_greedy(kv, logits, drafts, b, q, n_verify, acc, out)
    flags = ctx.get_error()
    return acc.cpu().tolist(), out.cpu().view(b, q).tolist(), flags, ctx.kv_lengths(kv).cpu().tolist()


def _oracle_accept(lg, drafts, b, q, n_verify, lens, temperature=0.0, top_p=1.0, seed=0, top_k=0):
    accs, outs = [], []
    for s in range(b):
        t = [OS.select(lg[s * q + j], temperature, top_p, seed, lens[s] + j + 1, s, top_k)[0] for j in range(q)]
        m = OD.verify(t, drafts[s * q:(s + 1) * q], n_verify)
        accs.append(1 + m)
        outs.append(t)
    return accs, outs


@pytest.mark.parametrize("b,q,n_verify", [(1, 6, 0), (1, 6, 5), (4, 6, 5), (2, 16, 15), (3, 1, 0)])
def test_accept_greedy_bit_exact(accept_env, b, q, n_verify):
    V = accept_env.shape.vocab
    lg = _logits(b * 100 + q, b * q, V)
    lg[0, 17] = lg[0].max() + 1.0
    lg[0, 3] = lg[0, 17]                                   # a tie: lowest id wins
    lgc = lg.cpu().numpy()
    # drafts: copy the oracle's targets for a prefix, then break
    _, tg = _oracle_accept(lgc, [0] * (b * q), b, q, 0, [10] * b)
    drafts = []
    for s in range(b):
        row = [0] + [tg[s][j - 1] if j <= 2 + s else (tg[s][j - 1] + 1) % V for j in range(1, q)]
        drafts += row
    dr = torch.tensor(drafts, dtype=torch.int32, device="cuda")
    lens = [10 + s for s in range(b)]
    acc, out, flags, newlen = _run_accept(accept_env, lg, dr, b, q, n_verify, lens)
    racc, rout = _oracle_accept(lgc, drafts, b, q, n_verify, lens)
    assert out == rout and acc == racc and flags == 0
    assert newlen == [lens[s] + racc[s] for s in range(b)]          # commit: len += 1 + m


def test_accept_nan_rows(accept_env):
    V = accept_env.shape.vocab
    lg = _logits(9, 6, V)
    lg[1, 5] = float("nan")
    lg[2, :] = float("nan")
    dr = torch.zeros(6, dtype=torch.int32, device="cuda")
    acc, out, flags, _ = _run_accept(accept_env, lg, dr, 1, 6, 0, [0])
    _, rout = _oracle_accept(lg.cpu().numpy(), [0] * 6, 1, 6, 0, [0])
    assert out[0] == rout[0] and flags & 0x1


@pytest.mark.parametrize("T,top_p,top_k", [(0.2, 0.95, 0), (1.0, 0.95, 0), (1.0, 0.95, 10), (0.7, 0.5, 0),
                                           (1.0, 1.0, 0), (2.0, 0.0, 0), (0.2, 0.95, 1)])
def test_accept_nucleus_bit_exact(accept_env, T, top_p, top_k):
    """The acceptance kernel is bit-exact on identical logits (the required tolerance for it)."""
    V = accept_env.shape.vocab
    b, q = 2, 6
    for trial in range(3):
        lg = _logits(1000 + trial, b * q, V, std=1.3 + trial)
        if trial == 2:
            lg[:, 100:110] = lg[:, 100:101]               # tied weights
        lgc = lg.cpu().numpy()
        _, tg = _oracle_accept(lgc, [0] * (b * q), b, q, 0, [50, 60], T, top_p, 7, top_k)
        drafts = []
        for s in range(b):
            drafts += [0] + [tg[s][j - 1] if j < 4 else 0 for j in range(1, q)]
        dr = torch.tensor(drafts, dtype=torch.int32, device="cuda")
        acc, out, flags, _ = _run_accept(accept_env, lg, dr, b, q, q - 1, [50, 60], T, top_p, 7, top_k)
        racc, rout = _oracle_accept(lgc, drafts, b, q, q - 1, [50, 60], T, top_p, 7, top_k)
        assert out == rout, (trial, out, rout)
        assert acc == racc


def test_accept_nucleus_full_vocab(sd):
    """32016-entry vocabulary (the 7B/13B LM head): bit-exact vs the oracle."""
    big = synth.ModelShape("v32k", 1, 256, 4, 64, 688, 32016, 32011)
    w = synth.make_model(big, seed=0, device="cuda")
    ctx = sd.Context(big, w, max_position=4096)
    b, q = 4, 6
    lg = _logits(4242, b * q, 32016)
    lgc = lg.cpu().numpy()
    for T, p, k in [(0.2, 0.95, 0), (1.0, 0.95, 10)]:
        lens = [1024, 1030, 1100, 1200]
        _, tg = _oracle_accept(lgc, [0] * (b * q), b, q, 0, lens, T, p, 11, k)
        drafts = []
        for s in range(b):
            drafts += [0] + [tg[s][j - 1] for j in range(1, q)]
        dr = torch.tensor(drafts, dtype=torch.int32, device="cuda")
        acc, out, flags, _ = _run_accept(ctx, lg, dr, b, q, q - 1, lens, T, p, 11, k)
        racc, rout = _oracle_accept(lgc, drafts, b, q, q - 1, lens, T, p, 11, k)
        assert out == rout and acc == racc


def _sorted_list_rows(V, sizes, seed):
    """Rows whose heavy set has exactly n ids (the rest at -100, weight 0): tied logit values
    for even rows, a narrow continuum for odd ones, so that kept sets of more than 32 take
    the sampler's sorted-list path at list sizes that are not powers of two."""
    g = torch.Generator().manual_seed(seed)
    rows = []
    for i, n in enumerate(sizes):
        r = torch.full((V,), -100.0)
        ids = torch.randperm(V, generator=g)[:n]
        if i % 2 == 0:
            vals = torch.tensor([0.0, -0.05, -0.1, -0.2])[torch.randint(0, 4, (n,), generator=g)]
        else:
            vals = torch.randn(n, generator=g) * 0.5
        r[ids] = vals
        rows.append(r)
    return torch.stack(rows).float()


@pytest.mark.parametrize("T,top_p,top_k", [(1.0, 0.95, 0), (0.2, 0.95, 0), (1.0, 0.9, 100), (1.0, 0.999, 0)])
def test_accept_nucleus_sorted_list_sizes(sd, T, top_p, top_k):
    """The sorted-list path (kept sets beyond 32, lists of 65-4096) on a 32016-entry vocabulary:
    bit-exact against the oracle, ties in W included."""
    big = synth.ModelShape("v32k", 1, 256, 4, 64, 688, 32016, 32011)
    w = synth.make_model(big, seed=0, device="cuda")
    ctx = sd.Context(big, w, max_position=4096)
    sizes = [65, 100, 257, 690, 1000, 1023, 1025, 2049, 3000, 4000, 4096, 130, 513, 777]
    b, q = 2, 7
    lg = _sorted_list_rows(32016, sizes, 31 + int(T * 10) + top_k)
    lgc = lg.numpy()
    lens = [300, 2000]
    acc, out, flags, _ = _run_accept(ctx, lg.cuda(), torch.zeros(b * q, dtype=torch.int32, device="cuda"), b, q, 0,
                                     lens, T, top_p, 5, top_k)
    _, rout = _oracle_accept(lgc, [0] * (b * q), b, q, 0, lens, T, top_p, 5, top_k)
    assert out == rout
    assert flags == 0


def _nucleus_rows(V):
    """Rows that steer the sampler's list path (heavy weights compacted, at each floor) and its
    block-wide path (too many heavy weights), at the boundaries between them."""
    rows = []
    flat = torch.zeros(V)                                            # every weight 2^24: block-wide path
    rows.append(flat)
    peaked = torch.full((V,), -100.0)                                # three non-zero weights
    peaked[[7, 300, 301]] = torch.tensor([0.0, -0.5, -0.5])
    rows.append(peaked)
    for n in (4096, 4097):                                           # list capacity, and one past it
        r = torch.full((V,), -100.0)
        r[torch.arange(n) * (V // n)] = 0.0
        rows.append(r)
    mid = torch.full((V,), -100.0)                                   # mass above 2^-8 of the max < 0.95
    mid[5] = 0.0
    mid[1000:1200] = -8.0
    rows.append(mid)
    g = torch.Generator().manual_seed(5)
    rows.append(torch.randn(V, generator=g) * 0.3)                   # nearly flat
    rows.append(torch.randn(V, generator=g) * 6.0)                   # peaked at T = 1
    return torch.stack(rows).float()


@pytest.mark.parametrize("T,top_p,top_k", [(1.0, 0.95, 0), (1.0, 0.95, 10), (0.2, 1.0, 0), (1.0, 0.5, 3),
                                           (0.2, 0.95, 10), (1.0, 0.999, 0)])
def test_accept_nucleus_list_and_block_paths(accept_env, T, top_p, top_k):
    """Bit-exact against the oracle on rows built to take each of the sampler's paths."""
    V = accept_env.shape.vocab
    lg = _nucleus_rows(V)
    n = lg.shape[0]
    lgc = lg.numpy()
    drafts = [0] * n
    acc, out, flags, _ = _run_accept(accept_env, lg.cuda(), torch.zeros(n, dtype=torch.int32, device="cuda"), 1, n,
                                     0, [40], T, top_p, 3, top_k)
    _, rout = _oracle_accept(lgc, drafts, 1, n, 0, [40], T, top_p, 3, top_k)
    assert out == rout
    assert flags == 0


@pytest.mark.parametrize("N,K", [(15360, 5120), (27648, 5120), (5120, 13824), (32016, 5120)])
def test_gemm_13b_shapes_sampled(tiny_ctx, N, K):
    """The 13B model's projection shapes (QKV, gate+up, down, LM head) at M = 6; 384 sampled
    output columns against fp64 dot products."""
    M = 6
    x = synth.normal_f32(4, M, (M, K), 1.0, device="cuda")
    w = synth.normal_bf16(4, N + K, (N, K), 0.02, device="cuda")
    y = torch.empty((M, N), device="cuda")
    tiny_ctx.op_gemm(x, w, y)
    torch.cuda.synchronize()
    cols = torch.cat([torch.arange(0, 128), torch.randint(0, N, (128,), generator=torch.Generator().manual_seed(N)),
                      torch.arange(N - 128, N)])
    ref = OM.linear(x.cpu().double().numpy(), w[cols.cuda()].cpu().double().numpy())
    err = np.abs(y[:, cols.cuda()].cpu().double().numpy() - ref).max()
    assert err <= 5e-5 * math.sqrt(K) * 0.02 + 1e-6 * np.abs(ref).max(), err


@pytest.mark.parametrize("M", [6, 24])
@pytest.mark.parametrize("K,N", [(2048, 49152), (3072, 24576), (4096, 16384)])
def test_gemm_streamk_snapped_full(tiny_ctx, M, K, N):
    """Shapes whose stream-K split gives every CTA >= 24 units (304 CTAs on GB300), so split
    points that land in a tile's first 3 units move to the tile's start (16-32 of them here),
    at the two operand widths (M = 6: MPAD 16; M = 24: MPAD 32): every output element against
    fp64 dot products, so every tile's contributor set and partial slots are exercised."""
    x = synth.normal_f32(6, M * 7 + K, (M, K), 1.0, device="cuda")
    w = synth.normal_bf16(6, N + K, (N, K), 0.02, device="cuda")
    y = torch.empty((M, N), device="cuda")
    tiny_ctx.op_gemm(x, w, y)
    torch.cuda.synchronize()
    ref = OM.linear(x.cpu().double().numpy(), w.cpu().double().numpy())
    err = np.abs(y.cpu().double().numpy() - ref).max()
    assert err <= 5e-5 * math.sqrt(K) * 0.02 + 1e-6 * np.abs(ref).max(), err
    assert tiny_ctx.get_error() == 0


def test_attention_40_heads_sampled(big_ctx):
    """40 heads (the 13B shape) at context 4096, q = 6: three sampled heads against the oracle."""
    b, q, H, hd, n = 1, 6, 40, 128, 4096
    cap = n + q
    K = synth.normal_bf16(6, 1, (H * cap, hd), 1.0, device="cuda").reshape(1, H, cap, hd)
    V = synth.normal_bf16(6, 2, (H * cap, hd), 1.0, device="cuda").reshape(1, H, cap, hd)
    qm = synth.normal_f32(6, 3, (q, H * hd), 1.0, device="cuda")
    ln = torch.tensor([n], dtype=torch.int32, device="cuda")
    out = torch.empty((q, H * hd), device="cuda")
    big_ctx.op_attention(qm, K, V, ln, b, q, H, hd, cap, out)
    torch.cuda.synchronize()
    for h in (0, 21, 39):
        qs = qm.cpu().double().numpy().reshape(q, H, hd)[:, h:h + 1]
        o = OM.attend(qs, K[0, h:h + 1].cpu().double().numpy(), V[0, h:h + 1].cpu().double().numpy(),
                      [n + j + 1 for j in range(q)])
        err = np.abs(out.cpu().double().numpy().reshape(q, H, hd)[:, h] - o[:, 0]).max()
        assert err <= 2e-5, (h, err)
