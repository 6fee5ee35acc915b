"""Failure detection on the GPU without a GPU fault: every failure here is made on the host
(bad arguments, an oversized request, out-of-range ids) or is a bounded wait that nothing
completes; the library reports it through its status codes and device error bits, and the
context keeps working afterwards."""
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

DEV_TIMEOUT, DEV_CAPACITY, DEV_TOKEN, DEV_POSITION = 0x2, 0x4, 0x8, 0x10


@pytest.fixture(scope="module")
def sd():
    import paper_2403_18647_gb300 as sd
    return sd


@pytest.fixture(scope="module")
def tiny(sd):
    shape = synth.SHAPES["tiny"]
    w = synth.make_model(shape, seed=0, device="cuda")
    return shape, sd.Context(shape, w, max_position=256)


def _i32(x):
    return torch.tensor(list(x), dtype=torch.int32, device="cuda")


def _healthy(shape, ctx):
    """A block forward and greedy accept run and report no device error."""
    kv = ctx.kv(1, 64)
    ctx.prefill(kv, 0, synth.prompt_ids(0, 90, 20, 4096).cuda())
    lg = torch.empty(6, shape.vocab, device="cuda")
    toks = _i32([1, 2, 3, 4, 5, 6])
    ctx.block_forward(kv, toks, lg, 1, 6)
    acc = torch.empty(1, dtype=torch.int32, device="cuda")
    out = torch.empty(6, dtype=torch.int32, device="cuda")
    ctx.accept_greedy(kv, lg, toks, 1, 6, 5, acc, out)
    assert ctx.get_error() == 0
    assert torch.isfinite(lg).all()


def test_bounded_wait_runs_out_and_the_context_survives(sd, tiny):
    shape, ctx = tiny
    ctx.debug_wait_timeout()
    assert ctx.get_error() == DEV_TIMEOUT
    assert ctx.get_error() == 0            # read and cleared
    _healthy(shape, ctx)


def test_block_past_capacity_is_not_written(sd, tiny):
    shape, ctx = tiny
    kv = ctx.kv(1, 24)
    ctx.prefill(kv, 0, synth.prompt_ids(0, 91, 20, 4096).cuda())
    k_before, v_before = ctx.kv_read(kv, 0, 0, 0, 24)
    lg = torch.empty(6, shape.vocab, device="cuda")
    ctx.block_forward(kv, _i32([1, 2, 3, 4, 5, 6]), lg, 1, 6)   # slots 20..25, capacity 24
    assert ctx.get_error() & DEV_CAPACITY
    k_after, _ = ctx.kv_read(kv, 0, 0, 0, 20)
    assert torch.equal(k_after, k_before[:, :20])               # committed slots untouched
    acc = torch.empty(1, dtype=torch.int32, device="cuda")
    out = torch.empty(6, dtype=torch.int32, device="cuda")
    drafts = _i32([0] * 6)
    ctx.accept_greedy(kv, lg, drafts, 1, 6, 0, acc, out)            # commit 1: 21 <= 24
    assert ctx.get_error() == 0
    ctx.kv_commit(kv, _i32([30]), 1)                                # past capacity: clamped, reported
    assert ctx.get_error() & DEV_CAPACITY
    assert ctx.kv_lengths(kv).item() == 24
    _healthy(shape, ctx)


def test_token_and_position_out_of_range(sd, tiny):
    shape, ctx = tiny
    kv = ctx.kv(1, 64)
    lg = torch.empty(2, shape.vocab, device="cuda")
    ctx.block_forward(kv, _i32([shape.vocab + 5, -3]), lg, 1, 2)   # ids outside [0, vocab): read as 0
    assert ctx.get_error() & DEV_TOKEN
    lg1 = torch.empty(1, shape.vocab, device="cuda")
    ctx.block_forward(kv, _i32([7]), lg1, 1, 1, positions=_i32([10_000]))   # past max_position: clamped
    assert ctx.get_error() & DEV_POSITION
    _healthy(shape, ctx)


def test_oversized_requests_fail_on_the_host(sd, tiny):
    shape, ctx = tiny
    with pytest.raises(sd.SdsatError):
        ctx.kv(1, 100_000)                     # max_len past max_position (256): ECAPACITY
    big = synth.SHAPES["7b"]
    bctx = sd.Context(big, None, max_position=32768)
    with pytest.raises(sd.SdsatError):
        bctx.kv(4096, 32768)                   # ~68 TB of cache: the allocation fails (ENOMEM)
    lg = torch.empty(17, shape.vocab, device="cuda")
    kv = ctx.kv(1, 64)
    with pytest.raises(sd.SdsatError):
        ctx.block_forward(kv, _i32(range(17)), lg, 1, 17)      # q > 16: EINVAL
    _healthy(shape, ctx)
