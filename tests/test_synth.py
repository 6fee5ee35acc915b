"""The seeded input generator: deterministic, row-addressable, right moments."""
import torch

import synth


def test_normal_moments_and_determinism():
    a = synth.normal_bf16(0, 123, (512, 1024), 0.02)
    b = synth.normal_bf16(0, 123, (512, 1024), 0.02)
    assert torch.equal(a, b)
    x = a.float()
    assert abs(x.mean().item()) < 2e-4
    assert abs(x.std().item() - 0.02) < 2e-4
    assert x.abs().max().item() <= 0.02 * 3.47
    c = synth.normal_bf16(1, 123, (512, 1024), 0.02)
    assert not torch.equal(a, c)


def test_row_subsets_match_full():
    full = synth.normal_bf16(5, 7, (300, 96), 0.02)
    rows = torch.tensor([0, 17, 299, 3])
    assert torch.equal(synth.normal_bf16(5, 7, (300, 96), 0.02, rows=rows), full[rows])


def test_hash_known_values():
    """fmix32 of MurmurHash3 maps 0 to 0 and is a bijection on small samples."""
    assert synth._fmix32_int(0) == 0
    xs = torch.arange(1 << 16, dtype=torch.int64)
    h = synth._fmix32(xs)
    assert torch.unique(h).numel() == xs.numel()
    assert all(int(h[i]) == synth._fmix32_int(i) for i in (1, 2, 1000, 65535))


def test_ids_and_stub():
    ids = synth.uniform_ids(0, 9, 10000, 4104)
    assert ids.min() >= 0 and ids.max() < 4104
    ref = torch.arange(1000, dtype=torch.int32)
    t = synth.stub_table(0, 0, ref, 0.7, 4104)
    rate = (t == ref).float().mean().item()
    assert 0.65 < rate < 0.75
    assert torch.equal(t, synth.stub_table(0, 0, ref, 0.7, 4104))
