"""The seeded input generator (host build): conversions, statistics, determinism (CPU only)."""
import numpy as np
import pytest
import torch

import synth


@pytest.mark.parametrize("sigma", [1.0, 80 ** -0.5])
def test_value_rounding_matches_library_conversions(sigma):
    scale = synth.scale_for(sigma)
    c = np.arange(-131070, 131071, dtype=np.int64)
    x32 = c.astype(np.float32) * scale  # one binary32 rounding, as the generator defines
    ours16 = synth.f32_to_f16_bits(x32)
    assert np.array_equal(ours16, x32.astype(np.float16).view(np.uint16))
    oursb = synth.f32_to_bf16_bits(x32)
    ref = torch.from_numpy(x32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oursb, ref)


def test_fill_tokens_is_value_of_centred_sum():
    seed, tag = 1234567, synth.tag(synth.K_TENSOR, 5)
    tok_t = np.array([0, 7, 4095, 70000], dtype=np.int32)
    tok_s = np.array([3, 0, 127, 1], dtype=np.int32)
    H, d = 3, 80
    for dtype in ("f16", "bf16"):
        scale = synth.scale_for(1.0)
        out = synth.fill_tokens_host(seed, dtype, scale, tag, tok_t, tok_s, H, d)
        i0 = np.repeat(tok_t, H * d).astype(np.uint32)
        i1 = np.repeat(tok_s, H * d).astype(np.uint32)
        i2 = np.tile((np.arange(H)[:, None] * 1024 + np.arange(d)[None, :]).reshape(-1), tok_t.size).astype(np.uint32)
        c = synth.centred_sums(seed, tag, i0, i1, i2)
        x = c.astype(np.float32) * scale
        ref = synth.f32_to_f16_bits(x) if dtype == "f16" else synth.f32_to_bf16_bits(x)
        assert np.array_equal(out.reshape(-1), ref)


def test_generator_statistics():
    n = 1 << 20
    i0 = np.arange(n, dtype=np.uint32)
    c = synth.centred_sums(99, 0, i0, np.zeros(n, np.uint32), np.zeros(n, np.uint32))
    assert c.min() >= -131070 and c.max() <= 131070
    std = 65536 / np.sqrt(3)
    assert abs(c.mean()) < 5 * std / np.sqrt(n)
    assert abs(c.std() / std - 1) < 0.01
    x = synth.fill_tokens_host(7, "f16", synth.scale_for(1.0), 1, np.arange(4096), np.zeros(4096), 4, 64)
    v = x.view(np.float16).astype(np.float64)
    assert abs(v.std() - 1) < 0.01 and np.abs(v).max() <= 3.47


def test_philox_outputs_decorrelated_across_counters():
    ctr = np.zeros((4096, 4), dtype=np.uint32)
    ctr[:, 0] = np.arange(4096)
    out = synth.philox_blocks(ctr, np.zeros((4096, 2), dtype=np.uint32))
    bits = np.unpackbits(out.view(np.uint8))
    assert abs(bits.mean() - 0.5) < 0.005
    assert len(np.unique(out[:, 0])) == 4096
    # different keys give different streams
    out2 = synth.philox_blocks(ctr, np.ones((4096, 2), dtype=np.uint32))
    assert (out2 != out).mean() > 0.99
