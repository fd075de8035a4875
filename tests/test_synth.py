"""The seeded input generator: deterministic, with the requested distributions."""
import numpy as np

from paper_2309_00754_gb300 import synth


def test_deterministic_and_stream_separated():
    a = synth.normal_bf16(7, (64, 33), 0.02)
    b = synth.normal_bf16(7, (64, 33), 0.02)
    c = synth.normal_bf16(8, (64, 33), 0.02)
    assert a.dtype == np.uint16 and np.array_equal(a, b) and not np.array_equal(a, c)


def test_moments_and_ranges():
    x = synth.bf16_bits_to_f32(synth.normal_bf16(11, (1 << 18,), 0.02)).astype(np.float64)
    assert abs(x.mean()) < 3e-4 and abs(x.std() - 0.02) < 3e-4
    ids = synth.randint(12, (1 << 16,), 0, 32000)
    assert ids.min() >= 0 and ids.max() < 32000 and abs(ids.mean() - 16000) < 300
    lens = synth.randint(13, (4096,), 64, 513)
    assert lens.min() == 64 and lens.max() == 512


def test_bf16_round_to_nearest_even():
    v = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5], dtype=np.float32)
    got = synth.bf16_bits_to_f32(synth.f32_to_bf16_bits(v))
    assert list(got) == [1.0, 1.0, 1.0 + 2 ** -6, -2.5]
