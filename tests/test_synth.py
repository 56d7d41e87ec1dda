"""The seeded input generators: deterministic, counter-based, with the stated distributions."""
import numpy as np

import synth


def test_deterministic_and_prefix_stable():
    a = synth.normal_bf16(0, 7, (1000,), std=0.02)
    b = synth.normal_bf16(0, 7, (100,), std=0.02)
    np.testing.assert_array_equal(a[:100], b)
    np.testing.assert_array_equal(a, synth.normal_bf16(0, 7, (1000,), std=0.02))
    assert not np.array_equal(a, synth.normal_bf16(0, 8, (1000,), std=0.02))
    assert not np.array_equal(a, synth.normal_bf16(1, 7, (1000,), std=0.02))


def test_normal_statistics():
    x = synth.bf16_to_f64(synth.normal_bf16(3, 1, (1 << 20,), std=0.02))
    assert abs(x.mean()) < 1e-4
    assert abs(x.std() - 0.02) < 1e-4
    z = synth.normal_f64(3, 2, (1 << 20,))
    assert abs(np.mean(z ** 4) - 3.0) < 0.05          # Gaussian kurtosis


def test_uniform_ints_cover_range():
    v = synth.uniform_i32(0, 41, (200000,), 0, 2048)
    assert v.min() == 0 and v.max() == 2047
    counts = np.bincount(v, minlength=2048)
    assert counts.min() > 50 and counts.max() < 150


def test_bf16_rounding_is_nearest_even():
    f = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 1.0 + 2 ** -9], dtype=np.float32)
    bits = synth.f32_to_bf16(f)
    back = synth.bf16_to_f32(bits)
    # halfway cases go to the even mantissa: 1+2^-8 -> 1, 1+3*2^-8 -> 1+2^-6
    np.testing.assert_array_equal(back, np.array([1.0, 1.0, 1.0 + 2 ** -6, -2.5, 1.0], dtype=np.float32))


def test_workload_shapes():
    w = synth.LLAVA7B
    assert w.prompt_len == 640 and w.shape.qdim == 4096
    assert w.shape.layer_bytes_bf16() - 4 * 4096 == 2 * (4 * 4096 ** 2 + 3 * 4096 * 11008)
    sc = w.resid_scale()
    assert sc[:8].tolist() == [1.0] * 8 and np.all(sc[8:] == np.float32(0.2))
