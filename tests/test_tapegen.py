"""Host-side checks of the seeded synthetic tape generator."""
import numpy as np

import tapegen


def test_geometric_tape_structure():
    rng = np.random.default_rng(0)
    L = 1_000_000
    lens = tapegen.episode_lengths_geometric(rng, L, 500.0, 1, 10000)
    assert lens.sum() == L and lens.min() >= 1 and lens.max() <= 10000
    # every episode but the truncated last one is a full Geometric draw
    assert abs(lens[:-1].mean() - 500.0) < 50.0
    start = tapegen.starts_from_lengths(lens, L)
    assert start[0] == 1 and start.sum() == len(lens)


def test_seeded_and_reproducible():
    a = tapegen.diag_tape(2, 300, 8, seed=5)
    b = tapegen.diag_tape(2, 300, 8, seed=5)
    for k in ("lam", "u", "start", "grad_h"):
        np.testing.assert_array_equal(a[k], b[k])


def test_complex_normal_moments():
    rng = np.random.default_rng(1)
    z = tapegen.complex_normal(rng, (200_000,))
    assert z.dtype == np.complex64
    assert abs(np.var(z.real) - 0.5) < 0.01 and abs(np.var(z.imag) - 0.5) < 0.01


def test_lambda_ranges():
    lam = tapegen.diag_lambda(np.random.default_rng(2), (10_000,))
    m = np.abs(lam)
    assert m.min() >= 0.9 - 1e-6 and m.max() <= 0.999 + 1e-6


def test_bf16_rounding_round_trip():
    x = np.array([1.0, -2.5, 3.14159265, 1e-20, 65504.0, 0.1], dtype=np.float32)
    bits = tapegen.f32_to_bf16_bits(x)
    back = tapegen.bf16_bits_to_f32(bits)
    assert np.all(np.abs(back - x) <= np.abs(x) * 2.0 ** -8)
    # values already representable in bf16 are exact
    np.testing.assert_array_equal(tapegen.bf16_bits_to_f32(tapegen.f32_to_bf16_bits(back)), back)
    # ties round to even: 1 + 2^-8 lies halfway between 1 and 1 + 2^-7
    assert tapegen.bf16_bits_to_f32(tapegen.f32_to_bf16_bits(np.float32([1 + 2 ** -8])))[0] == 1.0


def test_linattn_tape_k_normalised():
    t = tapegen.linattn_tape(1, 64, 2, 16, 16, seed=3)
    k = tapegen.bf16_bits_to_f32(t["k"])
    n = np.linalg.norm(k, axis=-1)
    assert np.all(np.abs(n - 1.0) < 0.02)
