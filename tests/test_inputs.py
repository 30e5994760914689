"""The seeded input generator shared by the CUDA path's tests and the oracle,
checked against definitions outside itself (CPU only).

* SplitMix64 (Steele, Lea and Flood, 2014; the reference C code by Vigna):
  starting from state 0, the first output is 0xE220A8397B1DCDAF.
* The bf16 rounding equals PyTorch's float32 -> bfloat16 conversion (round to
  nearest, ties to even) on random values, on ties and on values near the
  largest finite bf16.
* The standardised Irwin-Hall(4) draws have mean 0 and variance 1, and the
  value patterns used for V are finite bf16 numbers.
"""
import numpy as np
import pytest

from paper_2606_15157_gb300 import inputs as gen


def test_splitmix64_published_first_output():
    assert int(gen.hash64(0, np.array([0], np.uint64))[0]) == 0xE220A8397B1DCDAF


def test_splitmix64_counters_are_the_sequence():
    # hash64(key, i) is output i + 1 of the generator started at state `key`:
    # advancing the key by one step shifts the sequence by one
    key = 0x0123456789ABCDEF
    a = gen.hash64(key, np.arange(1, 65, dtype=np.uint64))
    b = gen.hash64((key + gen.GAMMA) & gen.MASK64, np.arange(0, 64, dtype=np.uint64))
    assert np.array_equal(a, b)


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(3)
    x = np.concatenate([
        rng.standard_normal(100000).astype(np.float32) * np.float32(10.0) ** rng.integers(-30, 30, 100000).astype(np.float32),
        # exact ties between two bf16 values, both parities of the kept bit
        (np.arange(0, 4096, dtype=np.uint32) << 16 | 0x8000).view(np.float32)[1:-1],
        np.array([3.3895314e38, -3.3895314e38, 1e-40, -1e-40, 0.0, -0.0], np.float32),
    ])
    x = x[np.isfinite(x)]
    ours = gen.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_gauss_moments_and_value_bits_finite():
    idx = np.arange(1 << 20, dtype=np.uint64)
    g = gen.gauss_f32(gen.stream_key(7, gen.T_K, 3), idx).astype(np.float64)
    assert abs(g.mean()) < 5e-3 and abs(g.var() - 1.0) < 5e-3
    assert np.abs(g).max() <= 2 * np.sqrt(3) + 1e-6   # Irwin-Hall(4) support: +-2 sqrt(3)
    v = gen.value_bits(gen.stream_key(7, gen.T_V, 3), idx)
    assert np.all(np.isfinite(gen.bf16_bits_to_f32(v)))
