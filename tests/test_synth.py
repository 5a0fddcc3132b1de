"""The seeded input generator shared by the CUDA path and the oracle, pinned to the published
definitions it names: SplitMix64 (Steele, Lea, Flood 2014) and 64-bit FNV-1a, with their
published test vectors; plus the properties the tests rely on (bounded draws stay in range and
reach both ends, the draw order of tensors does not matter, Laplace draws are clipped)."""
import numpy as np

from paper_2607_24981_gb300 import synth


def test_splitmix64_published_vectors():
    """SplitMix64 started from state 0 yields e220a8397b1dcdaf, 6e789e6aa1b965f4,
    06c45d188009454f, f88bb8a8724c81ec (the reference implementation's first four outputs);
    output i of a stream keyed k is the mixer applied to k + i * 0x9e3779b97f4a7c15."""
    states = np.arange(1, 5, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    got = [int(v) for v in synth._mix(states)]
    assert got == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F, 0xF88BB8A8724C81EC]


def test_fnv1a_published_vectors():
    """64-bit FNV-1a of "", "a" and "foobar" (the FNV test suite's values)."""
    assert synth._fnv1a("") == 0xCBF29CE484222325
    assert synth._fnv1a("a") == 0xAF63DC4C8601EC8C
    assert synth._fnv1a("foobar") == 0x85944171F73967E8


def test_streams_are_keyed_not_ordered():
    """A tensor's bytes depend on (seed, name) only: drawing other tensors first, or drawing a
    prefix, changes nothing; another name or seed gives another stream."""
    a = synth.raw_u64(3, "x", 100)
    synth.raw_u64(3, "y", 1000)
    assert np.array_equal(synth.raw_u64(3, "x", 100), a)
    assert np.array_equal(synth.raw_u64(3, "x", 10), a[:10])
    assert not np.array_equal(synth.raw_u64(3, "y", 100), a)
    assert not np.array_equal(synth.raw_u64(4, "x", 100), a)


def test_bounded_draws_cover_their_range():
    """Multiply-shift of the top 32 bits maps onto [lo, hi] inclusive: every value of a small
    range appears and nothing falls outside, also at the int8 extremes and a full 2^32 span."""
    v = synth.uniform_int(1, "small", (20000,), -3, 4)
    assert set(np.unique(v).tolist()) == set(range(-3, 5))
    w = synth.uniform_int(1, "w", (100000,), -127, 127, np.int8)
    assert w.min() == -127 and w.max() == 127
    f = synth.uniform_int(1, "full", (1000,), -(1 << 31), (1 << 31) - 1, np.int64)
    assert f.min() >= -(1 << 31) and f.max() <= (1 << 31) - 1 and f.min() < 0 < f.max()


def test_laplace_draws_are_clipped_and_symmetric():
    x = synth.laplace_int(2, "lap", (200000,), 20.0, 127, np.int16)
    assert x.min() == -127 and x.max() == 127
    assert abs(float(x.mean())) < 0.5
    assert 18.0 < float(np.abs(x).mean()) < 21.0  # E|X| = scale for Laplace(0, scale), lightly clipped
