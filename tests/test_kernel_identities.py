"""Integer identities the CUDA kernels use in place of the paper's literal steps, checked
exhaustively on the CPU over the ranges the kernels admit (numpy int64 arithmetic)."""
import numpy as np
import pytest


def test_shiftexp_exponent_on_magnitudes():
    """Algorithm 1 floors I + (I >> 1) - (I >> 4) for I <= 0.  The kernels take a = -I >= 0 and
    form -I_e = a + ((a+1) >> 1) - ((a+15) >> 4), shifting only non-negative values."""
    a = np.arange(0, 1 << 22, dtype=np.int64)
    I = -a
    literal = I + (I >> 1) - (I >> 4)  # numpy >> on int64 floors, as the paper's shifts do
    kernel = a + ((a + 1) >> 1) - ((a + 15) >> 4)
    assert np.array_equal(-literal, kernel)
    big = np.array([(1 << 30) - 1, 1 << 30], dtype=np.int64)
    assert np.array_equal(-(-big + ((-big) >> 1) - ((-big) >> 4)), big + ((big + 1) >> 1) - ((big + 15) >> 4))


@pytest.mark.parametrize("I0", [1, 2, 3, 7, 255, 256, 300, 1000, 4095, 4096, 16383, (1 << 15) - 1])
def test_invariant_divisor_reciprocal(I0):
    """q = floor(n / I0) as floor(n * M / 2^40) with M = ceil(2^40 / I0) (Granlund & Montgomery,
    1994), computed the kernels' way: (umulhi(n, M_lo) + n * M_hi) >> 8, for every n in [0, 16 I0]."""
    k = 16
    n = np.arange(0, k * I0 + 1, dtype=np.uint64)
    M = ((1 << 40) + I0 - 1) // I0
    m_lo, m_hi = np.uint64(M & 0xFFFFFFFF), np.uint64(M >> 32)
    t = ((n * m_lo) >> np.uint64(32)) + n * m_hi
    q = (t & np.uint64(0xFFFFFFFF)) >> np.uint64(8)
    assert np.array_equal(q, n // np.uint64(I0))


def test_sigmoid_uses_one_shiftexp():
    """SD-ShiftGELU: with I_shift = ReLU(I_p), I_delta = I_p - I_shift, exactly one of I_delta
    and -I_shift is 0 (both when I_p = 0), so {I_delta, -I_shift} = {0, -|I_p|}."""
    Ip = np.arange(-100000, 100001, dtype=np.int64)
    Ish = np.maximum(Ip, 0)
    Id = Ip - Ish
    pair = np.sort(np.stack([Id, -Ish]), axis=0)
    assert np.array_equal(pair[0], -np.abs(Ip)) and np.all(pair[1] == 0)
