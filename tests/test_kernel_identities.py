"""Integer identities the CUDA kernels use in place of the paper's literal steps, checked
exhaustively on the CPU over the ranges the kernels admit (numpy int64 arithmetic)."""
import math

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


def test_shiftexp_exponent_from_biased_float_bits():
    """Attention reads a = max - s off the bits of the fp32 value (max + 2^23) - s: for integer
    scores |s|, |max| < 2^20 that value is exact, so its bits are 0x4B000000 + a; and since
    0x4B000000 is a multiple of 16, -I_e = a + ceil(a/2) - ceil(a/16) equals
    b + ((b+1) >> 1) - ((b+15) >> 4) - 1808793600 in wrapping 32-bit arithmetic."""
    rng = np.random.default_rng(11)
    s = rng.integers(-(1 << 20) + 1, 1 << 20, size=1 << 20)
    mx = np.maximum(s, rng.integers(-(1 << 20) + 1, 1 << 20, size=s.size))
    mb = mx.astype(np.float32) + np.float32(8388608.0)
    bits = (mb - s.astype(np.float32)).view(np.uint32).astype(np.int64)
    assert np.array_equal(bits, 0x4B000000 + (mx - s))
    a = np.arange(0, 1 << 22, dtype=np.int64)
    b = (0x4B000000 + a).astype(np.uint32)
    n_bits = b + ((b + np.uint32(1)) >> np.uint32(1)) - ((b + np.uint32(15)) >> np.uint32(4)) - np.uint32(1808793600)
    assert np.array_equal(n_bits.astype(np.int64), a + ((a + 1) >> 1) - ((a + 15) >> 4))
    assert 0x4B000000 % 16 == 0 and 0x4B000000 + 0x4B000000 // 2 - 0x4B000000 // 16 == 1808793600


@pytest.mark.parametrize("I0", [2, 3, 7, 255, 1000, 4096, 6151, 9999, 12289, 16383])
def test_single_multiply_quotient_and_half_remainder(I0):
    """With m32 = ceil(2^32 / I0) and k I0^2 < 2^32, umulhi(n, m32) = floor(n / I0) for every
    n <= k I0 (the error n (m32 I0 - 2^32) / 2^32 stays below 1/I0); and I0 - ceil(r/2) for
    r = n - q I0 equals ((q + 2) I0 - n) >> 1."""
    k = 16
    assert k * I0 * I0 < (1 << 32)
    n = np.arange(0, k * I0 + 1, dtype=np.uint64)
    m32 = np.uint64(((1 << 32) + I0 - 1) // I0)
    q = (n * m32) >> np.uint64(32)
    assert np.array_equal(q, n // np.uint64(I0))
    r = n - q * np.uint64(I0)
    assert np.array_equal(np.uint64(I0) - ((r + np.uint64(1)) >> np.uint64(1)),
                          ((q + np.uint64(2)) * np.uint64(I0) - n) >> np.uint64(1))


def test_single_multiply_quotient_fails_past_the_bound():
    """The bound matters: for I0 = 30000, k = 16 (k I0^2 >= 2^32) the single multiply misreads
    n = 359999 as 12 instead of 11, so the kernels keep the 40-bit reciprocal there."""
    I0, k = 30000, 16
    assert k * I0 * I0 >= (1 << 32)
    n = np.uint64(359999)
    m32 = np.uint64(((1 << 32) + I0 - 1) // I0)
    assert int((n * m32) >> np.uint64(32)) == 12 and int(n) // I0 == 11


def _newton_fixed(V, iters):
    r = 1 << 16
    for _ in range(iters):
        if r == 0:
            break
        r = (r + V // r) >> 1
    return max(r, 1)


def _newton_early(V, iters):
    """The I-LayerNorm kernels' schedule: stop at a fixed point, or resolve a 2-cycle by parity."""
    r, prev = 1 << 16, None
    for it in range(iters):
        if r == 0:
            break
        nx = (r + V // r) >> 1
        if nx == r:
            break
        if nx == prev:
            r = r if (iters - it - 1) & 1 else nx
            break
        prev, r = r, nx
    return max(r, 1)


def test_newton_early_exit_matches_fixed_iteration_count():
    """Cutting Newton's integer square root short (fixed point, or the s <-> s+1 alternation at
    V = s^2 + 2s) gives exactly the value of the full `iters` steps, for every iteration count."""
    rng = np.random.default_rng(5)
    Vs = [0, 1, 2, 3, 8, 15, 24, 35, (1 << 32) - 1, 1 << 32, (1 << 40) - 1]
    Vs += [s * s + 2 * s for s in (1, 2, 3, 255, 256, 65535, 65536, 70000, 1 << 19)]
    Vs += [int(v) for v in rng.integers(0, 1 << 40, size=3000)]
    Vs += [int(v) for v in rng.integers(0, 1 << 20, size=2000)]
    for V in Vs:
        for iters in range(0, 21):
            assert _newton_early(V, iters) == _newton_fixed(V, iters), (V, iters)


def test_shiftmax_output_from_shiftexp_parts():
    """Attention forms the Constrained Shiftmax output (I_exp F) >> sh from ShiftExp's parts: with
    I_exp = I_b << (k - q) and sh = 31 - k_out + 1 + s_d >= k, floor(I_exp F / 2^sh) equals
    floor(I_b F / 2^(sh - k + q)), and a shift amount of 32 or more gives 0 (PTX shr saturates).
    Also checked: I_b F < 2^32 under the conditions the host requires (per-row s_d,
    m_p <= M_hw - 15), with F from the bounds of S_R."""
    rng = np.random.default_rng(5)
    k, k_out = 16, 8
    for s_d in range(0, 16):
        sh = 31 - k_out + 1 + s_d
        Ib = rng.integers(1, 1 << 15, size=1 << 16).astype(object)
        q = rng.integers(0, k + 1, size=Ib.size)
        F = rng.integers(1, 1 << 15, size=Ib.size).astype(object)
        lit = [((int(b) << (k - int(qq))) * int(f)) >> sh for b, qq, f in zip(Ib, q, F)]
        amt = [sh - k + int(qq) for qq in q]
        direct = [0 if n >= 32 else (((int(b) * int(f)) & 0xFFFFFFFF) >> n) for b, f, n in zip(Ib, F, amt)]
        assert lit == direct
    # F bounds: s_d > 0 puts S_R in [2^(M_hw - m_p - 1), 2^31) ; s_d = 0 has S_R >= I0 2^k > I_b 2^k
    for m_p, M_hw in [(4, 31), (0, 15), (16, 31)]:
        F_max = (2**31 - 1) // (1 << (M_hw - m_p - 1))
        assert (2**15 - 1) * F_max < 2**32
    I0 = np.arange(1, 1 << 15, dtype=object)
    assert all(int(i) * ((2**31 - 1) // (int(i) << k)) < 2**32 for i in I0[: (1 << 15) >> 1])


def _div_u48_u32(V, r):
    """The kernels' floor(V / r) for V < 2^48, r < 2^32 (quotient < 2^26), in float32 arithmetic:
    correctly rounded reciprocal, 64-bit integers converted as two 32-bit halves joined by one fma,
    truncation / floor back to integers."""
    f32 = np.float32

    def to_f32(v):  # the kernels' conversion of a 64-bit integer: two 32-bit halves and one fma
        hi, lo = v >> 32, v & 0xFFFFFFFF
        return f32(float(f32(hi)) * 4294967296.0 + float(f32(lo)))  # exact in float64, rounded once

    rinv = f32(1.0) / f32(r)
    q = np.uint64(np.trunc(to_f32(int(V)) * rinv))
    rem = int(V) - int(q) * int(r)
    dq = int(np.floor(to_f32(rem) * rinv))
    q = int(q) + dq
    rem -= dq * int(r)
    if rem < 0:
        q -= 1
    elif rem >= r:
        q += 1
    return q


def test_float_assisted_division_in_newton():
    """I-LayerNorm's Newton steps divide V < 2^48 by r >= isqrt(V) (r < 2^32, quotient < 2^25); the
    float-estimate division with one refinement and a +-1 test gives floor(V / r) exactly."""
    import math

    rng = np.random.default_rng(3)
    cases = []
    for e in range(1, 48):
        for _ in range(300):
            V = int(rng.integers(1 << (e - 1), 1 << e))
            s = math.isqrt(V)
            for r in (max(s, 1), s + 1, s + 2, 2 * s + 7, max(1, (1 << 16) + (V >> 16)) >> 1):
                if 1 <= r < 2**32 and V // r < 2**26:
                    cases.append((V, r))
    for V in ((1 << 48) - 1, (1 << 47), 12345678901234):
        s = math.isqrt(V)
        cases += [(V, s), (V, s + 1), (V, s - 1 if s > 1 else 1)]
    for V, r in cases:
        assert _div_u48_u32(V, r) == V // r, (V, r)


def test_high_word_requantisation_forms():
    """For int32 v, |m| < 2^31 and s in [33, 62] the kernels requantise from the high word of v m:
    rq(v; m, s) = ((hi >> (s-33)) + 1) >> 1 = (hi + 2^(s-33)) >> (s-32), hi = floor(v m / 2^32)
    (the second form is one mad.hi plus a shift), against exact rq = floor((v m + 2^(s-1)) / 2^s)."""
    rng = np.random.default_rng(17)
    v = np.concatenate([rng.integers(-(2**31), 2**31, 20000), [-(2**31), 2**31 - 1, 0, 1, -1]])
    m = np.concatenate([rng.integers(-(2**31) + 1, 2**31, 20000), [2**31 - 1, -(2**31) + 1, 2**30, -(2**30), 7]])
    for s in (33, 34, 40, 47, 51, 62):
        for vi, mi in zip(v.tolist(), m.tolist()):
            p = vi * mi
            exact = (p + (1 << (s - 1))) >> s
            hi = p >> 32
            assert ((hi >> (s - 33)) + 1) >> 1 == exact
            assert (hi + (1 << (s - 33))) >> (s - 32) == exact
            assert -(2**31) <= hi + (1 << (s - 33)) < 2**31



def test_relu_on_packed_bytes():
    """The int8 ReLU kernel clears each byte whose sign bit is set: w & ~(((w & 0x80808080) >> 7) *
    0xFF) (the product has no carries: one low bit per byte), against bytewise max(0, b)."""
    rng = np.random.default_rng(0)
    w = rng.integers(0, 1 << 32, size=200000, dtype=np.uint64)
    w[:4] = [0, 0xFFFFFFFF, 0x80808080, 0x7F7F7F7F]
    neg = (w & np.uint64(0x80808080)) >> np.uint64(7)
    got = w & ~(neg * np.uint64(0xFF)) & np.uint64(0xFFFFFFFF)
    b = w.astype(np.uint32).view(np.int8).reshape(-1, 4)
    want = np.maximum(b, 0).astype(np.int8).view(np.uint32).reshape(-1)
    assert np.array_equal(got.astype(np.uint32), want)


def test_topk_key_order():
    """The top-K sort key (value biased to unsigned) << 32 | (2^32 - 1 - index), sorted in decreasing
    order, is the order value descending, index ascending; padding keys (0) sort after every key."""
    rng = np.random.default_rng(1)
    v = rng.integers(-3, 4, size=5000).astype(np.int64)
    v[:3] = [-(1 << 31), (1 << 31) - 1, -(1 << 31)]
    i = np.arange(v.size, dtype=np.int64)
    key = (((v + (1 << 31)) & 0xFFFFFFFF).astype(np.uint64) << np.uint64(32)) | (np.uint64(0xFFFFFFFF) - i.astype(np.uint64))
    by_key = sorted(range(v.size), key=lambda j: -int(key[j]))  # exact 64-bit comparisons
    assert by_key == list(np.lexsort((i, -v)))
    assert int(key.min()) > 0


@pytest.mark.parametrize("nq,H,Z", [(1, 1, 1), (13, 6, 8), (4, 6, 32), (1, 8, 3), (2, 1, 5)])
def test_attention_cta_order_is_a_bijection(nq, H, Z):
    """The tensor-memory attention maps CTA L to (query tile, head, group): the first (nq - 1) H Z
    CTAs take the tiles of every group but its last (tile fastest), the remaining H Z CTAs the last
    tiles.  Every (tile, head, group) is taken exactly once, and the last tiles come last."""
    F = (nq - 1) * H * Z
    seen = []
    for L in range(nq * H * Z):
        if L < F:
            t = (L % (nq - 1), (L // (nq - 1)) % H, L // ((nq - 1) * H))
        else:
            t = (nq - 1, (L - F) % H, (L - F) // H)
        seen.append(t)
    assert sorted(seen) == sorted((q, h, z) for q in range(nq) for h in range(H) for z in range(Z))
    assert all(t[0] == nq - 1 for t in seen[F:]) and all(t[0] < nq - 1 for t in seen[:F])


@pytest.mark.parametrize("nq,H,Z", [(1, 1, 1), (1, 3, 3), (13, 6, 8), (8, 3, 3), (2, 8, 1)])
def test_attention_paired_last_tiles_cover_every_unit(nq, H, Z):
    """Global attention whose last tile has at most 64 queries: CTA j < ceil(H Z / 2) holds the last
    tiles of units 2 j and 2 j + 1 (unit = head + H image; the second absent when H Z is odd), the
    paired CTAs first; the remaining (nq - 1) H Z CTAs keep the one-tile mapping.  Every
    (tile, unit) is taken once, pairs may span two images, and the grid shrinks by floor(H Z / 2)
    CTAs."""
    F = (nq - 1) * H * Z
    units = H * Z
    npr = (units + 1) // 2
    grid = F + npr
    seen = []
    for cta in range(grid):
        L = F + cta if cta < npr else cta - npr
        if L < F:
            seen.append((L % (nq - 1), (L // (nq - 1)) % H, L // ((nq - 1) * H)))
        else:
            u0 = 2 * (L - F)
            seen.append((nq - 1, u0 % H, u0 // H))
            if u0 + 1 < units:
                seen.append((nq - 1, (u0 + 1) % H, (u0 + 1) // H))
            else:
                assert cta == npr - 1 and units % 2 == 1
    assert sorted(seen) == sorted((q, h, z) for q in range(nq) for h in range(H) for z in range(Z))
    assert grid == nq * units - units // 2


@pytest.mark.parametrize("nkb", [1, 2, 3, 13, 25])
def test_attention_piece_stream_matches_mma_order(nkb):
    """The loader's piece sequence (k blocks of passes 1 and 2, then k0, k(j + 1), v(j) ..., v(nkb - 1))
    is exactly the order in which the MMA issuer consumes ring slots: scores of block kb + 1 before
    the P V of block kb in pass 3."""
    loads = []
    for i in range(4 * nkb):
        if i < 2 * nkb:
            loads.append(("k", i if i < nkb else i - nkb))
        else:
            j = i - 2 * nkb
            if j == 0:
                loads.append(("k", 0))
            elif j == 2 * nkb - 1:
                loads.append(("v", nkb - 1))
            elif j & 1:
                loads.append(("k", (j + 1) >> 1))
            else:
                loads.append(("v", (j - 2) >> 1))
    mma = [("k", j % nkb) for j in range(2 * nkb)] + [("k", 0)]
    for kb in range(nkb - 1):
        mma += [("k", kb + 1), ("v", kb)]
    mma.append(("v", nkb - 1))
    assert loads == mma


@pytest.mark.parametrize("ws", [1, 5, 7, 12, 20, 40, 64, 100, 128])
def test_attention_window_key_boxes(ws):
    """Window key blocks are 3-D boxes of R = min(floor(128 / ws), ws) whole window rows: row z,
    column y of the box of block kb is grid cell (wy ws + kb R + z, wx ws + y), which is key
    kb R ws + z ws + y of the window in row-major order; the blocks cover every key once and the
    keys at or past ws^2 are the ones masked."""
    R = min(128 // ws, ws)
    kbk = R * ws
    nkb = -(-ws * ws // kbk)
    wy, wx = 1, 2
    got = {}
    for kb in range(nkb):
        for z in range(R):
            for y in range(ws):
                key = kb * kbk + z * ws + y
                cell = (wy * ws + kb * R + z, wx * ws + y)
                if key < ws * ws:
                    assert cell == (wy * ws + key // ws, wx * ws + key % ws)
                    got[key] = cell
                else:
                    assert kb * R + z >= ws  # past the window: a masked column
    assert sorted(got) == list(range(ws * ws)) and kbk <= 128


def _shift_exp_mag_model(a, I0, k):
    """The kernels' ShiftExp of -a in 32-bit unsigned arithmetic (a <= 2^30): n = a + ceil(a/2) -
    ceil(a/16), clamped at k I0; q = floor(n / I0); I_b = I0 - ceil(r / 2); I_b << (k - q)."""
    a = np.asarray(a, dtype=np.uint64)
    n = (a + ((a + 1) >> np.uint64(1)) - ((a + 15) >> np.uint64(4))) & np.uint64(0xFFFFFFFF)
    n = np.minimum(n, np.uint64(k * I0))
    q = n // np.uint64(I0)
    r = n - q * np.uint64(I0)
    Ib = np.uint64(I0) - ((r + 1) >> np.uint64(1))
    return (Ib << (np.uint64(k) - q)).astype(np.int64)


@pytest.mark.parametrize("I0,k", [(1, 0), (3, 16), (600, 8), (1024, 8), (18764, 8), (32767, 0)])
def test_clamped_magnitude_shiftexp(orc, I0, k):
    """The detection-head and I-ViT kernels clamp the ShiftExp magnitude at 2^30 before the 32-bit
    form: past k I0 ShiftExp sits in its clamp region, so for every a >= 0 (up to 2^31 and the
    int32 extreme) ShiftExp(-min(a, 2^30)) in the kernels' arithmetic equals Algorithm 1's
    ShiftExp(-a)."""
    rng = np.random.default_rng(I0)
    edge = np.array([0, 1, 2, 15, 16, 17, k * I0 - 1, k * I0, k * I0 + 1, (1 << 30) - 1, 1 << 30,
                     (1 << 30) + 1, (1 << 31) - 1, 1 << 31], dtype=np.int64)
    a = np.concatenate([edge[edge >= 0], np.arange(0, 40 * I0 + 64, max(1, I0 // 50)),
                        rng.integers(0, 1 << 31, 2000)])
    got = _shift_exp_mag_model(np.minimum(a, 1 << 30), I0, k)
    want = np.array([orc.shiftexp(-int(x), I0, k) for x in a], dtype=np.int64)
    assert np.array_equal(got, want)


def test_shiftexp_exponent_from_negative_biased_bits():
    """The attention kernel's score MMA adds -C = -(2^23 + max + 1) to q.k, so TMEM holds the fp32
    value s - C = -(2^23 + a + 1) for a = max - s.  For every integer score pair with a in
    [0, 2^22] (|scores| < 2^20, so a <= 2^21 in practice) that value is exact, its bits are
    0xCB000000 + a + 1, and w + (w >> 1) - ((w + 14) >> 4) - 0x23D00001 (32-bit wrap-around) equals
    a + ceil(a/2) - ceil(a/16)."""
    a = np.arange(0, (1 << 22) + 1, dtype=np.int64)
    mx = np.int64(12345)
    s = mx - a
    C = (1 << 23) + mx + 1
    val = (s - C).astype(np.float32)  # exact: |s - C| < 2^24
    assert np.array_equal(val.astype(np.int64), s - C)
    w = val.view(np.uint32).astype(np.uint64)
    assert np.array_equal(w, 0xCB000000 + a + 1)
    M32 = np.uint64(0xFFFFFFFF)
    n = (w + (w >> np.uint64(1)) - ((w + np.uint64(14)) >> np.uint64(4)) - np.uint64(0x23D00001)) & M32
    assert np.array_equal(n.astype(np.int64), a + ((a + 1) >> 1) - ((a + 15) >> 4))



def test_shiftmax_rows_one_multiply_output():
    """The standalone Shiftmax rows kernel writes floor(e F / 2^sh) as umulhi(e, Fs) >> rs: for
    sh <= 32 and F < 2^sh, Fs = F 2^(32 - sh), rs = 0; for sh > 32, Fs = F, rs = min(sh - 32, 31);
    other rows take the 64-bit form.  Checked against the exact floor for e < 2^31 over the whole
    range of F and sh, extremes included."""
    rng = np.random.default_rng(7)
    es = np.concatenate([rng.integers(0, 1 << 31, 4000), [0, 1, (1 << 31) - 1, (1 << 30), 12345]])
    checked = 0
    for sh in list(range(17, 64)):
        Fs_list = np.concatenate([rng.integers(1, 1 << 31, 60), [1, 2, 31, 32, (1 << 31) - 1, 1 << 24]])
        for F in Fs_list:
            F = int(F)
            if sh <= 32:
                ok = sh == 32 or (F >> sh) == 0
                Fs, rs = (F << (32 - sh)) if ok else 0, 0
            else:
                ok, Fs, rs = True, F, min(sh - 32, 31)
            if not ok:
                continue
            assert Fs < (1 << 32)
            for e in es:
                e = int(e)
                assert ((e * Fs) >> 32) >> rs == (e * F) >> sh
                checked += 1
    assert checked > 100000


def test_attention_p_as_one_high_word_product():
    """Attention's pass 3 writes P = floor(I_b F / 2^(sh0 + q)) as umulhi(I_b, G) >> q, with
    G = F 2^(32 - sh0) when sh0 <= 32 and F < 2^sh0, and G = 0 when sh0 > 32 (there I_b F < 2^32
    <= 2^sh0, so every P is 0).  Checked against the exact floor over I_b < 2^15, the F and sh0 a
    row can have, and every q <= 31."""
    rng = np.random.default_rng(11)
    ibs = np.concatenate([rng.integers(0, 1 << 15, 300), [0, 1, (1 << 15) - 1, 1 << 14]])
    checked = 0
    for sh0 in range(0, 48):
        for F in np.concatenate([rng.integers(1, 1 << 31, 40), [1, 2, 31, 32, 255, 256, (1 << 31) - 1]]):
            F = int(F)
            ok = sh0 >= 32 or (F >> sh0) == 0
            if not ok:
                continue
            G = 0 if sh0 > 32 else (F if sh0 == 32 else F << (32 - sh0))
            assert G < (1 << 32)
            for ib in ibs:
                ib = int(ib)
                if sh0 > 32 and ib * F >= (1 << 32):
                    continue  # outside the kernel's condition I_b F < 2^32
                for q in (0, 1, 7, 15, 16, 31):
                    assert ((ib * G) >> 32) >> q == (ib * F) >> (sh0 + q)
                    checked += 1
    assert checked > 100000


@pytest.mark.parametrize("LPR,CPL,C,EPC", [(4, 12, 192, 4), (8, 12, 384, 4), (8, 6, 384, 8), (16, 6, 704, 8),
                                            (32, 6, 1024, 8)])
@pytest.mark.parametrize("rows,grid", [(1, 1), (77, 3), (12800, 400), (1000, 7)])
def test_layernorm_rows_mapping(LPR, CPL, C, EPC, rows, grid):
    """The I-LayerNorm row kernel: 256 threads, LPR lanes per row, RPW = 32 / LPR rows per warp and
    RPC = 8 RPW rows per CTA step; CTA b takes the steps at rows r0 = b RPC + k grid RPC.  Lane l
    of warp w owns row r0 + lrow, lrow = w RPW + l / LPR, and chunks sub + LPR i (i < CPL, sub =
    l % LPR) of its C / EPC 16-byte chunks.  Every element of every row is read by exactly one
    thread, once; the lanes with sub = 0 write one sum slot per row of the step (slots 0 .. RPC-1,
    each once), and the per-row threads t < RPC read exactly those slots."""
    RPW = 32 // LPR
    RPC = 8 * RPW
    nch = C // EPC
    assert nch <= LPR * CPL  # the launcher's choice of LPR for this row length
    hits = np.zeros((rows, nch), dtype=np.int64)
    for b in range(grid):
        r0 = b * RPC
        while r0 < rows:
            slots = []
            for t in range(256):
                w, l = divmod(t, 32)
                sub, rr = l % LPR, l // LPR
                lrow = w * RPW + rr
                row = r0 + lrow
                if sub == 0:
                    slots.append(lrow)
                if row >= rows:
                    continue
                for i in range(CPL):
                    j = sub + LPR * i
                    if j < nch:
                        hits[row, j] += 1
            assert sorted(slots) == list(range(RPC))  # the slots the per-row threads t < RPC read
            r0 += grid * RPC
    assert (hits == 1).all()


@pytest.mark.parametrize("tiles_m,tiles_n", [(1, 1), (100, 6), (100, 3), (50, 8), (3, 200), (7, 152), (200, 1)])
def test_gemm_resident_weight_grid(tiles_m, tiles_n, sms=152):
    """The persistent GEMM with resident weights: tile t is (row block t / tiles_n, column block
    t % tiles_n) and CTA b takes the tiles b, b + grid, ...; the launcher makes the grid a multiple
    of tiles_n (per_n = clamp(sms / tiles_n, 1, tiles_m) CTAs per column block).  So every tile is
    computed once and each CTA only ever needs the one column block of W it keeps in shared memory;
    the column blocks' tiles are spread over their per_n CTAs within one tile of each other."""
    tiles = tiles_m * tiles_n
    per_n = min(max(sms // tiles_n, 1), tiles_m)
    grid = per_n * tiles_n
    seen = np.zeros(tiles, dtype=np.int64)
    for b in range(grid):
        mine = list(range(b, tiles, grid))
        seen[mine] += 1
        assert len({t % tiles_n for t in mine}) <= 1  # one resident column block per CTA
        assert tiles_m // per_n <= len(mine) <= -(-tiles_m // per_n)
    assert (seen == 1).all()


def test_layernorm_fast_normalisation_fits_int32():
    """I-LayerNorm's 32-bit normalisation: after at least one Newton step from 2^16 the iterate R is
    at least isqrt(V) >= |y| for every y = x - mu of the row, so F = floor((2^31 - 1) / R) gives
    |y F| < 2^31; the kernel then forms (y F) >> 1 as the wrapping 32-bit x F + mF (mF = -mu F mod
    2^32), and n + beta stays in int32 for |beta| <= 2^30.  Checked on random, constant and
    single-spike rows of int16 and int32 inputs for 1 to 20 Newton steps."""
    rng = np.random.default_rng(23)

    def newton(V, iters):
        r = 1 << 16
        for _ in range(iters):
            if r == 0:
                break
            r = (r + V // r) >> 1
        return max(r, 1)

    def wrap32(v):
        v &= 0xFFFFFFFF
        return v - (1 << 32) if v >= 1 << 31 else v

    rows = []
    for C in (1, 7, 64, 192, 384, 1024):
        for lim in (127, 32767, 1 << 24):
            rows.append(rng.integers(-lim, lim + 1, C))
            spike = np.zeros(C, dtype=np.int64)
            spike[0] = lim
            rows.append(spike)
            rows.append(np.full(C, -lim, dtype=np.int64))
    for x in rows:
        x = [int(t) for t in x]
        C = len(x)
        mu = (2 * sum(x) + C) // (2 * C)
        V = sum((t - mu) ** 2 for t in x)
        for iters in (1, 2, 3, 10, 20):
            R = newton(V, iters)
            assert R >= math.isqrt(V) >= max(abs(t - mu) for t in x)
            F = ((1 << 31) - 1) // R
            mF = wrap32(-mu * F)
            for t in x:
                y = t - mu
                assert abs(y * F) < 1 << 31
                n = (y * F) >> 1
                assert wrap32(wrap32(t * F) + mF) >> 1 == n
                assert -(1 << 31) <= n - (1 << 30) and n + (1 << 30) < 1 << 31
