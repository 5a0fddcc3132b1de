// ilw_device.cuh -- device-side integer building blocks of the I-LW-DETR path (sm_103a).
//
// All helpers are exact integer arithmetic; each cites the operator it implements.
#pragma once
#include <cstdint>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "ilwdetr.h"

namespace ilw {

constexpr uint32_t kInt31Max = 0x7fffffffu;

// ---- dyadic requantisation and symmetric saturation (Sec. 3.2.1, 3.2.2)
// rq(v; m, s) = (v*m + 2^(s-1)) >> s, arithmetic shift; the callers keep |v*m| < 2^62.
__device__ __forceinline__ int64_t rq(int64_t v, int32_t m, int32_t s) {
    return (v * (int64_t)m + ((int64_t)1 << (s - 1))) >> s;
}
__device__ __forceinline__ int32_t sat8(int64_t v) { return (int32_t)(v < -127 ? -127 : (v > 127 ? 127 : v)); }
__device__ __forceinline__ int32_t sat16(int64_t v) {
    return (int32_t)(v < -32767 ? -32767 : (v > 32767 ? 32767 : v));
}
__device__ __forceinline__ int32_t clamp8(int32_t v) { return max(-127, min(127, v)); }
__device__ __forceinline__ int32_t clamp16(int32_t v) { return max(-32767, min(32767, v)); }

// rq(v; m, s) for int32 v and s >= 33, given sh1 = s - 33.  With v m = H 2^32 + L (0 <= L < 2^32),
// L / 2^32 < 1 added to an integer numerator never changes floor(. / 2^(s-32)), so
// rq = floor((H + 2^(s-33)) / 2^(s-32)); and floor((h + 2^(k-1)) / 2^k) = (floor(h / 2^(k-1)) + 1) >> 1
// for k >= 1, which needs no rounding constant.  |result| < 2^29.
__device__ __forceinline__ int32_t rq_hi1(int32_t v, int32_t m, int32_t sh1) {
    return ((__mulhi(v, m) >> sh1) + 1) >> 1;
}
// The same rq with the rounding folded into the multiply: rq = (h + 2^(s-33)) >> (s-32), where
// h + 2^(s-33) is one mad.hi (high word of v m plus a constant; |h| <= 2^30, so no overflow).
// rnd = 2^(s-33) and sh = s - 32 are precomputed by the caller (s >= 33).
__device__ __forceinline__ int32_t rq_hi(int32_t v, int32_t m, int32_t rnd, int32_t sh) {
    int32_t h;
    asm("mad.hi.s32 %0, %1, %2, %3;" : "=r"(h) : "r"(v), "r"(m), "r"(rnd));
    return h >> sh;
}

// ---- ShiftExp (Algorithm 1) with per-launch constants.
// The integer part q = floor(n / I0) of n = -I_e in [0, k I0] is taken with the round-up
// reciprocal method of Granlund & Montgomery (1994), "Division by invariant integers using
// multiplication": M = ceil(2^40 / I0), q = floor(n M / 2^40), exact while n * I0 < 2^40
// (n <= k I0 < 2^20 and I0 < 2^15 here).  n M / 2^32 is formed as umulhi(n, M_lo) + n M_hi.
struct ShiftExpC {
    int32_t I0;
    int32_t kI0;    // k_inter * I0: the clamp bound of -I_e
    uint32_t m_lo;  // low 32 bits of M
    uint32_t m_hi;  // high bits of M (M <= 2^40)
    int32_t k;      // k_inter
    uint32_t m32;   // ceil(2^32 / I0) when k I0^2 < 2^32 (then floor(n / I0) = umulhi(n, m32) for
                    // every n <= k I0), else 0
};

// Arithmetic (flooring) right shift of a signed value.
__device__ __forceinline__ int32_t asr(int32_t v, int32_t s) {
    int32_t r;
    asm("shr.s32 %0, %1, %2;" : "=r"(r) : "r"(v), "r"(s));
    return r;
}

// I_exp = ShiftExp(-a) for a magnitude a = -I >= 0 with a <= 2^30 (callers clamp above that:
// every such input is already in the clamp region, where the result is the constant I0).
// Algorithm 1's I_e = I + (I >> 1) - (I >> 4) floors negative values; with I = -a,
// floor(-a/2) = -((a+1) >> 1) and floor(-a/16) = -((a+15) >> 4), so
//   -I_e = a + ((a+1) >> 1) - ((a+15) >> 4)
// exactly, and every shift here acts on a non-negative value.  (A device probe of the direct form,
// (-|x|) >> 4 with the operand's sign known to the compiler, returned truncated rather than floored
// results; the cause was not pursued, and the magnitude form does not depend on it.)
__device__ __forceinline__ uint32_t shift_exp_mag(uint32_t a, const ShiftExpC &c) {
    uint32_t n = a + ((a + 1u) >> 1) - ((a + 15u) >> 4);  // -I_e (I * log2 e with shifts)
    n = min(n, (uint32_t)c.kI0);                            // -clamp_min(I_e, -k I0)
    uint32_t q = (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    uint32_t r = n - q * (uint32_t)c.I0;               // decimal part, in [0, I0)
    uint32_t Ib = (uint32_t)c.I0 - ((r + 1u) >> 1);    // ((-r) >> 1) + I0
    return Ib << (c.k - (int32_t)q);
}

// shift_exp_mag with the single-multiply quotient (FASTQ: c.m32 set) and I0 - ceil(r/2) written as
// ((q + 2) I0 - n) / 2 (r = n - q I0): the same value in fewer operations.
template <bool FASTQ>
__device__ __forceinline__ uint32_t shift_exp_mag_q(uint32_t a, const ShiftExpC &c) {
    uint32_t n = a + ((a + 1u) >> 1) - ((a + 15u) >> 4);
    n = min(n, (uint32_t)c.kI0);
    const uint32_t q = FASTQ ? __umulhi(n, c.m32) : (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    const uint32_t Ib = ((q + 2u) * (uint32_t)c.I0 - n) >> 1;
    return Ib << (c.k - (int32_t)q);
}

// The same ShiftExp of the magnitude a = max - s, taken from b = bits of the fp32 value
// (max + 2^23) - s.  For integer scores with 0 <= a < 2^23 that value is exact and b = 0x4B000000 + a.
// Because 0x4B000000 is a multiple of 16, ceil(b/2) and ceil(b/16) are ceil(a/2) and ceil(a/16) plus
// fixed constants, so n = a + ceil(a/2) - ceil(a/16) is read off b with the constants folded into one
// (1.4375 * 0x4B000000 = 1808793600).  The quotient uses the single-multiply reciprocal when c.m32 is
// set (FASTQ), and I0 - ceil(r/2) is written as ((q + 2) I0 - n) / 2 (r = n - q I0, floored).
template <bool FASTQ>
__device__ __forceinline__ uint32_t shift_exp_bits(uint32_t b, const ShiftExpC &c) {
    uint32_t n = b + ((b + 1u) >> 1) - ((b + 15u) >> 4) - 1808793600u;
    n = min(n, (uint32_t)c.kI0);
    const uint32_t q = FASTQ ? __umulhi(n, c.m32) : (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    const uint32_t Ib = ((q + 2u) * (uint32_t)c.I0 - n) >> 1;
    return Ib << (c.k - (int32_t)q);
}

// The same ShiftExp of the magnitude a = max - s, taken from w = bits of the fp32 value s - C with
// C = 2^23 + max + 1 (the attention kernel's score MMA adds -C to q.k directly).  For integer scores
// with 0 <= a < 2^23 - 1 that value is -(2^23 + a + 1), exact, so w = 0xCB000000 + a + 1.  Both
// 0xCB000000 terms are multiples of 16, so w >> 1 and (w + 14) >> 4 are ceil(a/2) and ceil(a/16)
// plus fixed constants, and with 32-bit wrap-around n = a + ceil(a/2) - ceil(a/16) is
// w + (w >> 1) - ((w + 14) >> 4) - 0x23D00001.
__device__ __forceinline__ uint32_t exp_arg_from_neg_bits(uint32_t w) {
    return w + (w >> 1) - ((w + 14u) >> 4) - 0x23D00001u;
}
template <bool FASTQ>
__device__ __forceinline__ uint32_t shift_exp_nbits(uint32_t w, const ShiftExpC &c) {
    uint32_t n = exp_arg_from_neg_bits(w);
    n = min(n, (uint32_t)c.kI0);
    const uint32_t q = FASTQ ? __umulhi(n, c.m32) : (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    const uint32_t Ib = ((q + 2u) * (uint32_t)c.I0 - n) >> 1;
    return Ib << (c.k - (int32_t)q);
}

// ---- Constrained Shiftmax row constants (Algorithm 2): from S_sum to (F, output shift).
struct RowNorm {
    uint32_t F;
    int32_t sh;  // 31 - k_out + 1 + s_d
};
__device__ __forceinline__ RowNorm shiftmax_norm(uint64_t S_sum, int32_t s_d_static, int32_t m_p,
                                                 int32_t M_hw, int32_t k_out) {
    int32_t s_d = s_d_static;
    if (s_d < 0) {  // CalibrateShift: max(ceil(log2 S_sum) + m_p - M_hw, 0)
        int32_t M_req = 64 - __clzll((long long)(S_sum - 1ull));  // ceil(log2 S) for S >= 1
        s_d = max(M_req + m_p - M_hw, 0);
    }
    uint64_t S_R = S_sum >> s_d;  // = sum Q_i + (sum r_i >> s_d), the exact shifted denominator
    S_R = S_R < 1ull ? 1ull : (S_R > (uint64_t)kInt31Max ? (uint64_t)kInt31Max : S_R);
    RowNorm rn;
    rn.F = kInt31Max / (uint32_t)S_R;
    rn.sh = 31 - k_out + 1 + s_d;
    return rn;
}
// (e * F) >> sh for e, F < 2^31 and sh >= 24 (k_out <= 8): from the 32-bit halves of the
// product, so no 64-bit shift is needed (e * F < 2^62, so any sh >= 63 gives 0).
__device__ __forceinline__ uint32_t shiftmax_out(uint32_t e, const RowNorm &rn) {
    const uint32_t lo = e * rn.F, hi = __umulhi(e, rn.F);
    return rn.sh < 32 ? __funnelshift_r(lo, hi, rn.sh) : (hi >> min(rn.sh - 32, 31));
}

// ---- SD-ShiftGELU sigmoid factor I_div (Algorithm 1), for |x| < 2^26 (callers clamp: beyond
// that both ShiftExp calls sit in their clamp regions and I_div no longer changes).
struct GeluC {
    ShiftExpC se;
    int32_t out_sh;  // 31 - k_out + 1
};
// floor((2^31 - 1) / den) for den >= 1, exact.  For den >= 2^16 the quotient is < 2^15 and a
// float estimate (relative error < 2^-21, so absolute error < 2^-6) rounded to the nearest
// integer is q or q + 1; one integer remainder test corrects it.  Smaller denominators use the
// integer divide.
__device__ __forceinline__ uint32_t div_int31(uint32_t den) {
    if (den < 65536u) return kInt31Max / den;
    uint32_t q = __float2uint_rn(__fdividef(2147483647.0f, __uint2float_rn(den)));
    const int64_t r = (int64_t)kInt31Max - (int64_t)q * den;
    if (r < 0) --q;
    else if (r >= (int64_t)den) ++q;
    return q;
}

// With I_shift = ReLU(I_p) and I_delta = I_p - I_shift, one of the two ShiftExp inputs is always
// 0, and ShiftExp(0) = I0 * 2^k exactly; so a single ShiftExp of -|I_p| gives both E and E'.
__device__ __forceinline__ int32_t gelu_idiv(int32_t x, const GeluC &c) {
    int32_t Ip = x + asr(x, 1) + asr(x, 3) + asr(x, 4);  // 1.702 x
    uint32_t e = shift_exp_mag((uint32_t)abs(Ip), c.se);   // ShiftExp(I_delta) or ShiftExp(-I_shift)
    uint32_t top = (uint32_t)c.se.I0 << c.se.k;         // ShiftExp(0)
    uint32_t E = Ip >= 0 ? top : e;                    // numerator: ShiftExp(I_delta)
    uint32_t F = div_int31(top + e);  // IntDiv: Algorithm 2's fixed-point division, s_d = 0
    return (int32_t)(((uint64_t)E * F) >> c.out_sh);
}

}  // namespace ilw
