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
};

// I_exp = ShiftExp(delta) for delta <= 0 with delta >= -2^30 (callers clamp below that: every
// such delta is already in the clamp region, where the result is the constant I0).
__device__ __forceinline__ uint32_t shift_exp(int32_t delta, const ShiftExpC &c) {
    int32_t Ie = delta + (delta >> 1) - (delta >> 4);  // I * log2(e) with shifts
    uint32_t n = (uint32_t)min(-Ie, c.kI0);            // -clamp_min(I_e, -k I0)
    uint32_t q = (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    uint32_t r = n - q * (uint32_t)c.I0;               // decimal part, in [0, I0)
    uint32_t Ib = (uint32_t)c.I0 - ((r + 1u) >> 1);    // ((-r) >> 1) + I0
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
__device__ __forceinline__ uint32_t shiftmax_out(uint32_t e, const RowNorm &rn) {
    return (uint32_t)(((uint64_t)e * rn.F) >> rn.sh);
}

// ---- SD-ShiftGELU sigmoid factor I_div (Algorithm 1), for |x| < 2^26 (callers clamp: beyond
// that both ShiftExp calls sit in their clamp regions and I_div no longer changes).
struct GeluC {
    ShiftExpC se;
    int32_t out_sh;  // 31 - k_out + 1
};
__device__ __forceinline__ int32_t gelu_idiv(int32_t x, const GeluC &c) {
    int32_t Ip = x + (x >> 1) + (x >> 3) + (x >> 4);  // 1.702 x
    int32_t Ish = max(Ip, 0);                          // ReLU(I_p)
    int32_t Id = Ip - Ish;                             // <= 0
    uint32_t E = shift_exp(Id, c.se);
    uint32_t E2 = shift_exp(-Ish, c.se);
    uint32_t F = kInt31Max / (E + E2);  // IntDiv: Algorithm 2's fixed-point division, s_d = 0
    return (int32_t)(((uint64_t)E * F) >> c.out_sh);
}

}  // namespace ilw
