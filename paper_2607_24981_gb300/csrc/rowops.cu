// rowops.cu -- bandwidth-bound integer nonlinearities: Constrained Shiftmax over rows
// (Algorithm 2), SD-ShiftGELU (Algorithm 1) and I-LayerNorm (Sec. 3.3).
//
// One warp owns one row; the row stays in registers between the two dependent reductions, so
// HBM sees each input byte once.  Rows are read with 128-bit loads when the layout allows.
#include <algorithm>
#include <climits>
#include <cstdint>
#include <mutex>

#include "ilw_kernels.h"

namespace ilw {
namespace {

__device__ __forceinline__ int32_t warp_max(int32_t v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ int64_t warp_sum_i64(int64_t v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// ------------------------------------------------------------------ Constrained Shiftmax rows
// NCH = 4-element chunks per lane (row length <= 128 * NCH); vector loads need len % 4 == 0
// and 16-byte aligned rows.
template <int LANES>
__device__ __forceinline__ int32_t group_max(int32_t v) {
#pragma unroll
    for (int o = LANES / 2; o; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o, LANES));
    return v;
}
template <int LANES>
__device__ __forceinline__ uint64_t group_sum_u64(uint64_t v) {
#pragma unroll
    for (int o = LANES / 2; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o, LANES);
    return v;
}

// The output floor(e F / 2^sh) as one high-word product: for sh <= 32 and F < 2^sh,
// F 2^(32 - sh) < 2^32 and floor(e F 2^(32 - sh) / 2^32) is the same floor; for sh > 32 the high word
// of e F shifted right by sh - 32 (floors compose).  `ok` is false for the rows neither form covers
// (sh < 32 with F >= 2^sh, i.e. a reduced denominator below 2^(31 - sh)), which take shiftmax_out.
struct RowOut {
    uint32_t Fs;
    uint32_t rs;
    bool ok;
};
__device__ __forceinline__ RowOut row_out(const RowNorm &rn) {
    RowOut o;
    if (rn.sh <= 32) {
        o.ok = rn.sh == 32 || (rn.F >> rn.sh) == 0;
        o.Fs = o.ok ? rn.F << (32 - rn.sh) : 0u;
        o.rs = 0;
    } else {
        o.ok = true;
        o.Fs = rn.F;
        o.rs = (uint32_t)min(rn.sh - 32, 31);
    }
    return o;
}

// LANES lanes own one row (32 / LANES rows per warp); NCH = 4-element chunks per lane (row length
// <= 4 * LANES * NCH).  Vector loads need len % 4 == 0 and 16-byte aligned rows.  All NCH loads of a
// lane are issued before the first use, so each warp keeps 32 * NCH * 16 bytes in flight.
// SUM4: I0 2^k < 2^30, so four ShiftExp values add up in 32 bits (two always do: I0 2^k < 2^31).
template <int NCH, int LANES, bool FASTQ, bool SUM4>
__global__ void __launch_bounds__(256) shiftmax_rows_vec(const int32_t *__restrict__ X, int64_t ldx,
                                                          int64_t rows, int32_t len, const ShiftmaxC c,
                                                          uint8_t *__restrict__ P, int64_t ldp) {
    constexpr int RPW = 32 / LANES;
    const int lane = threadIdx.x & 31, sub = lane % LANES;
    const int64_t row = ((int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5)) * RPW + lane / LANES;
    const bool live = row < rows;  // every lane stays for the shuffles
    const int nch = live ? (len >> 2) : 0;
    const int4 *xr = (const int4 *)(X + (live ? row : 0) * ldx);
    int4 v[NCH];
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
        const int ch = sub + LANES * j;
        v[j] = ch < nch ? __ldcs(xr + ch) : make_int4(INT_MIN, INT_MIN, INT_MIN, INT_MIN);
    }
    int32_t mx = INT_MIN;
#pragma unroll
    for (int j = 0; j < NCH; ++j) mx = max(mx, max(max(v[j].x, v[j].y), max(v[j].z, v[j].w)));
    mx = group_max<LANES>(mx);
    // a = mx - x >= 0 as an unsigned difference; magnitudes beyond 2^30 are deep in ShiftExp's
    // clamp region and are replaced by 2^30 (same value).  Padding lanes (INT_MIN) give a >= 2^30
    // and are not summed.
    uint64_t sum = 0;
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
        const int ch = sub + LANES * j;
        uint32_t *e = (uint32_t *)&v[j];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t a = min((uint32_t)mx - e[q], 1u << 30);
            e[q] = shift_exp_mag_q<FASTQ>(a, c.se);
        }
        if (ch < nch) {
            if constexpr (SUM4) sum += (uint64_t)(e[0] + e[1] + e[2] + e[3]);
            else sum += (uint64_t)(e[0] + e[1]) + (uint64_t)(e[2] + e[3]);
        }
    }
    sum = group_sum_u64<LANES>(sum);
    if (!live) return;
    const RowNorm rn = shiftmax_norm(sum, c.s_d, c.m_p, c.M_hw, c.k_out);
    const RowOut ro = row_out(rn);
    uint32_t *pr = (uint32_t *)(P + row * ldp);
    // every output is below 2^k_out <= 256: the four bytes of a chunk by two byte permutations
    if (ro.ok && ro.rs == 0) {  // sh <= 32: one high-word product per output
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int ch = sub + LANES * j;
            if (ch < nch) {
                const uint32_t *e = (const uint32_t *)&v[j];
                const uint32_t b01 = __byte_perm(__umulhi(e[0], ro.Fs), __umulhi(e[1], ro.Fs), 0x0040);
                const uint32_t b23 = __byte_perm(__umulhi(e[2], ro.Fs), __umulhi(e[3], ro.Fs), 0x0040);
                __stcs(pr + ch, __byte_perm(b01, b23, 0x5410));
            }
        }
    } else if (ro.ok) {
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int ch = sub + LANES * j;
            if (ch < nch) {
                const uint32_t *e = (const uint32_t *)&v[j];
                const uint32_t b01 = __byte_perm(__umulhi(e[0], ro.Fs) >> ro.rs, __umulhi(e[1], ro.Fs) >> ro.rs, 0x0040);
                const uint32_t b23 = __byte_perm(__umulhi(e[2], ro.Fs) >> ro.rs, __umulhi(e[3], ro.Fs) >> ro.rs, 0x0040);
                __stcs(pr + ch, __byte_perm(b01, b23, 0x5410));
            }
        }
    } else {
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int ch = sub + LANES * j;
            if (ch < nch) {
                const uint32_t *e = (const uint32_t *)&v[j];
                const uint32_t o = shiftmax_out(e[0], rn) | (shiftmax_out(e[1], rn) << 8) |
                                   (shiftmax_out(e[2], rn) << 16) | (shiftmax_out(e[3], rn) << 24);
                __stcs(pr + ch, o);
            }
        }
    }
}

// Any length / alignment: three passes over the row from global memory (L1/L2 resident).
__global__ void __launch_bounds__(256) shiftmax_rows_generic(const int32_t *__restrict__ X, int64_t ldx,
                                                              int64_t rows, int32_t len, const ShiftmaxC c,
                                                              uint8_t *__restrict__ P, int64_t ldp) {
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (row >= rows) return;
    const int32_t *x = X + row * ldx;
    int32_t mx = INT_MIN;
    for (int i = lane; i < len; i += 32) mx = max(mx, x[i]);
    mx = warp_max(mx);
    const int32_t lowb = mx > INT_MIN + (1 << 30) ? mx - (1 << 30) : INT_MIN;
    uint64_t sum = 0;
    for (int i = lane; i < len; i += 32) {
        uint32_t a = x[i] > lowb ? (uint32_t)(mx - x[i]) : (1u << 30);
        sum += shift_exp_mag(a, c.se);
    }
    sum = warp_sum_u64(sum);
    const RowNorm rn = shiftmax_norm(sum, c.s_d, c.m_p, c.M_hw, c.k_out);
    for (int i = lane; i < len; i += 32) {
        uint32_t a = x[i] > lowb ? (uint32_t)(mx - x[i]) : (1u << 30);
        P[row * ldp + i] = (uint8_t)shiftmax_out(shift_exp_mag(a, c.se), rn);
    }
}

// ------------------------------------------------------------------ SD-ShiftGELU
__device__ __forceinline__ int32_t gelu_one(int32_t x, const GeluC &c) {
    int32_t xc = min(max(x, -(1 << 26)), 1 << 26);  // I_div is constant beyond |x| = 2^19
    return x * gelu_idiv(xc, c);
}

__global__ void __launch_bounds__(256) sdshiftgelu_vec(const int4 *__restrict__ X, int4 *__restrict__ Y,
                                                        int64_t n4, const GeluC c) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
        int4 v = __ldcs(X + i);
        int4 o;
        o.x = gelu_one(v.x, c);
        o.y = gelu_one(v.y, c);
        o.z = gelu_one(v.z, c);
        o.w = gelu_one(v.w, c);
        __stcs(Y + i, o);
    }
}
// Table form: I_div depends on x alone and is constant for |x| >= T (both ShiftExp inputs are in
// their clamp regions there), so each CTA tabulates I_div(x) for x in [-T, T] with the same device
// function (exact by construction) and streams the data through lookups.
__global__ void __launch_bounds__(256) sdshiftgelu_table(const int4 *__restrict__ X, int4 *__restrict__ Y, int64_t n4,
                                                          const GeluC c, int32_t T) {
    extern __shared__ uint8_t tab[];
    for (int i = threadIdx.x; i <= 2 * T; i += blockDim.x) tab[i] = (uint8_t)gelu_idiv(i - T, c);
    __syncthreads();
    const uint8_t *t0 = tab + T;
    auto f = [&](int32_t x) { return x * (int32_t)t0[min(max(x, -T), T)]; };
    // 4 vectors per thread per step, all loaded before the first lookup (64 bytes in flight)
    constexpr int U = 4;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (; i + (U - 1) * stride < n4; i += U * stride) {
        int4 v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) v[u] = __ldcs(X + i + u * stride);
#pragma unroll
        for (int u = 0; u < U; ++u) __stcs(Y + i + u * stride, make_int4(f(v[u].x), f(v[u].y), f(v[u].z), f(v[u].w)));
    }
    for (; i < n4; i += stride) {
        const int4 v = __ldcs(X + i);
        __stcs(Y + i, make_int4(f(v.x), f(v.y), f(v.z), f(v.w)));
    }
}

__global__ void sdshiftgelu_tail(const int32_t *X, int32_t *Y, int64_t start, int64_t n, const GeluC c) {
    int64_t i = start + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) Y[i] = gelu_one(X[i], c);
}

// ------------------------------------------------------------------ I-LayerNorm
// Newton's integer square root r <- (r + V / r) >> 1 from r = 2^16, exactly `iters` steps (the loop
// stops at 0, which only V = 0 reaches), cut short once the rest of the sequence is known: a fixed
// point repeats forever, and once r_{i+1} = r_{i-1} the iterates alternate between two values, so
// r_iters is read off the parity of the steps left.  Identical result, fewer 64-bit divisions.
__device__ __noinline__ uint64_t newton_isqrt_early(uint64_t V, int iters) {
    uint64_t r = 1ull << 16, prev = ~0ull;
    for (int it = 0; it < iters; ++it) {
        if (r == 0) break;
        const uint64_t nx = (r + V / r) >> 1;
        if (nx == r) break;
        if (nx == prev) {
            r = ((iters - it - 1) & 1) ? r : nx;
            break;
        }
        prev = r;
        r = nx;
    }
    return r < 1 ? 1 : r;
}

// floor(V / r) for V < 2^48 and 1 <= r < 2^32 with a quotient below 2^26: a float estimate (relative
// error < 2^-20, so absolute error < 2^6), one float refinement from the exact 64-bit remainder
// (error < 1 on a remainder below 2^7 r), and a final +-1 test on the remainder.
// A 64-bit integer of magnitude below 2^62 as a float from its two 32-bit halves (two 32-bit
// conversions and one multiply-add: relative error below 2^-22), instead of a 64-bit conversion.
__device__ __forceinline__ float u64_to_float(uint64_t v) {
    return fmaf(__uint2float_rn((uint32_t)(v >> 32)), 4294967296.0f, __uint2float_rn((uint32_t)v));
}
__device__ __forceinline__ float i64_to_float(int64_t v) {
    return fmaf(__int2float_rn((int32_t)(v >> 32)), 4294967296.0f, __uint2float_rn((uint32_t)v));
}
__device__ __forceinline__ uint32_t div_u48_u32(uint64_t V, uint32_t r) {
    const float rinv = __frcp_rn(__uint2float_rn(r));
    uint32_t q = __float2uint_rz(u64_to_float(V) * rinv);
    int64_t rem = (int64_t)V - (int64_t)q * r;
    const int32_t dq = __float2int_rd(i64_to_float(rem) * rinv);
    q += dq;
    rem -= (int64_t)dq * r;
    if (rem < 0) --q;
    else if (rem >= (int64_t)r) ++q;
    return q;
}
// newton_isqrt_early for V < 2^48: the first step from 2^16 is a shift, and every later divisor r
// is at least isqrt(V) (a floored Newton step from any positive start lands at or above isqrt(V),
// and the iterates then decrease), so r < 2^32 and V / r < isqrt(V) + 3 < 2^25.
__device__ __forceinline__ uint64_t newton_isqrt_fast(uint64_t V, int iters) {
    if (iters <= 0) return 1ull << 16;
    uint64_t r = ((1ull << 16) + (V >> 16)) >> 1, prev = 1ull << 16;
    if (r == prev) return r;
    for (int it = 1; it < iters; ++it) {
        if (r == 0) break;
        const uint64_t nx = (r + div_u48_u32(V, (uint32_t)r)) >> 1;
        if (nx == r) break;
        if (nx == prev) {
            r = ((iters - it - 1) & 1) ? r : nx;
            break;
        }
        prev = r;
        r = nx;
    }
    return r < 1 ? 1 : r;
}

// Output element types of I-LayerNorm: int8, int16, or the int8 values carried in fp16.
template <typename TOut> struct LnOut { static constexpr int bits = 8 * (int)sizeof(TOut); };
template <> struct LnOut<__half> { static constexpr int bits = 8; };
// 4 outputs of one row, stored at y (4-element aligned)
template <typename TOut>
__device__ __forceinline__ void ln_store4(TOut *y, const int32_t (&o)[4]) {
    if constexpr (sizeof(TOut) == 1) {
        *(uint32_t *)y = (uint32_t)(uint8_t)o[0] | ((uint32_t)(uint8_t)o[1] << 8) | ((uint32_t)(uint8_t)o[2] << 16) |
                         ((uint32_t)(uint8_t)o[3] << 24);
    } else if constexpr (LnOut<TOut>::bits == 16) {
        *(uint2 *)y = make_uint2((uint32_t)(uint16_t)o[0] | ((uint32_t)(uint16_t)o[1] << 16),
                                 (uint32_t)(uint16_t)o[2] | ((uint32_t)(uint16_t)o[3] << 16));
    } else {
        // |v| <= 127: the fp16 bits of 1152 + v are 0x6480 + v; one half2 subtract of 1152 leaves v
        const __half2 k1152 = __half2half2(__ushort_as_half((unsigned short)0x6480));
        uint32_t w[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
            uint32_t x = (uint32_t)(0x6480 + o[2 * j]) | ((uint32_t)(0x6480 + o[2 * j + 1]) << 16);
            __half2 h = __hsub2(*reinterpret_cast<__half2 *>(&x), k1152);
            w[j] = *reinterpret_cast<uint32_t *>(&h);
        }
        *(uint2 *)y = make_uint2(w[0], w[1]);
    }
}

// acc += a * b with a 64-bit accumulator in one wide multiply-add
__device__ __forceinline__ void madw(int64_t &acc, int32_t a, int32_t b) {
    asm("mad.wide.s32 %0, %1, %2, %0;" : "+l"(acc) : "r"(a), "r"(b));
}

// The normalisation of 4 elements in 64-bit arithmetic, for rows or columns outside the 32-bit
// fast path's conditions (kept out of line so that its registers do not weigh on the fast path).
__device__ __noinline__ void ln_norm4_exact(const int32_t (&x)[4], int64_t mu, int64_t F, const int32_t (&be)[4],
                                            const int32_t (&mm)[4], const int32_t (&ss)[4], int out_bits,
                                            int32_t (&o)[4]) {
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const int64_t n = (((int64_t)x[u] - mu) * F) >> 1;
        const int64_t tq = rq(n + be[u], mm[u], ss[u]);
        o[u] = out_bits == 8 ? sat8(tq) : sat16(tq);
    }
}

// I-LayerNorm by row groups (Sec. 3.3; mean, variance, Newton's integer square root,
// F = floor((2^31 - 1) / R), n = (y F) >> 1, out = sat(rq(n + beta; m, s))).  LPR lanes own one row,
// 32 / LPR rows per warp, 256 / LPR rows per CTA and step (persistent grid).  A lane reads 16-byte
// chunks sub, sub + LPR, ... of its row (CPL at most; the LPR lanes of a row read adjacent chunks, so
// a warp's load covers 32 / LPR row segments of LPR * 16 bytes) and keeps them in registers, sums x
// and x^2 (int64), and the LPR lanes combine them with shuffles; the row's sums go to shared memory.
// The per-row scalar work (mean, variance, Newton, F) then runs once per row, one row per thread of
// the first 256 / LPR threads, instead of on every lane of the row: it is most of the instructions
// when each of the LPR lanes repeats it.  Every lane reads its row's mean and F back and normalises
// its own chunks with the per-column parameters from shared memory.
// 32-bit normalisation: after at least one Newton step R >= isqrt(V) >= |y| for every y = x - mu of
// the row (a floored Newton step from any positive start lands at or above isqrt(V)), so
// |y F| <= |y| (2^31 - 1) / R < 2^31 and y F fits int32; with one shift s >= 33 for every column and
// |beta| <= 2^30 the requantisation is the high-word form with a scalar rounding constant; otherwise
// (or for rows with iters = 0 and V >= 2^32) the 64-bit formulas run.
template <typename TIn, typename TOut, int LPR, int CPL>
__global__ void __launch_bounds__(256, 3) layernorm_rows(const LnParams p) {
    extern __shared__ __align__(16) int32_t ln_par[];  // beta[C], mult[C], shift[C]
    constexpr int EB = sizeof(TIn), EPC = 16 / EB;      // elements per 16-byte chunk
    constexpr int RPW = 32 / LPR;
    const int C = p.C, nch = C / EPC;
    int32_t *s_beta = ln_par, *s_mult = ln_par + C, *s_shift = ln_par + 2 * C;
    for (int i = threadIdx.x; i < C / 4; i += blockDim.x) {
        ((int4 *)s_beta)[i] = __ldg((const int4 *)p.beta + i);
        ((int4 *)s_mult)[i] = __ldg((const int4 *)p.mult + i);
        ((int4 *)s_shift)[i] = __ldg((const int4 *)p.shift + i);
    }
    __syncthreads();
    const int32_t uniform_shift = s_shift[0];  // the fast form needs one shift >= 33 for every column
    bool col_fast = true;
    for (int c = threadIdx.x; c < C; c += blockDim.x)
        col_fast &= s_beta[c] >= -(1 << 30) && s_beta[c] <= (1 << 30) && s_shift[c] == uniform_shift;
    const bool cols_fast = __syncthreads_and(col_fast) != 0 && uniform_shift >= 33;
    const int32_t rnd = cols_fast ? 1 << (uniform_shift - 33) : 0, sh = uniform_shift - 32;

    constexpr int RPC = 8 * RPW;  // rows per CTA and step (256 threads)
    __shared__ int64_t s_S[RPC], s_Q[RPC], s_mu[RPC], s_F[RPC];
    __shared__ int32_t s_ok[RPC];
    const int lane = threadIdx.x & 31, sub = lane % LPR, rr = lane / LPR;
    const int lrow = (threadIdx.x >> 5) * RPW + rr;  // the lane's row within the CTA's rows
    for (int64_t r0 = (int64_t)blockIdx.x * RPC; r0 < p.rows; r0 += (int64_t)gridDim.x * RPC) {
        const int64_t row = r0 + lrow;
        const bool live = row < p.rows;  // every lane stays for the shuffles and the barriers
        const uint8_t *xr = (const uint8_t *)p.X + (live ? row : 0) * p.ldx * EB;
        int4 v[CPL];
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
            const int j = sub + LPR * i;
            v[i] = (live && j < nch) ? __ldg((const int4 *)xr + j) : make_int4(0, 0, 0, 0);
        }
        // sum x and sum x^2 of the lane's chunks
        int64_t S = 0, Q = 0;
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
            if constexpr (EB == 2) {
                const uint32_t w[4] = {(uint32_t)v[i].x, (uint32_t)v[i].y, (uint32_t)v[i].z, (uint32_t)v[i].w};
                int32_t s32 = 0;
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int32_t lo = (int32_t)(w[u] << 16) >> 16, hi = (int32_t)w[u] >> 16;
                    s32 += lo + hi;
                    Q += (int64_t)((uint32_t)(lo * lo) + (uint32_t)(hi * hi));  // <= 2^31
                }
                S += s32;
            } else {
                const int32_t e[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    madw(S, e[u], 1);
                    madw(Q, e[u], e[u]);
                }
            }
        }
#pragma unroll
        for (int o = LPR / 2; o; o >>= 1) {
            S += __shfl_xor_sync(0xffffffffu, S, o, LPR);
            Q += __shfl_xor_sync(0xffffffffu, Q, o, LPR);
        }
        if (sub == 0) {
            s_S[lrow] = S;
            s_Q[lrow] = Q;
        }
        __syncthreads();
        if (threadIdx.x < RPC) {
            // one row per thread: mu = floor((2S + C) / (2C)); V = Q - 2 mu S + C mu^2 (= sum (x - mu)^2)
            const int64_t S1 = s_S[threadIdx.x], Q1 = s_Q[threadIdx.x];
            const int64_t num = 2 * S1 + C, den = 2 * (int64_t)C;
            int64_t mu;
            if (num >= -(1ll << 31) && num < (1ll << 31)) {
                const int32_t n32 = (int32_t)num, d32 = (int32_t)den;
                const int32_t qt = n32 / d32;
                mu = qt - ((n32 % d32 != 0 && n32 < 0) ? 1 : 0);
            } else {
                mu = num / den;
                if ((num % den) != 0 && num < 0) mu -= 1;
            }
            const uint64_t V = (uint64_t)(Q1 - 2 * mu * S1 + (int64_t)C * mu * mu);
            const uint64_t R = V < (1ull << 48) ? newton_isqrt_fast(V, p.iters) : newton_isqrt_early(V, p.iters);
            s_mu[threadIdx.x] = mu;
            s_F[threadIdx.x] = R < (1ull << 32) ? (int64_t)div_int31((uint32_t)R) : 0;
            s_ok[threadIdx.x] = p.iters >= 1 || V < (1ull << 32);
        }
        __syncthreads();
        const int64_t mu = s_mu[lrow], F = s_F[lrow];
        const bool fast = cols_fast && __all_sync(0xffffffffu, s_ok[lrow] != 0);
        const int32_t F32 = (int32_t)F, mF = (int32_t)(0u - (uint32_t)mu * (uint32_t)F);
        TOut *yr = (TOut *)p.Y + (live ? row : 0) * p.ldy;
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
            const int j = sub + LPR * i;
            if (!live || j >= nch) continue;
            int32_t x[EPC];
            if constexpr (EB == 2) {
                const uint32_t w[4] = {(uint32_t)v[i].x, (uint32_t)v[i].y, (uint32_t)v[i].z, (uint32_t)v[i].w};
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    x[2 * u] = (int32_t)(w[u] << 16) >> 16;
                    x[2 * u + 1] = (int32_t)w[u] >> 16;
                }
            } else {
                x[0] = v[i].x; x[1] = v[i].y; x[2] = v[i].z; x[3] = v[i].w;
            }
            const int c0 = j * EPC;
            int32_t o[EPC];
            if (fast) {
#pragma unroll
                for (int u4 = 0; u4 < EPC; u4 += 4) {
                    const int4 b4 = *(const int4 *)(s_beta + c0 + u4), m4 = *(const int4 *)(s_mult + c0 + u4);
                    const int32_t be[4] = {b4.x, b4.y, b4.z, b4.w}, mm[4] = {m4.x, m4.y, m4.z, m4.w};
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        // (x - mu) F = x F + mF in wrapping 32-bit arithmetic (the product fits int32)
                        const int32_t n = (int32_t)((uint32_t)x[u4 + u] * (uint32_t)F32 + (uint32_t)mF) >> 1;
                        const int32_t tq = rq_hi(n + be[u], mm[u], rnd, sh);
                        o[u4 + u] = LnOut<TOut>::bits == 8 ? clamp8(tq) : clamp16(tq);
                    }
                }
            } else {
#pragma unroll
                for (int u4 = 0; u4 < EPC; u4 += 4) {
                    int32_t xx[4], be[4], mm[4], ss[4], oo[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        xx[u] = x[u4 + u];
                        be[u] = s_beta[c0 + u4 + u];
                        mm[u] = s_mult[c0 + u4 + u];
                        ss[u] = s_shift[c0 + u4 + u];
                    }
                    ln_norm4_exact(xx, mu, F, be, mm, ss, LnOut<TOut>::bits, oo);
#pragma unroll
                    for (int u = 0; u < 4; ++u) o[u4 + u] = oo[u];
                }
            }
#pragma unroll
            for (int u4 = 0; u4 < EPC; u4 += 4) {
                const int32_t oo[4] = {o[u4], o[u4 + 1], o[u4 + 2], o[u4 + 3]};
                ln_store4<TOut>(yr + c0 + u4, oo);
            }
        }
    }
}

template <typename TIn, typename TOut, int EPL>
__global__ void __launch_bounds__(256) layernorm_kernel(const LnParams p) {
    const int lane = threadIdx.x & 31;
    const int64_t row = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    if (row >= p.rows) return;
    const TIn *x = (const TIn *)p.X + row * p.ldx;
    const int C = p.C;
    int32_t v[EPL];
    int64_t s = 0;
#pragma unroll
    for (int j = 0; j < EPL; ++j) {
        int c = lane + 32 * j;
        v[j] = c < C ? (int32_t)x[c] : 0;
        s += v[j];
    }
    s = warp_sum_i64(s);
    // mu = floor((2 sum + C) / (2C))
    const int64_t num = 2 * s + C, den = 2 * (int64_t)C;
    int64_t mu = num / den;
    if ((num % den) != 0 && num < 0) mu -= 1;
    uint64_t V = 0;
#pragma unroll
    for (int j = 0; j < EPL; ++j) {
        int c = lane + 32 * j;
        if (c < C) {
            int64_t y = (int64_t)v[j] - mu;
            V += (uint64_t)(y * y);
        }
    }
    V = warp_sum_u64(V);
    // Newton integer square root from 2^16, `iters` steps (stops at 0 only if V = 0)
    const uint64_t r = newton_isqrt_early(V, p.iters);
    const int64_t F = (int64_t)(0x7fffffffull / r);
    TOut *yo = (TOut *)p.Y + row * p.ldy;
#pragma unroll
    for (int j = 0; j < EPL; ++j) {
        int c = lane + 32 * j;
        if (c < C) {
            int64_t y = (int64_t)v[j] - mu;
            int64_t n = (y * F) >> 1;
            int64_t o = rq(n + p.beta[c], p.mult[c], p.shift[c]);
            const int32_t v = LnOut<TOut>::bits == 8 ? sat8(o) : sat16(o);
            if constexpr (sizeof(TOut) == 2 && LnOut<TOut>::bits == 8) yo[c] = __int2half_rn(v);
            else yo[c] = (TOut)v;
        }
    }
}

template <typename TIn, typename TOut>
cudaError_t ln_dispatch(const LnParams &p, cudaStream_t s) {
    const int eb = sizeof(TIn), ob = sizeof(TOut);
    const bool tiled = p.C % 4 == 0 && (p.C * eb) % 16 == 0 && (p.ldx * eb) % 16 == 0 && p.ldy % 4 == 0 &&
                       ((uintptr_t)p.X % 16) == 0 && ((uintptr_t)p.Y % (4 * ob)) == 0 &&
                       (((uintptr_t)p.beta | (uintptr_t)p.mult | (uintptr_t)p.shift) % 16) == 0 && p.C * eb <= 2048;
    if (tiled) {
        const int nch = p.C * eb / 16;
        const size_t smem = (size_t)3 * p.C * sizeof(int32_t);
        auto go = [&](auto kern, int lpr) -> cudaError_t {
            int dev = 0, sms = 0, per_sm = 0;
            cudaError_t e = cudaGetDevice(&dev);
            if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, 256, smem);
            if (e != cudaSuccess) return e;
            // persistent CTAs of 8 warps, each step of a CTA covering 256 / LPR rows
            const int64_t rpc = 256 / lpr;
            const int64_t grid = std::max<int64_t>(1, std::min<int64_t>((int64_t)std::max(per_sm, 1) * sms,
                                                                        (p.rows + rpc - 1) / rpc));
            kern<<<(unsigned)grid, 256, smem, s>>>(p);
            return cudaGetLastError();
        };
        // chunks per lane: 6 for int16 rows (8 values each), 12 for int32 rows (4 values each), so a
        // lane holds at most 48 values; lanes per row from the row's chunk count
        constexpr int CPL = sizeof(TIn) == 2 ? 6 : 12;
        if (nch <= 4 * CPL) return go(layernorm_rows<TIn, TOut, 4, CPL>, 4);
        if (nch <= 8 * CPL) return go(layernorm_rows<TIn, TOut, 8, CPL>, 8);
        if (nch <= 16 * CPL) return go(layernorm_rows<TIn, TOut, 16, CPL>, 16);
        if (nch <= 32 * CPL) return go(layernorm_rows<TIn, TOut, 32, CPL>, 32);
    }
    const int rows_per_block = 8;
    dim3 grid((unsigned)((p.rows + rows_per_block - 1) / rows_per_block));
    if (p.C <= 128) layernorm_kernel<TIn, TOut, 4><<<grid, 256, 0, s>>>(p);
    else if (p.C <= 256) layernorm_kernel<TIn, TOut, 8><<<grid, 256, 0, s>>>(p);
    else if (p.C <= 384) layernorm_kernel<TIn, TOut, 12><<<grid, 256, 0, s>>>(p);
    else if (p.C <= 512) layernorm_kernel<TIn, TOut, 16><<<grid, 256, 0, s>>>(p);
    else if (p.C <= 1024) layernorm_kernel<TIn, TOut, 32><<<grid, 256, 0, s>>>(p);
    else if (p.C <= 2048) layernorm_kernel<TIn, TOut, 64><<<grid, 256, 0, s>>>(p);
    else layernorm_kernel<TIn, TOut, 128><<<grid, 256, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_shiftmax_rows(const int32_t *X, int64_t ldx, int64_t rows, int32_t len,
                                 const ShiftmaxC &c, uint8_t *P, int64_t ldp, cudaStream_t s) {
    if (rows == 0 || len == 0) return cudaSuccess;
    dim3 grid((unsigned)((rows + 7) / 8));
    dim3 grid2((unsigned)((rows + 15) / 16));
    bool vec = (len % 4 == 0) && (ldx % 4 == 0) && (ldp % 4 == 0) && (((uintptr_t)X & 15) == 0) &&
               (((uintptr_t)P & 3) == 0);
    const bool fq = c.se.m32 != 0;
    // rows per CTA: 8 warps x (32 / LANES) rows
    auto g = [&](int lanes) { return dim3((unsigned)((rows + 8 * (32 / lanes) - 1) / (8 * (32 / lanes)))); };
    const bool s4 = ((int64_t)c.se.I0 << c.se.k) < ((int64_t)1 << 30);
#define ILW_SMX(NCH, LANES)                                                                                         \
    (fq ? (s4 ? (shiftmax_rows_vec<NCH, LANES, true, true><<<g(LANES), 256, 0, s>>>(X, ldx, rows, len, c, P, ldp), 0)  \
              : (shiftmax_rows_vec<NCH, LANES, true, false><<<g(LANES), 256, 0, s>>>(X, ldx, rows, len, c, P, ldp), 0)) \
        : (s4 ? (shiftmax_rows_vec<NCH, LANES, false, true><<<g(LANES), 256, 0, s>>>(X, ldx, rows, len, c, P, ldp), 0) \
              : (shiftmax_rows_vec<NCH, LANES, false, false><<<g(LANES), 256, 0, s>>>(X, ldx, rows, len, c, P, ldp), 0)))
    if (vec && len <= 64) ILW_SMX(4, 4);
    else if (vec && len <= 128) ILW_SMX(4, 8);
    else if (vec && len <= 416) ILW_SMX(13, 8);
    else if (vec && len <= 1024) ILW_SMX(8, 32);
    else if (vec && len <= 1664) ILW_SMX(13, 32);
    else if (vec && len <= 2048) ILW_SMX(16, 32);
#undef ILW_SMX
    else shiftmax_rows_generic<<<grid, 256, 0, s>>>(X, ldx, rows, len, c, P, ldp);
    return cudaGetLastError();
}

cudaError_t launch_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, const GeluC &c, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    int64_t n4 = 0;
    // the clamp threshold of both ShiftExp inputs: |x| >= ((k I0 + 1)/1.4375 + 3)/1.6875 (< T)
    const double bound = 0.7 * ((double)c.se.kI0 + 1.0) + 8.0;
    if ((((uintptr_t)X | (uintptr_t)Y) & 15) == 0) {
        n4 = n / 4;
        if (n4 && bound <= 32767.0 && n4 >= (1 << 16)) {
            const int32_t T = (int32_t)bound;
            const int smem = 2 * T + 1;
            static SmemLimit limit;
            const cudaError_t e = raise_smem_limit(limit, (const void *)sdshiftgelu_table, 65536);
            if (e != cudaSuccess) return e;
            int64_t blocks = (n4 + 255) / 256;
            if (blocks > 6 * (int64_t)sm_count()) blocks = 6 * (int64_t)sm_count();
            sdshiftgelu_table<<<(unsigned)blocks, 256, smem, s>>>((const int4 *)X, (int4 *)Y, n4, c, T);
        } else if (n4) {
            int64_t blocks = (n4 + 255) / 256;
            if (blocks > 16 * (int64_t)sm_count()) blocks = 16 * (int64_t)sm_count();
            sdshiftgelu_vec<<<(unsigned)blocks, 256, 0, s>>>((const int4 *)X, (int4 *)Y, n4, c);
        }
    }
    int64_t start = n4 * 4;
    if (start < n) sdshiftgelu_tail<<<(unsigned)((n - start + 255) / 256), 256, 0, s>>>(X, Y, start, n, c);
    return cudaGetLastError();
}

cudaError_t launch_layernorm(const LnParams &p, cudaStream_t s) {
    if (p.rows == 0) return cudaSuccess;
    if (p.out_bits == kOutI8InF16)
        return p.in_bits == 16 ? ln_dispatch<int16_t, __half>(p, s) : ln_dispatch<int32_t, __half>(p, s);
    if (p.in_bits == 16 && p.out_bits == 8) return ln_dispatch<int16_t, int8_t>(p, s);
    if (p.in_bits == 16 && p.out_bits == 16) return ln_dispatch<int16_t, int16_t>(p, s);
    if (p.in_bits == 32 && p.out_bits == 8) return ln_dispatch<int32_t, int8_t>(p, s);
    return ln_dispatch<int32_t, int16_t>(p, s);
}

}  // namespace ilw
