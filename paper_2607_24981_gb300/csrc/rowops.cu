// rowops.cu -- bandwidth-bound integer nonlinearities: Constrained Shiftmax over rows
// (Algorithm 2), SD-ShiftGELU (Algorithm 1) and I-LayerNorm (Sec. 3.3).
//
// One warp owns one row; the row stays in registers between the two dependent reductions, so
// HBM sees each input byte once.  Rows are read with 128-bit loads when the layout allows.
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

// LANES lanes own one row (32 / LANES rows per warp); NCH = 4-element chunks per lane (row length
// <= 4 * LANES * NCH).  Vector loads need len % 4 == 0 and 16-byte aligned rows.  All NCH loads of a
// lane are issued before the first use, so each warp keeps 32 * NCH * 16 bytes in flight.
template <int NCH, int LANES, bool FASTQ>
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
        int32_t *e = (int32_t *)&v[j];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t a = min((uint32_t)mx - (uint32_t)e[q], 1u << 30);
            const uint32_t ex = shift_exp_mag_q<FASTQ>(a, c.se);
            e[q] = (int32_t)ex;
            if (ch < nch) sum += ex;
        }
    }
    sum = group_sum_u64<LANES>(sum);
    if (!live) return;
    const RowNorm rn = shiftmax_norm(sum, c.s_d, c.m_p, c.M_hw, c.k_out);
    uint32_t *pr = (uint32_t *)(P + row * ldp);
#pragma unroll
    for (int j = 0; j < NCH; ++j) {
        const int ch = sub + LANES * j;
        if (ch < nch) {
            const int32_t *e = (const int32_t *)&v[j];
            const uint32_t o = shiftmax_out((uint32_t)e[0], rn) | (shiftmax_out((uint32_t)e[1], rn) << 8) |
                               (shiftmax_out((uint32_t)e[2], rn) << 16) | (shiftmax_out((uint32_t)e[3], rn) << 24);
            __stcs(pr + ch, o);
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
// error < 2^-21, so absolute error < 2^5), one float refinement from the exact 64-bit remainder
// (error < 1 on a remainder below 2^6 r), and a final +-1 test on the remainder.
__device__ __forceinline__ uint32_t div_u48_u32(uint64_t V, uint32_t r) {
    const float rinv = __frcp_rn(__uint2float_rn(r));
    uint32_t q = __float2uint_rz(__ull2float_rn(V) * rinv);
    int64_t rem = (int64_t)V - (int64_t)q * r;
    const int32_t dq = __float2int_rd(__ll2float_rn(rem) * rinv);
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

// I-LayerNorm over tiles of LN_RB rows (Sec. 3.3; mean, variance, Newton's
// integer square root, F = floor((2^31 - 1) / R), n = (y F) >> 1, out = sat(rq(n + beta; m, s))):
//  (1) cp.async copies the tile into shared memory, rows padded by 16 bytes; the CTAs are
//      persistent and double-buffered, so the next tile streams in while one is processed;
//  (2) each warp sums slices of the columns of all the tile's rows, one row per lane (sum x, sum x^2 in
//      int64; the padded pitch keeps the lanes' 16-byte reads on distinct banks);
//  (3) warp 0 finishes the statistics, one row per lane: the Newton sequences of the tile run
//      side by side instead of once per warp;
//  (4) each thread owns 4 fixed columns (beta, m, s in registers) and normalises one 4-element
//      group of a row per pass, with coalesced stores.
// 32-bit arithmetic in (4) is exact: after at least one Newton step R >= isqrt(V) >= |y| for every
// y = x - mu of the row (a floored Newton step from any positive start lands at or above isqrt(V)),
// so |y F| <= |y| (2^31 - 1) / R < 2^31; with |beta| <= 2^30, n + beta fits int32 and for s >= 33 the
// requantisation takes the high-word form.  Rows or columns outside those conditions use the
// 64-bit formulas.

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

struct LnRowStat {
    int64_t mu, F;
    int32_t fast;
    int32_t mF;  // -mu * F in wrapping 32-bit arithmetic: (x F + mF) = (x - mu) F exactly when that fits int32
};

// The normalisation of 4 elements in 64-bit arithmetic, for tiles or columns outside the 32-bit
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

template <typename TIn>
__device__ __forceinline__ void ln_get4(const uint8_t *p, int32_t (&x)[4]) {
    if (sizeof(TIn) == 4) {
        const int4 v = *(const int4 *)p;
        x[0] = v.x; x[1] = v.y; x[2] = v.z; x[3] = v.w;
    } else {
        const uint2 v = *(const uint2 *)p;
        x[0] = (int32_t)(v.x << 16) >> 16; x[1] = (int32_t)v.x >> 16;
        x[2] = (int32_t)(v.y << 16) >> 16; x[3] = (int32_t)v.y >> 16;
    }
}

template <typename TIn, typename TOut, int LN_RB>
__global__ void __launch_bounds__(256) layernorm_tile(const LnParams p, int32_t pitch, int64_t ntiles) {
    extern __shared__ __align__(16) uint8_t ln_smem[];
    constexpr int EB = sizeof(TIn);
    const int C = p.C, nc16 = C * EB / 16, nc4 = C / 4;
    const int T = blockDim.x, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nwarps = T >> 5;  // full warps (T >= 128)
    constexpr int SPW = 32 / LN_RB;  // column slices per warp in (2): lane = slice * LN_RB + row
    const int nslice = nwarps * SPW;
    uint8_t *tiles = ln_smem;                                             // [2][LN_RB * pitch]
    int64_t *part = (int64_t *)(tiles + 2 * LN_RB * pitch);               // [nslice][LN_RB][2]
    LnRowStat *stat = (LnRowStat *)(part + 2 * LN_RB * nslice);          // [LN_RB]

    // (1) tile t -> shared buffer `buf` with cp.async (one commit group per tile)
    // T is a multiple of the 16-byte chunks per row (T = nc4 k and nc16 = nc4 EB / 4), so a thread
    // copies the same chunk column of rows r_c, r_c + T / nc16, ...
    const int ch_c = tid % nc16, r_c = tid / nc16, r_step = T / nc16;
    const int64_t ld_bytes = p.ldx * EB;
    const uint32_t tiles_s = (uint32_t)__cvta_generic_to_shared(tiles);
    auto issue = [&](int64_t t, int buf) {
        if (t < ntiles) {
            const int64_t r0 = t * LN_RB;
            const int nr = (int)min((int64_t)LN_RB, p.rows - r0);
            const uint8_t *src = (const uint8_t *)p.X + r0 * ld_bytes + ch_c * 16;
            const uint32_t dst0 = tiles_s + (uint32_t)(buf * LN_RB * pitch + ch_c * 16);
            const uint8_t *g = src + r_c * ld_bytes;
            const int64_t g_step = r_step * ld_bytes;
            uint32_t dst = dst0 + (uint32_t)(r_c * pitch);
            const uint32_t d_step = (uint32_t)(r_step * pitch);
            for (int r = r_c; r < LN_RB; r += r_step, g += g_step, dst += d_step) {
                const bool ok = r < nr;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(ok ? g : src),
                             "r"(ok ? 16 : 0)
                             : "memory");
            }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    int64_t t = blockIdx.x;
    issue(t, 0);
    // this thread's 4 columns and their parameters, fetched while the first copies are in flight
    const int cc = tid % nc4, rs = tid / nc4, kpass = T / nc4;
    int32_t be[4], mm[4], ss[4];
    {
        const int4 b4 = __ldg((const int4 *)(p.beta + 4 * cc)), m4 = __ldg((const int4 *)(p.mult + 4 * cc)),
                   s4 = __ldg((const int4 *)(p.shift + 4 * cc));
        be[0] = b4.x; be[1] = b4.y; be[2] = b4.z; be[3] = b4.w;
        mm[0] = m4.x; mm[1] = m4.y; mm[2] = m4.z; mm[3] = m4.w;
        ss[0] = s4.x; ss[1] = s4.y; ss[2] = s4.z; ss[3] = s4.w;
    }
    bool col_fast = true;
#pragma unroll
    for (int u = 0; u < 4; ++u) col_fast &= ss[u] >= 33 && be[u] >= -(1 << 30) && be[u] <= (1 << 30);
    int32_t rnd[4], sh[4];  // rq_hi constants of the 4 columns (used only when every shift is >= 33)
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        rnd[u] = col_fast ? 1 << (ss[u] - 33) : 0;
        sh[u] = ss[u] - 32;
    }
    // uniform over the CTA, so that (4) branches once per tile instead of predicating both forms
    const bool cols_fast = __syncthreads_and(col_fast) != 0;
    __shared__ int tile_fast;

    for (int buf = 0; t < ntiles; t += gridDim.x, buf ^= 1) {
        issue(t + gridDim.x, buf ^ 1);  // the next tile streams in while this one is processed
        asm volatile("cp.async.wait_group 1;" ::: "memory");
        __syncthreads();
        const uint8_t *tile = tiles + buf * LN_RB * pitch;
        const int64_t row0 = t * LN_RB;
        const int nrows = (int)min((int64_t)LN_RB, p.rows - row0);

        // (2) column slice `sl` of row `rr`
        {
            const int rr = lane % LN_RB, sl = warp * SPW + lane / LN_RB;
            const int per = (nc16 + nslice - 1) / nslice;
            const int c0 = sl * per, c1 = min(nc16, c0 + per);
            int64_t sx = 0, sq = 0;
            if (warp < nwarps) {
                const uint8_t *rp = tile + rr * pitch;
                for (int ch = c0; ch < c1; ++ch) {
                    const int4 v = *(const int4 *)(rp + ch * 16);
                    if (EB == 4) {
                        madw(sx, v.x, 1); madw(sx, v.y, 1); madw(sx, v.z, 1); madw(sx, v.w, 1);
                        madw(sq, v.x, v.x); madw(sq, v.y, v.y); madw(sq, v.z, v.z); madw(sq, v.w, v.w);
                    } else {
                        const uint32_t w[4] = {(uint32_t)v.x, (uint32_t)v.y, (uint32_t)v.z, (uint32_t)v.w};
                        int32_t s32 = 0;
#pragma unroll
                        for (int u = 0; u < 4; ++u) {
                            const int32_t lo = (int32_t)(w[u] << 16) >> 16, hi = (int32_t)w[u] >> 16;
                            s32 += lo + hi;
                            sq += (int64_t)((uint32_t)(lo * lo) + (uint32_t)(hi * hi));  // <= 2^31
                        }
                        sx += s32;
                    }
                }
                part[(sl * LN_RB + rr) * 2] = sx;
                part[(sl * LN_RB + rr) * 2 + 1] = sq;
            }
        }
        __syncthreads();

        // (3) statistics of row `lane`, Newton's iteration side by side for the tile's rows (lanes
        // past the tile's rows compute a dummy row)
        if (warp == 0) {
            const int lr = lane % LN_RB;
            int64_t S = 0, Q = 0;
            for (int w = 0; w < nslice; ++w) {
                S += part[(w * LN_RB + lr) * 2];
                Q += part[(w * LN_RB + lr) * 2 + 1];
            }
            const int64_t num = 2 * S + C, den = 2 * (int64_t)C;
            int64_t mu;
            if (num >= -(1ll << 31) && num < (1ll << 31)) {  // 32-bit floor division
                const int32_t n32 = (int32_t)num, d32 = (int32_t)den;
                const int32_t qt = n32 / d32;
                mu = qt - ((n32 % d32 != 0 && n32 < 0) ? 1 : 0);
            } else {
                mu = num / den;
                if ((num % den) != 0 && num < 0) mu -= 1;  // floor
            }
            const uint64_t V = (uint64_t)(Q - 2 * mu * S + (int64_t)C * mu * mu);
            const uint64_t R = V < (1ull << 48) ? newton_isqrt_fast(V, p.iters) : newton_isqrt_early(V, p.iters);
            LnRowStat st;
            st.mu = mu;
            st.F = R < (1ull << 32) ? (int64_t)div_int31((uint32_t)R) : 0;
            st.fast = (p.iters >= 1 || V < (1ull << 32)) ? 1 : 0;
            st.mF = (int32_t)(0u - (uint32_t)mu * (uint32_t)st.F);
            if (lane < LN_RB) stat[lane] = st;
            const bool all_fast = __all_sync(0xffffffffu, st.fast != 0);
            if (lane == 0) tile_fast = all_fast ? 1 : 0;
        }
        __syncthreads();

        // (4) normalise: rows rs, rs + kpass, ... of this thread's column group
        TOut *ybase = (TOut *)p.Y + row0 * p.ldy + 4 * cc;
        auto store = [&](int r, const int32_t (&o)[4]) { ln_store4<TOut>(ybase + (int64_t)r * p.ldy, o); };
        if (tile_fast && cols_fast) {
            // (x - mu) F = x F + mF in wrapping 32-bit arithmetic (the product fits int32), and
            // rq takes its high-word form with the rounding constant folded in
            for (int r = rs; r < nrows; r += kpass) {
                const int32_t F = (int32_t)stat[r].F, mF = stat[r].mF;
                int32_t x[4], o[4];
                ln_get4<TIn>(tile + r * pitch + cc * 4 * EB, x);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int32_t n = (int32_t)((uint32_t)x[u] * (uint32_t)F + (uint32_t)mF) >> 1;
                    const int32_t tq = rq_hi(n + be[u], mm[u], rnd[u], sh[u]);
                    o[u] = LnOut<TOut>::bits == 8 ? clamp8(tq) : clamp16(tq);
                }
                store(r, o);
            }
        } else {
            for (int r = rs; r < nrows; r += kpass) {
                int32_t x[4], o[4];
                ln_get4<TIn>(tile + r * pitch + cc * 4 * EB, x);
                ln_norm4_exact(x, stat[r].mu, stat[r].F, be, mm, ss, LnOut<TOut>::bits, o);
                store(r, o);
            }
        }
        __syncthreads();  // buffer `buf` and the statistics are free again
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
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
        constexpr int RB = 16;  // rows per tile
        const int nc4 = p.C / 4, T = nc4 * (256 / nc4);
        const int pitch = p.C * eb + 16;
        const size_t smem =
            (size_t)2 * RB * pitch + 2 * RB * (T / 32) * (32 / RB) * sizeof(int64_t) + RB * sizeof(LnRowStat);
        static std::once_flag once;
        static cudaError_t attr = cudaSuccess;
        std::call_once(once, [] {
            attr = cudaFuncSetAttribute(layernorm_tile<TIn, TOut, RB>, cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
        });
        if (attr != cudaSuccess) return attr;
        // persistent CTAs: as many as fit on the GPU at once, each striding over the tiles
        static thread_local int last_T = -1, last_per_sm = 0, sms = 0;
        static thread_local size_t last_smem = 0;
        if (T != last_T || smem != last_smem) {
            int dev = 0;
            cudaError_t e = cudaGetDevice(&dev);
            if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (e == cudaSuccess)
                e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&last_per_sm, layernorm_tile<TIn, TOut, RB>, T, smem);
            if (e != cudaSuccess) return e;
            last_T = T;
            last_smem = smem;
        }
        const int per_sm = last_per_sm;
        const int64_t ntiles = (p.rows + RB - 1) / RB;
        const int64_t grid = min(ntiles, (int64_t)max(per_sm, 1) * sms);
        layernorm_tile<TIn, TOut, RB><<<(unsigned)grid, T, smem, s>>>(p, pitch, ntiles);
        return cudaGetLastError();
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
#define ILW_SMX(NCH, LANES)                                                                                  \
    (fq ? (shiftmax_rows_vec<NCH, LANES, true><<<g(LANES), 256, 0, s>>>(X, ldx, rows, len, c, P, ldp), 0)   \
        : (shiftmax_rows_vec<NCH, LANES, false><<<g(LANES), 256, 0, s>>>(X, ldx, rows, len, c, P, ldp), 0))
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
            static bool attr = false;
            if (!attr) {
                cudaError_t e = cudaFuncSetAttribute(sdshiftgelu_table, cudaFuncAttributeMaxDynamicSharedMemorySize, 65536);
                if (e != cudaSuccess) return e;
                attr = true;
            }
            int dev = 0, sms = 148;
            cudaGetDevice(&dev);
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            int64_t blocks = (n4 + 255) / 256;
            if (blocks > 6 * sms) blocks = 6 * sms;
            sdshiftgelu_table<<<(unsigned)blocks, 256, smem, s>>>((const int4 *)X, (int4 *)Y, n4, c, T);
        } else if (n4) {
            int64_t blocks = (n4 + 255) / 256;
            if (blocks > 152 * 16) blocks = 152 * 16;
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
