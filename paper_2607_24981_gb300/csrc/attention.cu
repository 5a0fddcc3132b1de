// attention.cu -- fused integer attention: scores = q k^T, Constrained Shiftmax (Algorithm 2),
// O = P V, requantisation (Sec. 3.2.1, 3.3.2).
//
// ShiftExp floors its input, so the online rescaling of flash attention is not exact: the row
// maximum must be known before any exponential.  Each CTA therefore streams the keys of its
// attention group three times (they stay in L2): pass 1 takes the exact row max, pass 2 sums
// ShiftExp (int64), which fixes s_d and F, pass 3 forms P (u8) and accumulates P V.
// Scores and P V run on the int8 tensor-core MMA (m16n8k32, s8.s8 and u8.s8 -> s32), exact.
//
// P V reuses the score fragments as the A operand without shuffles: the MMA's k order is
// permuted (k-slot 4t + {0,1,2,3} <-> key 2t + {0,1,8,9} within each 16-key half), and V is
// transposed into shared memory with the same permutation.
#include <climits>
#include <cstdint>

#include "ilw_kernels.h"

namespace ilw {
namespace {

constexpr int QT = 64;   // query rows per CTA (4 warps x 16)
constexpr int KB = 64;   // keys per block
constexpr int THREADS = 128;

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem, bool valid) {
    uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
    int n = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::); }

__device__ __forceinline__ void mma_s8s8(int32_t (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_u8s8(int32_t (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.u8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

struct Group {
    int64_t base;  // b * T
    int32_t Tg;
    int32_t nw, ws, gs, wy, wx;
    __device__ __forceinline__ int64_t token(int32_t t) const {
        if (nw <= 1) return base + t;
        return base + (int64_t)(wy * ws + t / ws) * gs + wx * ws + t % ws;
    }
};

template <int DH>
__global__ void __launch_bounds__(THREADS) attn_kernel(const AttnParams p) {
    constexpr int LDK = DH + 16;  // padded q/k/v smem row (bytes)
    constexpr int LDV = KB + 16;  // padded transposed-V row (bytes)
    constexpr int KS = DH / 32;   // k32 steps of q k^T
    constexpr int NT = DH / 8;    // n-tiles of P V
    __shared__ __align__(16) int8_t Qs[QT * LDK];
    __shared__ __align__(16) int8_t Ks[KB * LDK];
    __shared__ __align__(16) int8_t Vr[KB * LDK];
    __shared__ __align__(16) int8_t Vt[DH * LDV];

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t = lane & 3;
    const int h = blockIdx.y;
    Group gr;
    {
        const int G2 = p.nw * p.nw;
        const int z = blockIdx.z;
        const int b = z / G2, w = z % G2;
        gr.base = (int64_t)b * p.T;
        gr.nw = p.nw;
        gr.gs = p.grid_side;
        gr.ws = p.nw > 1 ? p.grid_side / p.nw : 0;
        gr.wy = w / (p.nw > 0 ? p.nw : 1);
        gr.wx = w % (p.nw > 0 ? p.nw : 1);
        gr.Tg = p.nw > 1 ? gr.ws * gr.ws : p.T;
    }
    const int Tg = gr.Tg;
    const int q0 = blockIdx.x * QT;
    const int hoff = h * DH;

    // ---- Q tile -> registers (A fragments of the score MMA)
    for (int c = tid; c < QT * (DH / 16); c += THREADS) {
        int r = c / (DH / 16), kc = (c % (DH / 16)) * 16;
        bool v = (q0 + r) < Tg;
        const int8_t *src = v ? p.Q + gr.token(q0 + r) * p.ld_qkv + hoff + kc : p.Q;
        cp_async16(Qs + r * LDK + kc, src, v);
    }
    cp_async_commit();
    cp_async_wait_all();
    __syncthreads();
    uint32_t qa[KS][4];
#pragma unroll
    for (int ks = 0; ks < KS; ++ks) {
        const int8_t *q = Qs + (warp * 16 + g) * LDK + ks * 32 + 4 * t;
        qa[ks][0] = *(const uint32_t *)(q);
        qa[ks][1] = *(const uint32_t *)(q + 8 * LDK);
        qa[ks][2] = *(const uint32_t *)(q + 16);
        qa[ks][3] = *(const uint32_t *)(q + 8 * LDK + 16);
    }

    const int nkb = (Tg + KB - 1) / KB;
    auto load_k = [&](int kb) {
        for (int c = tid; c < KB * (DH / 16); c += THREADS) {
            int r = c / (DH / 16), kc = (c % (DH / 16)) * 16;
            int key = kb * KB + r;
            bool v = key < Tg;
            const int8_t *src = v ? p.K + gr.token(key) * p.ld_qkv + hoff + kc : p.K;
            cp_async16(Ks + r * LDK + kc, src, v);
        }
    };
    auto load_v = [&](int kb) {
        for (int c = tid; c < KB * (DH / 16); c += THREADS) {
            int r = c / (DH / 16), kc = (c % (DH / 16)) * 16;
            int key = kb * KB + r;
            bool v = key < Tg;
            const int8_t *src = v ? p.V + gr.token(key) * p.ld_qkv + hoff + kc : p.V;
            cp_async16(Vr + r * LDK + kc, src, v);
        }
    };
    // scores of this warp's 16 rows x the 64 keys of the block in Ks
    auto scores = [&](int32_t (&S)[8][4]) {
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            S[nt][0] = S[nt][1] = S[nt][2] = S[nt][3] = 0;
#pragma unroll
            for (int ks = 0; ks < KS; ++ks) {
                const int8_t *k = Ks + (nt * 8 + g) * LDK + ks * 32 + 4 * t;
                mma_s8s8(S[nt], qa[ks], *(const uint32_t *)k, *(const uint32_t *)(k + 16));
            }
        }
    };

    // ---- pass 1: exact row maxima
    int32_t mx0 = INT_MIN, mx1 = INT_MIN;
    for (int kb = 0; kb < nkb; ++kb) {
        load_k(kb);
        cp_async_commit();
        cp_async_wait_all();
        __syncthreads();
        int32_t S[8][4];
        scores(S);
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            int key = kb * KB + nt * 8 + 2 * t;
            if (key < Tg) { mx0 = max(mx0, S[nt][0]); mx1 = max(mx1, S[nt][2]); }
            if (key + 1 < Tg) { mx0 = max(mx0, S[nt][1]); mx1 = max(mx1, S[nt][3]); }
        }
        __syncthreads();
    }
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = max(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = max(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));

    // ---- pass 2: S_sum = sum ShiftExp(s - max) (|scores| <= dh 127^2 < 2^20: no clamp needed)
    const ShiftExpC se = p.smx.se;
    uint64_t sum0 = 0, sum1 = 0;
    for (int kb = 0; kb < nkb; ++kb) {
        load_k(kb);
        cp_async_commit();
        cp_async_wait_all();
        __syncthreads();
        int32_t S[8][4];
        scores(S);
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            int key = kb * KB + nt * 8 + 2 * t;
            if (key < Tg) {
                sum0 += shift_exp_mag((uint32_t)(mx0 - S[nt][0]), se);
                sum1 += shift_exp_mag((uint32_t)(mx1 - S[nt][2]), se);
            }
            if (key + 1 < Tg) {
                sum0 += shift_exp_mag((uint32_t)(mx0 - S[nt][1]), se);
                sum1 += shift_exp_mag((uint32_t)(mx1 - S[nt][3]), se);
            }
        }
        __syncthreads();
    }
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 1);
    sum0 += __shfl_xor_sync(0xffffffffu, sum0, 2);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 1);
    sum1 += __shfl_xor_sync(0xffffffffu, sum1, 2);
    // rows past Tg have sum 0: give them a harmless normaliser (their outputs are not stored)
    const RowNorm rn0 = shiftmax_norm(sum0 ? sum0 : 1, p.smx.s_d, p.smx.m_p, p.smx.M_hw, p.smx.k_out);
    const RowNorm rn1 = shiftmax_norm(sum1 ? sum1 : 1, p.smx.s_d, p.smx.m_p, p.smx.M_hw, p.smx.k_out);

    // ---- pass 3: P = (I_exp F) >> sh, O += P V
    int32_t o[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0;
    for (int kb = 0; kb < nkb; ++kb) {
        load_k(kb);
        load_v(kb);
        cp_async_commit();
        cp_async_wait_all();
        __syncthreads();
        // transpose V into Vt[dim][slot] with the k-slot permutation of the P fragments
        for (int m = tid; m < 16 * (DH / 4); m += THREADS) {
            int kg = m & 15, dq = m >> 4;
            int ch = kg >> 3, half = (kg >> 2) & 1, tt = kg & 3;
            int k0 = ch * 32 + half * 16 + 2 * tt;
            uint32_t w0 = *(const uint32_t *)(Vr + (k0 + 0) * LDK + 4 * dq);
            uint32_t w1 = *(const uint32_t *)(Vr + (k0 + 1) * LDK + 4 * dq);
            uint32_t w2 = *(const uint32_t *)(Vr + (k0 + 8) * LDK + 4 * dq);
            uint32_t w3 = *(const uint32_t *)(Vr + (k0 + 9) * LDK + 4 * dq);
            uint32_t t0 = __byte_perm(w0, w1, 0x5140), t1 = __byte_perm(w2, w3, 0x5140);
            uint32_t t2 = __byte_perm(w0, w1, 0x7362), t3 = __byte_perm(w2, w3, 0x7362);
            int sw = ch * 8 + half * 4 + tt;
            *(uint32_t *)(Vt + (4 * dq + 0) * LDV + 4 * sw) = __byte_perm(t0, t1, 0x5410);
            *(uint32_t *)(Vt + (4 * dq + 1) * LDV + 4 * sw) = __byte_perm(t0, t1, 0x7632);
            *(uint32_t *)(Vt + (4 * dq + 2) * LDV + 4 * sw) = __byte_perm(t2, t3, 0x5410);
            *(uint32_t *)(Vt + (4 * dq + 3) * LDV + 4 * sw) = __byte_perm(t2, t3, 0x7632);
        }
        __syncthreads();
        int32_t S[8][4];
        scores(S);
        uint32_t pv[8][4];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            int key = kb * KB + nt * 8 + 2 * t;
            bool v0 = key < Tg, v1 = key + 1 < Tg;
            pv[nt][0] = v0 ? shiftmax_out(shift_exp_mag((uint32_t)(mx0 - S[nt][0]), se), rn0) : 0u;
            pv[nt][1] = v1 ? shiftmax_out(shift_exp_mag((uint32_t)(mx0 - S[nt][1]), se), rn0) : 0u;
            pv[nt][2] = v0 ? shiftmax_out(shift_exp_mag((uint32_t)(mx1 - S[nt][2]), se), rn1) : 0u;
            pv[nt][3] = v1 ? shiftmax_out(shift_exp_mag((uint32_t)(mx1 - S[nt][3]), se), rn1) : 0u;
        }
#pragma unroll
        for (int ch = 0; ch < 2; ++ch) {
            uint32_t a[4];
            const int n0 = 4 * ch;
            a[0] = pv[n0][0] | (pv[n0][1] << 8) | (pv[n0 + 1][0] << 16) | (pv[n0 + 1][1] << 24);
            a[1] = pv[n0][2] | (pv[n0][3] << 8) | (pv[n0 + 1][2] << 16) | (pv[n0 + 1][3] << 24);
            a[2] = pv[n0 + 2][0] | (pv[n0 + 2][1] << 8) | (pv[n0 + 3][0] << 16) | (pv[n0 + 3][1] << 24);
            a[3] = pv[n0 + 2][2] | (pv[n0 + 2][3] << 8) | (pv[n0 + 3][2] << 16) | (pv[n0 + 3][3] << 24);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const int8_t *v = Vt + (nt * 8 + g) * LDV + ch * 32 + 4 * t;
                mma_u8s8(o[nt], a, *(const uint32_t *)v, *(const uint32_t *)(v + 16));
            }
        }
        __syncthreads();
    }

    // ---- epilogue: sat8(rq(O; m_o, s_o)), written back at the tokens' own positions
    const int r0 = q0 + warp * 16 + g, r1 = r0 + 8;
    const bool ok0 = r0 < Tg, ok1 = r1 < Tg;
    int8_t *O0 = ok0 ? p.O + gr.token(r0) * p.ld_o + hoff : nullptr;
    int8_t *O1 = ok1 ? p.O + gr.token(r1) * p.ld_o + hoff : nullptr;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        int col = nt * 8 + 2 * t;
        if (ok0) {
            O0[col] = (int8_t)sat8(rq(o[nt][0], p.m_o, p.s_o));
            O0[col + 1] = (int8_t)sat8(rq(o[nt][1], p.m_o, p.s_o));
        }
        if (ok1) {
            O1[col] = (int8_t)sat8(rq(o[nt][2], p.m_o, p.s_o));
            O1[col + 1] = (int8_t)sat8(rq(o[nt][3], p.m_o, p.s_o));
        }
    }
}

}  // namespace

cudaError_t launch_attention(const AttnParams &p, cudaStream_t s) {
    const int G2 = p.nw > 1 ? p.nw * p.nw : 1;
    const int Tg = p.nw > 1 ? (p.grid_side / p.nw) * (p.grid_side / p.nw) : p.T;
    if (p.B == 0 || Tg == 0) return cudaSuccess;
    dim3 grid((Tg + QT - 1) / QT, p.H, p.B * G2);
    if (p.dh == 64) attn_kernel<64><<<grid, THREADS, 0, s>>>(p);
    else attn_kernel<32><<<grid, THREADS, 0, s>>>(p);
    return cudaGetLastError();
}

}  // namespace ilw
