// gemm_mma.cu -- exact integer GEMM on the warp-level int8 tensor-core MMA
// (mma.sync m16n8k32 s8.s8 -> s32), with the bias, dyadic requantisation, residual,
// SD-ShiftGELU and split-convolution epilogues fused (Sec. 3.2.1, 3.2.2, 3.3.1).
//
// Tile 128 x 128 x 64, 8 warps (2 along M x 4 along N, 64 x 32 each), 4-stage cp.async
// pipeline.  Shared-memory rows are padded to 80 bytes so the 32-bit fragment loads of a
// quad-row pattern hit 32 distinct banks.
#include <cstdint>

#include "ilw_kernels.h"

namespace ilw {
namespace {

constexpr int BM = 128, BN = 128, BK = 64, STAGES = 4, THREADS = 256;
constexpr int LDS = BK + 16;  // padded smem row (bytes)
constexpr int STAGE_BYTES = (BM + BN) * LDS;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES;

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem, bool valid) {
    uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
    int n = valid ? 16 : 0;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void mma_s8(int32_t (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Epilogue: one output element (row, col) with the exact int32 accumulator (bias not yet added).
__device__ __forceinline__ void epilogue_store(const EpiParams &ep, int row, int col, int32_t acc) {
    int64_t v = (int64_t)acc + (ep.bias ? ep.bias[col] : 0);
    if (ep.kind == EPI_GELU) {
        int32_t g = sat16(rq(v, ep.mult[col], ep.shift[col]));
        int32_t idiv = gelu_idiv(g, ep.gelu);
        int8_t h = (int8_t)sat8(rq((int64_t)g * idiv, ep.m_g, ep.s_g));
        ((int8_t *)ep.C)[(int64_t)row * ep.ldc + col] = h;
        return;
    }
    if (ep.out_bits == 32) {
        ((int32_t *)ep.C)[(int64_t)row * ep.ldc + col] = (int32_t)v;
        return;
    }
    int64_t o = rq(v, ep.mult[col], ep.shift[col]);
    if (ep.res) o += rq((int64_t)ep.res[(row % ep.res_rows) * ep.ldr + col], ep.m_r, ep.s_r);
    if (ep.out_bits == 8)
        ((int8_t *)ep.C)[(int64_t)row * ep.ldc + col] = (int8_t)sat8(o);
    else
        ((int16_t *)ep.C)[(int64_t)row * ep.ldc + col] = (int16_t)sat16(o);
}

template <bool SPLIT>
__global__ void __launch_bounds__(THREADS) gemm_mma_kernel(const GemmProblem gp, const EpiParams ep) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, t = lane & 3;
    const int wm = warp >> 2, wn = warp & 3;  // 2 x 4 warps
    const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN;

    int32_t acc[4][4][4];
    int32_t run[SPLIT ? 4 : 1][SPLIT ? 4 : 1][SPLIT ? 4 : 1];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                acc[i][j][r] = 0;
                if (SPLIT) run[SPLIT ? i : 0][SPLIT ? j : 0][SPLIT ? r : 0] = 0;
            }

    for (int b = 0; b < gp.nb; ++b) {
        const GemmBranch br = gp.br[b];
        const int KT = (br.K + BK - 1) / BK;
        auto load_stage = [&](int kt, int stage) {
            uint8_t *As = smem + stage * STAGE_BYTES;
            uint8_t *Bs = As + BM * LDS;
            const int k0 = kt * BK;
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                int c = tid + i * THREADS;
                int row = c >> 2, kc = (c & 3) * 16;
                bool kv = (k0 + kc) < br.K;
                int gm = m0 + row;
                bool va = kv && gm < gp.M;
                cp_async16(As + row * LDS + kc, va ? (const void *)(br.A + (int64_t)gm * br.lda + k0 + kc) : (const void *)br.A, va);
                int gn = n0 + row;
                bool vb = kv && gn < gp.N;
                cp_async16(Bs + row * LDS + kc, vb ? (const void *)(br.W + (int64_t)gn * br.K + k0 + kc) : (const void *)br.W, vb);
            }
        };
#pragma unroll
        for (int s = 0; s < STAGES - 1; ++s) {
            if (s < KT) load_stage(s, s);
            cp_async_commit();
        }
        for (int kt = 0; kt < KT; ++kt) {
            cp_async_wait<STAGES - 2>();
            __syncthreads();
            int nk = kt + STAGES - 1;
            if (nk < KT) load_stage(nk, nk % STAGES);
            cp_async_commit();
            const uint8_t *As = smem + (kt % STAGES) * STAGE_BYTES;
            const uint8_t *Bs = As + BM * LDS;
#pragma unroll
            for (int kk = 0; kk < BK; kk += 32) {
                uint32_t af[4][4], bf[4][2];
#pragma unroll
                for (int mi = 0; mi < 4; ++mi) {
                    const uint8_t *p = As + (wm * 64 + mi * 16 + g) * LDS + kk + 4 * t;
                    af[mi][0] = *(const uint32_t *)(p);
                    af[mi][1] = *(const uint32_t *)(p + 8 * LDS);
                    af[mi][2] = *(const uint32_t *)(p + 16);
                    af[mi][3] = *(const uint32_t *)(p + 8 * LDS + 16);
                }
#pragma unroll
                for (int ni = 0; ni < 4; ++ni) {
                    const uint8_t *p = Bs + (wn * 32 + ni * 8 + g) * LDS + kk + 4 * t;
                    bf[ni][0] = *(const uint32_t *)(p);
                    bf[ni][1] = *(const uint32_t *)(p + 16);
                }
#pragma unroll
                for (int mi = 0; mi < 4; ++mi)
#pragma unroll
                    for (int ni = 0; ni < 4; ++ni) mma_s8(acc[mi][ni], af[mi], bf[ni][0], bf[ni][1]);
            }
        }
        cp_async_wait<0>();
        __syncthreads();
        if (SPLIT) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j)
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        int32_t v = gp.branch_rq ? (int32_t)rq(acc[i][j][r], br.m_b, br.s_b) : acc[i][j][r];
                        run[SPLIT ? i : 0][SPLIT ? j : 0][SPLIT ? r : 0] += v;
                        acc[i][j][r] = 0;
                    }
        }
    }

#pragma unroll
    for (int mi = 0; mi < 4; ++mi) {
#pragma unroll
        for (int ni = 0; ni < 4; ++ni) {
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                int row = m0 + wm * 64 + mi * 16 + g + (r >> 1) * 8;
                int col = n0 + wn * 32 + ni * 8 + 2 * t + (r & 1);
                if (row < gp.M && col < gp.N) {
                    int32_t v = SPLIT ? run[SPLIT ? mi : 0][SPLIT ? ni : 0][SPLIT ? r : 0] : acc[mi][ni][r];
                    epilogue_store(ep, row, col, v);
                }
            }
        }
    }
}

__global__ void pack_weight_kernel(const int8_t *W, int64_t n, int8_t *w8, __half *w16) {
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) {
        int8_t v = W[i];
        w8[i] = v;
        w16[i] = __int2half_rn((int)v);  // |v| <= 127: exact in fp16
    }
}

}  // namespace

size_t packed_weight_bytes(int32_t N, int32_t K) {
    size_t n = (size_t)N * K;
    return ((n + 255) & ~(size_t)255) + 2 * n;
}

cudaError_t launch_pack_weight(const int8_t *W, int32_t N, int32_t K, void *packed, cudaStream_t s) {
    int64_t n = (int64_t)N * K;
    int8_t *w8 = (int8_t *)packed;
    __half *w16 = (__half *)packed_f16(packed, N, K);
    pack_weight_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(W, n, w8, w16);
    return cudaGetLastError();
}

cudaError_t launch_gemm_mma(const GemmProblem &gp, const EpiParams &ep, cudaStream_t s) {
    if (gp.M == 0 || gp.N == 0) return cudaSuccess;
    dim3 grid((gp.M + BM - 1) / BM, (gp.N + BN - 1) / BN);
    bool split = gp.nb > 1 || gp.branch_rq;
    if (split) {
        static bool attr = false;
        if (!attr) {
            cudaError_t e = cudaFuncSetAttribute(gemm_mma_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
            if (e != cudaSuccess) return e;
            attr = true;
        }
        gemm_mma_kernel<true><<<grid, THREADS, SMEM_BYTES, s>>>(gp, ep);
    } else {
        static bool attr = false;
        if (!attr) {
            cudaError_t e = cudaFuncSetAttribute(gemm_mma_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
            if (e != cudaSuccess) return e;
            attr = true;
        }
        gemm_mma_kernel<false><<<grid, THREADS, SMEM_BYTES, s>>>(gp, ep);
    }
    return cudaGetLastError();
}

}  // namespace ilw
