// heads.cu -- the detection head's elementwise and selection kernels: integer sigmoid (the head's
// exponential by ShiftExp, Table 5, in SD-ShiftGELU's sign-dependent sigmoid form, Sec. 3.3.1 and
// Algorithm 1), ReLU on int8, per-row integer top-K (two-stage query selection) and row gather.
#include <climits>
#include <cstdint>

#include "ilw_kernels.h"

namespace ilw {
namespace {

// out = (E F) >> (32 - k_out), E = ShiftExp(min(x, 0)), E' = ShiftExp(-max(x, 0)),
// F = floor((2^31 - 1) / (E + E')).  One of the two ShiftExp inputs is always 0 and ShiftExp(0) =
// I0 2^k, so one ShiftExp of -|x| gives both.  |x| is clamped at 2^30 (past k I0 < 2^20 ShiftExp
// sits in its clamp region, so the clamp changes nothing).
__device__ __forceinline__ int32_t int_sigmoid1(int32_t x, const ShiftExpC &se, int32_t out_sh) {
    const uint32_t a = x < 0 ? 0u - (uint32_t)x : (uint32_t)x;
    const uint32_t e = shift_exp_mag(min(a, 1u << 30), se);
    const uint32_t top = (uint32_t)se.I0 << se.k;
    const uint32_t E = x >= 0 ? top : e;
    const uint32_t F = div_int31(top + e);
    return (int32_t)(((uint64_t)E * F) >> out_sh);
}

__global__ void __launch_bounds__(256) int_sigmoid_kernel(const int32_t *__restrict__ X, int32_t *__restrict__ Y,
                                                          int64_t n, ShiftExpC se, int32_t out_sh) {
    const int64_t n4 = n / 4;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
        const int4 v = ((const int4 *)X)[i];
        ((int4 *)Y)[i] = make_int4(int_sigmoid1(v.x, se, out_sh), int_sigmoid1(v.y, se, out_sh),
                                   int_sigmoid1(v.z, se, out_sh), int_sigmoid1(v.w, se, out_sh));
    }
    for (int64_t i = 4 * n4 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        Y[i] = int_sigmoid1(X[i], se, out_sh);
}

// ReLU of int8 values, four per thread step (n4 words), then the tail
__global__ void __launch_bounds__(256) relu_i8_kernel(const int8_t *__restrict__ X, int8_t *__restrict__ Y, int64_t n) {
    const int64_t n4 = n / 4;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4; i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t w = ((const uint32_t *)X)[i];
        // keep the bytes whose sign bit is clear
        const uint32_t neg = (w & 0x80808080u) >> 7;  // 1 in each negative byte's low bit
        ((uint32_t *)Y)[i] = w & ~(neg * 0xFFu);
    }
    for (int64_t i = 4 * n4 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        Y[i] = X[i] < 0 ? (int8_t)0 : X[i];
}

// Per-row top-K by a bitonic sort of (value, index) keys in shared memory: key = (value biased to
// unsigned) << 32 | (2^32 - 1 - index), so one descending order puts larger values first and, for
// equal values, smaller indices first.  Padding keys are 0, below every real key.
__global__ void topk_kernel(const int32_t *__restrict__ S, int64_t lds, int32_t N, int32_t npad, int32_t K,
                            int32_t *__restrict__ vals, int32_t *__restrict__ idx) {
    extern __shared__ unsigned long long keys[];
    const int32_t *s = S + (int64_t)blockIdx.x * lds;
    for (int i = threadIdx.x; i < npad; i += blockDim.x)
        keys[i] = i < N ? ((unsigned long long)((uint32_t)s[i] ^ 0x80000000u) << 32) | (0xFFFFFFFFu - (uint32_t)i) : 0ull;
    __syncthreads();
    for (int k = 2; k <= npad; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < npad; i += blockDim.x) {
                const int ixj = i ^ j;
                if (ixj > i) {
                    const unsigned long long a = keys[i], b = keys[ixj];
                    if (((i & k) == 0) ? (a < b) : (a > b)) {
                        keys[i] = b;
                        keys[ixj] = a;
                    }
                }
            }
            __syncthreads();
        }
    for (int i = threadIdx.x; i < K; i += blockDim.x) {
        const unsigned long long key = keys[i];
        vals[(int64_t)blockIdx.x * K + i] = (int32_t)((uint32_t)(key >> 32) ^ 0x80000000u);
        idx[(int64_t)blockIdx.x * K + i] = (int32_t)(0xFFFFFFFFu - (uint32_t)key);
    }
}

// K = 1: one warp per row keeps the largest value with the smallest index among its columns, and
// the warp combines the lanes' candidates (larger value, or equal value and smaller index, wins).
__global__ void __launch_bounds__(256) top1_kernel(const int32_t *__restrict__ S, int64_t lds, int32_t rows, int32_t N,
                                                   int32_t *__restrict__ vals, int32_t *__restrict__ idx) {
    const int lane = threadIdx.x & 31;
    const int64_t wpr = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t r = blockIdx.x * (int64_t)(blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += wpr) {
        const int32_t *s = S + r * lds;
        int32_t bv = INT32_MIN, bi = INT32_MAX;
        for (int j = lane; j < N; j += 32) {
            const int32_t v = s[j];
            if (v > bv || bi == INT32_MAX) {  // columns rise with j, so only a larger value replaces
                bv = v;
                bi = j;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const int32_t ov = __shfl_xor_sync(0xffffffffu, bv, o), oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ov > bv || (ov == bv && oi < bi)) {
                bv = ov;
                bi = oi;
            }
        }
        if (lane == 0) {
            vals[r] = bv;
            idx[r] = bi;
        }
    }
}

// Row gather in 4-byte words: dst row i = src row idx[i].  An index outside [0, src_rows) gives a
// zero row and latches kStatusBadIndex in the device status word.
__global__ void __launch_bounds__(256) gather_rows_kernel(const uint32_t *__restrict__ src, int64_t src_ldw,
                                                          int64_t src_rows, const int32_t *__restrict__ idx, int64_t n,
                                                          int64_t roww, uint32_t *__restrict__ dst, int64_t dst_ldw,
                                                          int *status) {
    const int64_t total = n * roww;
    for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
        const int64_t i = t / roww, w = t - i * roww;
        const int64_t r = idx[i];
        if (r < 0 || r >= src_rows) {
            dst[i * dst_ldw + w] = 0u;
            if (w == 0 && status) atomicExch(status, kStatusBadIndex);
            continue;
        }
        dst[i * dst_ldw + w] = src[r * src_ldw + w];
    }
}

// I-ViT's ShiftGELU (the baseline of Sec. 3.3.1), one warp per row: M = max(max_row 1.702 x, 0),
// E = ShiftExp(I_p - M), E' = ShiftExp(-M), I_div = (E F) >> out_sh, Y = x I_div.  1.702 x by shifts
// in 64 bits (no int32 overflow for any input); ShiftExp magnitudes clamped at 2^30 (past k I0 the
// result no longer changes).
__device__ __forceinline__ int64_t ip1702(int32_t x) {
    const int64_t v = x;
    return v + (v >> 1) + (v >> 3) + (v >> 4);
}
__global__ void __launch_bounds__(256) ivit_shiftgelu_kernel(const int32_t *__restrict__ X, int64_t ldx, int64_t rows,
                                                             int32_t L, int32_t *__restrict__ Y, int64_t ldy,
                                                             ShiftExpC se, int32_t out_sh) {
    const int lane = threadIdx.x & 31;
    const int64_t wpr = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t r = blockIdx.x * (int64_t)(blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += wpr) {
        const int32_t *x = X + r * ldx;
        int64_t M = 0;
        for (int c = lane; c < L; c += 32) M = max(M, ip1702(x[c]));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) M = max(M, (int64_t)__shfl_xor_sync(0xffffffffu, (long long)M, o));
        const uint32_t e2 = shift_exp_mag((uint32_t)min(M, (int64_t)1 << 30), se);
        for (int c = lane; c < L; c += 32) {
            const int32_t v = x[c];
            const uint32_t E = shift_exp_mag((uint32_t)min(M - ip1702(v), (int64_t)1 << 30), se);
            const uint32_t F = div_int31(E + e2);
            const int64_t idiv = (int64_t)(((uint64_t)E * F) >> out_sh);
            Y[r * ldy + c] = (int32_t)((int64_t)v * idiv);
        }
    }
}

unsigned grid_for(int64_t work, int per_block) {
    const int64_t g = (work + per_block - 1) / per_block;
    const int64_t cap = (int64_t)sm_count() * 16;  // grid-stride loops: 16 CTAs of 256 threads per SM
    return (unsigned)(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

cudaError_t launch_int_sigmoid(const int32_t *X, int32_t *Y, int64_t n, const ShiftExpC &se, int32_t k_out,
                               cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    int_sigmoid_kernel<<<grid_for((n + 3) / 4, 256), 256, 0, s>>>(X, Y, n, se, 32 - k_out);
    return cudaGetLastError();
}

cudaError_t launch_ivit_shiftgelu(const int32_t *X, int64_t ldx, int64_t rows, int32_t L, int32_t *Y, int64_t ldy,
                                  const GeluC &c, cudaStream_t s) {
    if (rows == 0) return cudaSuccess;
    ivit_shiftgelu_kernel<<<grid_for((rows + 7) / 8, 1), 256, 0, s>>>(X, ldx, rows, L, Y, ldy, c.se, c.out_sh);
    return cudaGetLastError();
}

cudaError_t launch_relu_i8(const int8_t *X, int8_t *Y, int64_t n, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    relu_i8_kernel<<<grid_for((n + 3) / 4, 256), 256, 0, s>>>(X, Y, n);
    return cudaGetLastError();
}

cudaError_t launch_topk(const int32_t *S, int64_t lds, int32_t rows, int32_t N, int32_t K, int32_t *vals,
                        int32_t *idx, cudaStream_t s) {
    if (rows == 0) return cudaSuccess;
    if (K == 1) {
        top1_kernel<<<grid_for(((int64_t)rows + 7) / 8, 1), 256, 0, s>>>(S, lds, rows, N, vals, idx);
        return cudaGetLastError();
    }
    int npad = 2;
    while (npad < N) npad <<= 1;
    const size_t smem = (size_t)npad * 8;
    const int threads = npad / 2 < 1024 ? (npad / 2 < 32 ? 32 : npad / 2) : 1024;
    if (smem > 48 * 1024) {
        const cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    topk_kernel<<<(unsigned)rows, threads, smem, s>>>(S, lds, N, npad, K, vals, idx);
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const void *src, int64_t src_ld_bytes, int64_t src_rows, const int32_t *idx, int64_t n,
                               int64_t row_bytes, void *dst, int64_t dst_ld_bytes, cudaStream_t s) {
    if (n == 0 || row_bytes == 0) return cudaSuccess;
    gather_rows_kernel<<<grid_for(n * (row_bytes / 4), 256), 256, 0, s>>>((const uint32_t *)src, src_ld_bytes / 4,
                                                                           src_rows, idx, n, row_bytes / 4,
                                                                           (uint32_t *)dst, dst_ld_bytes / 4,
                                                                           status_word_ptr());
    return cudaGetLastError();
}

}  // namespace ilw
