// patch.cu -- patch gathering for the ViT patch embedding (a p x p, stride-p integer
// convolution, computed as the integer GEMM of Sec. 3.2.1 over non-overlapping patches).
//
// Each thread moves one 16-byte row segment of one patch: img[b, ch, py*p + ky, px*p + 16j ..]
// -> A[b*T + t, (ch*p + ky)*p + 16j ..], so both sides are 16-byte vector accesses.
#include <cstdint>

#include "ilw_kernels.h"

namespace ilw {
namespace {

__global__ void __launch_bounds__(256) patchify_kernel(const int8_t *__restrict__ img, int32_t Cin, int32_t Hh,
                                                       int32_t Ww, int32_t p, int64_t total,
                                                       int8_t *__restrict__ A) {
    int64_t id = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (id >= total) return;
    const int segs = p >> 4;  // 16-byte segments per patch row
    const int Gw = Ww / p, T = (Hh / p) * Gw;
    const int j = (int)(id % segs);
    int64_t r = id / segs;
    const int ky = (int)(r % p);
    r /= p;
    const int ch = (int)(r % Cin);
    const int64_t bt = r / Cin;  // b * T + t
    const int t = (int)(bt % T);
    const int64_t b = bt / T;
    const int py = t / Gw, px = t % Gw;
    const int4 v = *(const int4 *)(img + ((b * Cin + ch) * Hh + (int64_t)py * p + ky) * Ww + (int64_t)px * p + 16 * j);
    *(int4 *)(A + bt * ((int64_t)Cin * p * p) + ((int64_t)ch * p + ky) * p + 16 * j) = v;
}

// The same gather with the patch matrix written as fp16 (the int8 values, exact): 16 int8 -> 32
// bytes of fp16.  0x6400 | (b ^ 0x80) is the fp16 of 1152 + b; one half2 subtract of 1152 leaves b.
__device__ __forceinline__ uint32_t i8x2_f16(uint32_t w) {
    const uint32_t x = __byte_perm(w ^ 0x8080u, 0x64646464u, 0x4140);
    __half2 h = __hsub2(*reinterpret_cast<const __half2 *>(&x), __half2half2(__ushort_as_half((unsigned short)0x6480)));
    return *reinterpret_cast<uint32_t *>(&h);
}
__global__ void __launch_bounds__(256) patchify_f16_kernel(const int8_t *__restrict__ img, int32_t Cin, int32_t Hh,
                                                           int32_t Ww, int32_t p, int64_t total,
                                                           __half *__restrict__ A) {
    int64_t id = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (id >= total) return;
    const int segs = p >> 4;
    const int Gw = Ww / p, T = (Hh / p) * Gw;
    const int j = (int)(id % segs);
    int64_t r = id / segs;
    const int ky = (int)(r % p);
    r /= p;
    const int ch = (int)(r % Cin);
    const int64_t bt = r / Cin;
    const int t = (int)(bt % T);
    const int64_t b = bt / T;
    const int py = t / Gw, px = t % Gw;
    const uint4 v = *(const uint4 *)(img + ((b * Cin + ch) * Hh + (int64_t)py * p + ky) * Ww + (int64_t)px * p + 16 * j);
    uint4 lo, hi;
    lo.x = i8x2_f16(v.x); lo.y = i8x2_f16(v.x >> 16); lo.z = i8x2_f16(v.y); lo.w = i8x2_f16(v.y >> 16);
    hi.x = i8x2_f16(v.z); hi.y = i8x2_f16(v.z >> 16); hi.z = i8x2_f16(v.w); hi.w = i8x2_f16(v.w >> 16);
    uint4 *dst = (uint4 *)(A + bt * ((int64_t)Cin * p * p) + ((int64_t)ch * p + ky) * p + 16 * j);
    dst[0] = lo;
    dst[1] = hi;
}

}  // namespace

cudaError_t launch_patchify_f16(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                                __half *A, cudaStream_t s) {
    int64_t total = (int64_t)B * (Hh / p) * (Ww / p) * Cin * p * (p / 16);
    if (total == 0) return cudaSuccess;
    patchify_f16_kernel<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(img, Cin, Hh, Ww, p, total, A);
    return cudaGetLastError();
}

cudaError_t launch_patchify(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                            int8_t *A, cudaStream_t s) {
    int64_t total = (int64_t)B * (Hh / p) * (Ww / p) * Cin * p * (p / 16);
    if (total == 0) return cudaSuccess;
    patchify_kernel<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(img, Cin, Hh, Ww, p, total, A);
    return cudaGetLastError();
}

}  // namespace ilw
