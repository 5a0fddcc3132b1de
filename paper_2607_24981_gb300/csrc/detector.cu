// detector.cu -- element and gather kernels of the detector's projector and decoder:
// per-tensor requantisation with an optional second term (the int16 residual stream -> the int8
// input of the next integer linear layer, Sec. 3.2.1; query + positional query in the decoder)
// and nearest-neighbour resampling of the projector's feature maps to the levels' strides.
#include <cstdint>

#include "ilw_kernels.h"

namespace ilw {
namespace {

template <typename T>
__device__ __forceinline__ void load4(const T *p, int64_t (&v)[4]);
template <>
__device__ __forceinline__ void load4<int16_t>(const int16_t *p, int64_t (&v)[4]) {
    const uint2 w = *(const uint2 *)p;
    v[0] = (int16_t)(w.x & 0xffff); v[1] = (int16_t)(w.x >> 16);
    v[2] = (int16_t)(w.y & 0xffff); v[3] = (int16_t)(w.y >> 16);
}
template <>
__device__ __forceinline__ void load4<int32_t>(const int32_t *p, int64_t (&v)[4]) {
    const int4 w = *(const int4 *)p;
    v[0] = w.x; v[1] = w.y; v[2] = w.z; v[3] = w.w;
}

// One thread per 4 consecutive elements of a row (C % 4 == 0, rows 8/16-byte aligned).
template <typename TIn, typename TOut>
__global__ void __launch_bounds__(256) requant_kernel(const RequantParams p) {
    const int32_t cq = p.C >> 2;
    const int64_t total = p.rows * cq;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cq;
        const int32_t c = (int32_t)(i - r * cq) * 4;
        int64_t x[4], z[4] = {0, 0, 0, 0};
        load4<TIn>((const TIn *)p.X + r * p.ldx + c, x);
        if (p.Z) load4<int16_t>(p.Z + (r % p.z_rows) * p.ldz + c, z);
        TOut o[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            int64_t v = rq(x[u], p.m1, p.s1);
            if (p.Z) v += rq(z[u], p.m2, p.s2);
            o[u] = (TOut)(sizeof(TOut) == 1 ? sat8(v) : (sizeof(TOut) == 2 ? sat16(v) : (int32_t)v));
        }
        TOut *y = (TOut *)p.Y + r * p.ldy + c;
        if (sizeof(TOut) == 1)
            *(uint32_t *)y = (uint32_t)(uint8_t)o[0] | ((uint32_t)(uint8_t)o[1] << 8) | ((uint32_t)(uint8_t)o[2] << 16) |
                             ((uint32_t)(uint8_t)o[3] << 24);
        else if (sizeof(TOut) == 2)
            *(uint2 *)y = make_uint2((uint32_t)(uint16_t)o[0] | ((uint32_t)(uint16_t)o[1] << 16),
                                     (uint32_t)(uint16_t)o[2] | ((uint32_t)(uint16_t)o[3] << 16));
        else
            *(int4 *)y = make_int4((int32_t)o[0], (int32_t)o[1], (int32_t)o[2], (int32_t)o[3]);
    }
}

// Nearest-neighbour resampling, one thread per 16 channels of one output pixel:
// Y[b][y*Wo + x] = X[b][floor(y*Hi/Ho)*Wi + floor(x*Wi/Wo)].
__global__ void __launch_bounds__(256) resample_kernel(const int8_t *__restrict__ X, int64_t x_bstride, int32_t B,
                                                       int32_t Hi, int32_t Wi, int32_t C, int8_t *__restrict__ Y,
                                                       int64_t y_bstride, int32_t Ho, int32_t Wo) {
    const int32_t c16 = C >> 4;
    const int64_t total = (int64_t)B * Ho * Wo * c16;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t ch = (int32_t)(i % c16);
        const int64_t pix = i / c16;
        const int32_t x = (int32_t)(pix % Wo);
        const int64_t by = pix / Wo;
        const int32_t y = (int32_t)(by % Ho), b = (int32_t)(by / Ho);
        const int64_t sy = (int64_t)y * Hi / Ho, sx = (int64_t)x * Wi / Wo;
        const uint4 v = *(const uint4 *)(X + ((int64_t)b * x_bstride + sy * Wi + sx) * C + ch * 16);
        *(uint4 *)(Y + ((int64_t)b * y_bstride + (int64_t)y * Wo + x) * C + ch * 16) = v;
    }
}

// Heads of dh < 64 columns widened to 64: Y[m, (p H + h) 64 + c] = X[m, (p H + h) dh + c] for c < dh,
// 0 above (the int8 values carried in fp16), for nparts consecutive groups of H heads.  Eight
// outputs (16 bytes) per item.
__global__ void head_pad64_kernel(const int8_t *__restrict__ X, int64_t ldx, int64_t M, int32_t nh, int32_t dh,
                                  __half *__restrict__ Y) {
    const int64_t per_row = (int64_t)nh * 8;  // 16-byte chunks of a padded row
    const int64_t items = M * per_row;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < items; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = i / per_row;
        const int32_t j = (int32_t)(i - m * per_row), head = j >> 3, c0 = (j & 7) * 8;
        uint32_t w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int c = c0 + 2 * u;
            const int8_t *x = X + m * ldx + (int64_t)head * dh + c;
            const int32_t a = c < dh ? (int32_t)x[0] : 0, b = c + 1 < dh ? (int32_t)x[1] : 0;
            // |v| <= 127: 1152 + v has the fp16 bits 0x6480 + v; subtracting 1152 leaves v
            uint32_t hb = (uint32_t)(0x6480 + a) | ((uint32_t)(0x6480 + b) << 16);
            const __half2 hh = __hsub2(*reinterpret_cast<__half2 *>(&hb), __half2half2(__ushort_as_half((unsigned short)0x6480)));
            w[u] = *reinterpret_cast<const uint32_t *>(&hh);
        }
        *(uint4 *)(Y + m * (per_row * 8) + (int64_t)j * 8) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// The inverse for int8 rows: O[m, h dh + c] = Y[m, h 64 + c] for c < dh.
__global__ void head_compact_kernel(const int8_t *__restrict__ Y, int64_t ldy, int64_t M, int32_t H, int32_t dh,
                                    int8_t *__restrict__ O, int64_t ldo) {
    const int64_t per_row = (int64_t)H * dh;
    const int64_t items = M * per_row;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < items; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = i / per_row;
        const int32_t j = (int32_t)(i - m * per_row), head = j / dh, c = j - head * dh;
        O[m * ldo + j] = Y[m * ldy + (int64_t)head * 64 + c];
    }
}

unsigned grid_for(int64_t items) {
    int64_t g = (items + 255) / 256;
    const int64_t cap = (int64_t)sm_count() * 16;  // grid-stride loops: 16 CTAs of 256 threads per SM
    return (unsigned)(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

cudaError_t launch_requant(const RequantParams &p, cudaStream_t s) {
    const int64_t items = p.rows * (p.C / 4);
    if (items == 0) return cudaSuccess;
    const unsigned g = grid_for(items);
    if (p.in_bits == 16) {
        if (p.out_bits == 8) requant_kernel<int16_t, int8_t><<<g, 256, 0, s>>>(p);
        else if (p.out_bits == 16) requant_kernel<int16_t, int16_t><<<g, 256, 0, s>>>(p);
        else requant_kernel<int16_t, int32_t><<<g, 256, 0, s>>>(p);
    } else {
        if (p.out_bits == 8) requant_kernel<int32_t, int8_t><<<g, 256, 0, s>>>(p);
        else if (p.out_bits == 16) requant_kernel<int32_t, int16_t><<<g, 256, 0, s>>>(p);
        else requant_kernel<int32_t, int32_t><<<g, 256, 0, s>>>(p);
    }
    return cudaGetLastError();
}

cudaError_t launch_head_pad64(const int8_t *X, int64_t ldx, int64_t M, int32_t nh, int32_t dh, __half *Y,
                              cudaStream_t s) {
    if (M == 0 || nh == 0) return cudaSuccess;
    head_pad64_kernel<<<grid_for(M * nh * 8), 256, 0, s>>>(X, ldx, M, nh, dh, Y);
    return cudaGetLastError();
}
cudaError_t launch_head_compact(const int8_t *Y, int64_t ldy, int64_t M, int32_t H, int32_t dh, int8_t *O, int64_t ldo,
                                cudaStream_t s) {
    if (M == 0 || H == 0) return cudaSuccess;
    head_compact_kernel<<<grid_for(M * H * dh), 256, 0, s>>>(Y, ldy, M, H, dh, O, ldo);
    return cudaGetLastError();
}

cudaError_t launch_resample(const int8_t *X, int64_t x_bstride, int32_t B, int32_t Hi, int32_t Wi, int32_t C,
                            int8_t *Y, int64_t y_bstride, int32_t Ho, int32_t Wo, cudaStream_t s) {
    const int64_t items = (int64_t)B * Ho * Wo * (C / 16);
    if (items == 0) return cudaSuccess;
    resample_kernel<<<grid_for(items), 256, 0, s>>>(X, x_bstride, B, Hi, Wi, C, Y, y_bstride, Ho, Wo);
    return cudaGetLastError();
}

}  // namespace ilw
