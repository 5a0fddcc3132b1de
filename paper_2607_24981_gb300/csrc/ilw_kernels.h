// ilw_kernels.h -- internal launch interface between the C-ABI layer and the kernels.
#pragma once
#include <cstdint>
#include <mutex>
#include <cuda_runtime.h>

#include "ilw_device.cuh"

namespace ilw {

// Records `msg` as this thread's ilwdetr_last_error() text and returns `code`.
int report_error(int code, const char *msg);
// True while the calling thread's entry points only check their arguments (ilwdetr_validate_only,
// or a composite entry point's checking pass): they return before any CUDA call that launches.
bool validate_only();

// Device status word (latched by kernels whose bounded waits expire): its device address on
// the current device (nullptr on failure), and a synchronous read-and-clear.
int *status_word_ptr();
cudaError_t read_and_clear_status(int *value);
// Streaming multiprocessors of the current device (read from the device once per device).
int sm_count();

// A kernel's dynamic shared-memory limit, raised once per device: a function attribute belongs
// to the device it was set on, so each device of the process gets its own call.  One SmemLimit
// (a function-local static) per kernel; later calls on a device return its first call's result.
constexpr int kMaxAttrDevices = 64;
struct SmemLimit {
    std::once_flag once[kMaxAttrDevices];
    cudaError_t err[kMaxAttrDevices] = {};
};
inline cudaError_t raise_smem_limit(SmemLimit &st, const void *kernel, int bytes) {
    int dev = 0;
    const cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxAttrDevices) return cudaErrorInvalidDevice;
    std::call_once(st.once[dev], [&] {
        st.err[dev] = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    });
    return st.err[dev];
}
constexpr int kStatusTimeoutTma = 1;     // a wait for a TMA load ran out
constexpr int kStatusTimeoutMma = 2;     // a wait for tensor-core completion ran out
constexpr int kStatusTimeoutOperand = 3; // a wait for the converted operand ran out
constexpr int kStatusTimeoutFree = 4;    // a wait for a free pipeline stage ran out
constexpr int kStatusBadIndex = 5;       // a gather index lay outside its source

// Host-side construction of the per-launch ShiftExp constants (Algorithm 1).
inline ShiftExpC make_shiftexp(int32_t I0, int32_t k) {
    ShiftExpC c;
    c.I0 = I0;
    c.kI0 = k * I0;
    uint64_t M = (((uint64_t)1 << 40) + (uint64_t)I0 - 1) / (uint64_t)I0;  // ceil(2^40 / I0)
    c.m_lo = (uint32_t)(M & 0xffffffffull);
    c.m_hi = (uint32_t)(M >> 32);
    c.k = k;
    const uint64_t kI0sq = (uint64_t)(k > 0 ? k : 0) * (uint64_t)I0 * (uint64_t)I0;
    c.m32 = (I0 >= 2 && kI0sq < ((uint64_t)1 << 32))
                ? (uint32_t)((((uint64_t)1 << 32) + (uint64_t)I0 - 1) / (uint64_t)I0)
                : 0u;
    return c;
}
inline GeluC make_gelu(const ilw_gelu_t &g) {
    GeluC c;
    c.se = make_shiftexp(g.I0, g.k_inter);
    c.out_sh = 31 - g.k_out + 1;
    return c;
}

// ---------------------------------------------------------------- GEMM
constexpr int kMaxBranches = 8;
struct GemmBranch {
    const int8_t *A;   // [M, K] row-major, lda
    int64_t lda;
    const int8_t *W;   // [N, K] row-major (ld = K)
    const void *Wp;    // packed weight (tensor-core operand form)
    int32_t K;
    int32_t m_b, s_b;  // split-conv branch rescale (ignored for a plain GEMM)
};
struct GemmProblem {
    int32_t M, N;
    int32_t nb;        // branches; 1 = plain GEMM
    bool branch_rq;    // rq each branch partial with (m_b, s_b) before the integer sum
    bool a_f16;        // A holds the int8 values as fp16 (plain GEMM only)
    GemmBranch br[kMaxBranches];
};
enum EpiKind { EPI_REQUANT = 0, EPI_GELU = 1 };
constexpr int32_t kOutI8InF16 = 108;  // the out_bits 8 values stored as fp16 (ILW_I8_IN_F16)
struct EpiParams {
    EpiKind kind;
    const int32_t *bias, *mult, *shift;
    int32_t out_bits;  // 8, 16, 32, or kOutI8InF16 (EPI_REQUANT)
    void *C;
    int64_t ldc;
    // residual (EPI_REQUANT, out_bits 8/16)
    const int16_t *res;
    int64_t ldr, res_rows;
    int32_t m_r, s_r;
    // GELU (EPI_GELU): int8 output in C
    GeluC gelu;
    int32_t m_g, s_g;
};

// Packed weight layout: the same integers as fp16 [N, K] (row-major), the tensor-core operand.
inline size_t packed_weight_bytes(int32_t N, int32_t K) { return (size_t)N * K * 2; }
inline const int8_t *packed_i8(const void *) { return nullptr; }
inline const void *packed_f16(const void *p, int32_t, int32_t) { return p; }
cudaError_t launch_pack_weight(const int8_t *W, int32_t N, int32_t K, void *packed, cudaStream_t s);
// tcgen05 tensor-core GEMM (exact integer via fp16 operands, fp32 TMEM accumulators)
cudaError_t launch_gemm(const GemmProblem &gp, const EpiParams &ep, cudaStream_t s);
// Test hook of the bounded waits (ilwdetr_debug_gemm_wait): later GEMM launches skip the load of
// K-block counter `skip` (-1: none) and bound every wait by `cycles` (0: the default, about 1 s).
void gemm_set_debug_wait(int32_t skip, long long cycles);

// ---------------------------------------------------------------- row / element kernels
struct ShiftmaxC {
    ShiftExpC se;
    int32_t s_d, m_p, M_hw, k_out;
};
cudaError_t launch_shiftmax_rows(const int32_t *X, int64_t ldx, int64_t rows, int32_t len,
                                 const ShiftmaxC &c, uint8_t *P, int64_t ldp, cudaStream_t s);
cudaError_t launch_sdshiftgelu(const int32_t *X, int32_t *Y, int64_t n, const GeluC &c, cudaStream_t s);
struct LnParams {
    const void *X;
    int32_t in_bits;
    int64_t ldx, rows;
    int32_t C;
    const int32_t *beta, *mult, *shift;
    int32_t iters;
    void *Y;
    int32_t out_bits;
    int64_t ldy;
};
cudaError_t launch_layernorm(const LnParams &p, cudaStream_t s);

// ---------------------------------------------------------------- attention
struct AttnParams {
    const void *Q, *K, *V;  // int8, or fp16 when qkv_f16 (the same integers)
    int64_t ld_qkv;         // elements
    int32_t qkv_f16;
    int32_t B, T, H, dh;
    int32_t nw;        // windows per side (1 = global)
    int32_t grid_side; // sqrt(T) when nw > 1
    ShiftmaxC smx;
    int32_t m_o, s_o;
    void *O;           // int8, or fp16 holding the int8 values when o_f16
    int32_t o_f16;
    int64_t ld_o;      // elements
    int *status;       // device status word (set by launch_attention)
};
cudaError_t launch_attention(const AttnParams &p, cudaStream_t s);
// The tensor-memory (tcgen05) form for dh = 64 with fp16-carried q|k|v, 16-byte aligned rows and
// windows of side <= 128; cudaErrorNotSupported when the problem is outside that.
cudaError_t launch_attention_tc(const AttnParams &p, cudaStream_t s);

// ---------------------------------------------------------------- deformable sampling
struct DeformParams {
    const int8_t *value;
    int32_t L;
    int32_t lh[8], lw[8];
    int64_t lstart[8];
    int64_t S_total;
    const int32_t *ref, *off;
    const uint8_t *w;
    int32_t B, Q, H, P, dh;
    int32_t m, s;
    int8_t *out;
};
cudaError_t launch_deform(const DeformParams &p, cudaStream_t s);

// ---------------------------------------------------------------- patch embedding
cudaError_t launch_patchify(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                            int8_t *A, cudaStream_t s);
cudaError_t launch_patchify_f16(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww, int32_t p,
                                __half *A, cudaStream_t s);

// ---------------------------------------------------------------- detection head, two-stage selection
cudaError_t launch_int_sigmoid(const int32_t *X, int32_t *Y, int64_t n, const ShiftExpC &se, int32_t k_out,
                               cudaStream_t s);
cudaError_t launch_relu_i8(const int8_t *X, int8_t *Y, int64_t n, cudaStream_t s);
cudaError_t launch_ivit_shiftgelu(const int32_t *X, int64_t ldx, int64_t rows, int32_t L, int32_t *Y, int64_t ldy,
                                  const GeluC &c, cudaStream_t s);
cudaError_t launch_topk(const int32_t *S, int64_t lds, int32_t rows, int32_t N, int32_t K, int32_t *vals,
                        int32_t *idx, cudaStream_t s);
cudaError_t launch_gather_rows(const void *src, int64_t src_ld_bytes, int64_t src_rows, const int32_t *idx, int64_t n,
                               int64_t row_bytes, void *dst, int64_t dst_ld_bytes, cudaStream_t s);

// ---------------------------------------------------------------- detector: requantisation, resampling
struct RequantParams {
    const void *X;       // int16 or int32 [rows, ldx]
    int32_t in_bits;     // 16 or 32
    int64_t ldx, rows;
    int32_t C;           // multiple of 4
    int32_t m1, s1;
    const int16_t *Z;    // optional second term [z_rows, ldz], row r uses r % z_rows
    int64_t ldz, z_rows;
    int32_t m2, s2;
    int32_t out_bits;    // 8, 16 (saturating) or 32
    void *Y;
    int64_t ldy;
};
cudaError_t launch_requant(const RequantParams &p, cudaStream_t s);
cudaError_t launch_resample(const int8_t *X, int64_t x_bstride, int32_t B, int32_t Hi, int32_t Wi, int32_t C,
                            int8_t *Y, int64_t y_bstride, int32_t Ho, int32_t Wo, cudaStream_t s);
// Attention heads of dh < 64 widened to 64 columns for the tensor-memory attention (zero columns
// add nothing to q.k and give zero outputs): nh heads of int8 rows -> fp16-carried [M, nh 64]; and
// the int8 outputs narrowed back to dh columns per head.
cudaError_t launch_head_pad64(const int8_t *X, int64_t ldx, int64_t M, int32_t nh, int32_t dh, __half *Y,
                              cudaStream_t s);
cudaError_t launch_head_compact(const int8_t *Y, int64_t ldy, int64_t M, int32_t H, int32_t dh, int8_t *O, int64_t ldo,
                                cudaStream_t s);

}  // namespace ilw
