#pragma once
// gemm_tc.cuh -- exact integer GEMM on the 5th-generation tensor cores (tcgen05.mma, sm_103a)
// with the bias / dyadic requantisation / residual / SD-ShiftGELU / split-convolution epilogues
// fused (Sec. 3.2.1, 3.2.2, 3.3.1).
//
// Exactness.  sm_103a has no int8 tcgen05 MMA, so the int8 values are carried in fp16 (every
// integer of magnitude <= 2048 is exact in fp16) and multiplied by tcgen05.mma.kind::f16 with
// fp32 accumulation in tensor memory.  Each product |a w| <= 127^2 < 2^14 is exact, and every
// partial sum of an accumulator is an integer of magnitude <= 127^2 * 1024 < 2^24, exactly
// representable in fp32, so the accumulation is exact as long as one accumulator never sees more
// than 1024 terms of K.  Longer K is cut into segments of <= 1024, each with its own TMEM
// accumulator; the epilogue converts every segment to int32 (exact) and adds them in integers.
// Split-convolution branches are segments too, each rescaled by its own dyadic (m_b, s_b)
// before the integer sum.
//
// Persistent kernel, one CTA per SM, 128 x BN output tiles, 14 warps:
//   warp 0      TMA producer: per K stage the activation tile (int8 128 x 64 bytes, or, when A is
//               carried in fp16, the fp16 128 x 64 tile in the MMA's 128-byte swizzled layout) and
//               the fp16 weight tile (BN x 64, 128-byte swizzle); with resident weights the CTA's
//               BN rows of W are loaded once, before its first tile; TMEM allocation
//   warp 1      MMA issuer (one thread): 4 x (128 x BN x 16) MMAs per 64-wide K stage
//   warps 2-5   operand converters (int8 A only): int8 activation rows (smem) -> fp16 rows in the
//               same 128-byte swizzled K-major layout TMA produces for the weights
//   warps 6-13  epilogue: TMEM -> registers -> integer epilogue -> HBM, one row per thread and
//               half of the tile's columns per warp (fp16 A with 192-wide tiles: warps 2-13, a
//               third of the columns each, since there is nothing to convert)
// Two TMEM accumulator sets (when they fit) let the epilogue of tile i overlap the MMAs of tile
// i+1.  With resident weights the grid is a multiple of the number of column blocks, so every
// tile of a CTA uses the same BN rows of W and L2 serves only the activations.
// Every mbarrier wait is bounded (about one second); on expiry the kernel latches the device
// status word, stops issuing work, drains the loads it issued and frees its TMEM.
#include <cuda.h>

#include <algorithm>
#include <climits>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <type_traits>

#include "ilw_kernels.h"

namespace ilw {
// Host helpers of the tensor-core GEMM shared by its translation units (defined in gemm_tc.cu).
bool gemm_make_map(CUtensorMap *m, const void *base, CUtensorMapDataType dt, int esize, int64_t rows, int64_t cols,
                   int64_t ld, int box_cols, int box_rows, CUtensorMapSwizzle sw);
const int8_t *gemm_gelu_table(const GeluC &c, int32_t m_g, int32_t s_g, cudaStream_t s, cudaError_t *err);
// The wait bound of the next GEMM launches and the K block whose load the producer skips (-1: none),
// as set by ilwdetr_debug_gemm_wait (defaults: about one second, none).
void gemm_debug_wait(int32_t *skip, long long *cycles);
struct GemmProblem;
struct EpiParams;
// The int8-A launch shapes (gemm_tc_i8.cu): run<BN, STAGES, NB, false, false, GELU>.
template <int BN, int STAGES, int NB, bool GELU>
cudaError_t run_i8(const GemmProblem &gp, const EpiParams &ep, cudaStream_t s);
namespace {

constexpr int BM = 128, BK = 64;
constexpr int kThreads = 448;
constexpr int kMaxSeg = 8;
constexpr int kSegK = 1024;  // max K per accumulator for exact fp32 accumulation
constexpr int kMaxWk = kSegK / 64;  // K blocks of resident weights (one barrier each)
constexpr int kStageBytes = 1024;   // per epilogue warp: the 32 x 16 output box of the TMA store
constexpr long long kWaitCycles = 2000000000ll;  // ~1 s at 2 GHz: the default bound of every wait

struct Seg {
    int32_t k0, klen;   // K range of this accumulator (same columns of A and W)
    int32_t map;        // index of the activation / weight tensor maps
    int32_t m_b, s_b;   // split-conv rescale of the branch partial
};

template <int NB>  // NB: tensor-map slots (1 for a plain GEMM, kMaxBranches for split convolution)
struct TcParams {  // CUtensorMap members keep the 64-byte alignment TMA needs
    CUtensorMap amap[NB];
    CUtensorMap wmap[NB];
    Seg seg[kMaxSeg];
    int32_t nseg;
    int32_t branch_rq;
    int32_t M, N;
    int32_t tiles_n, tiles;
    int32_t nbuf;       // TMEM accumulator sets (1 or 2)
    int32_t wres_bytes; // resident weight bytes (WRES), a multiple of 1024
    int32_t tmem_cols;
    int32_t tma_store;  // 1: outputs go out by TMA tensor stores of 32 x 16 boxes through shared memory
    int32_t dbg_skip;   // test hook: the producer issues no load for this K-block counter value (-1: none)
    long long wait_cycles;  // the bound of every wait (about one second, shorter for the test hook)
    CUtensorMap cmap;   // C [M, N] with 16 x 32 boxes (2-byte outputs: 32-byte swizzle)
    const int8_t *gelu_tab;  // SD-ShiftGELU output table in global memory (16-byte aligned, 65536 bytes)
    int *status;
    EpiParams ep;
};

// ------------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
// One try_wait; the waiting thread may be suspended (up to the hint, 20 us) until the phase completes,
// so that waiting roles do not spin on the issue slots the epilogue needs.
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred P;\n mbarrier.try_wait.parity.shared::cta.b64 P, [%1], %2, %3;\n selp.b32 %0, 1, 0, P;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(20000)
        : "memory");
    return ok != 0;
}
// Bounded wait: true when the phase completed; false (after latching `code` in the status word
// and raising the CTA's abort flag) when it ran out, or when another role already aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort, int *status, int code,
                                          long long limit) {
    if (mbar_try(bar, parity)) return true;  // the common case, without reading the clock
    long long t0 = clock64();
    for (uint32_t i = 0;; ++i) {
        if (mbar_try(bar, parity)) return true;
        if ((i & 255) == 255) {
            if (*abort) return false;
            if (clock64() - t0 > limit) {
                if (status) atomicExch(status, code);
                *abort = 1;
                return false;
            }
        }
    }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int32_t x, int32_t y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"((uint64_t)map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, int32_t x, int32_t y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"((uint64_t)map),
                 "r"(x), "r"(y), "r"(src)
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem_g() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void tma_store_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void tma_store_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1 << 16;             // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024 >> 4) << 32;   // stride byte offset: next 8-row group
    d |= (uint64_t)1 << 46;             // descriptor version
    d |= (uint64_t)2 << 61;             // 128-byte swizzle
    return d;
}

__device__ __forceinline__ void tc_mma(uint32_t dtmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(dtmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(acc)
        : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
          "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr));
}
// Waits for this thread's TMEM loads and marks the 16 destination registers as written by the
// wait, so that no use of them can be scheduled before the data has arrived.
__device__ __forceinline__ void tmem_wait_ld16(uint32_t (&v)[16]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                   "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15])
                 :
                 : "memory");
}

// TMEM load of 32 consecutive 32-bit columns of this thread's lane, and the matching wait (every
// destination register marked as written by the wait).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t *v) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
          "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
          "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
          "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_mark32(uint32_t *v) {
    asm volatile(""
                 : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                   "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15]),
                   "+r"(v[16]), "+r"(v[17]), "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]), "+r"(v[22]),
                   "+r"(v[23]), "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]), "+r"(v[29]),
                   "+r"(v[30]), "+r"(v[31])::"memory");
}
__device__ __forceinline__ void tmem_wait_only() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 4 int8 (one word) -> 2 words of fp16x2, exact: fp16 bits 0x6400 | (b ^ 0x80) encode 1152 + b.
__device__ __forceinline__ void i8x4_to_f16x4(uint32_t w, uint32_t &lo, uint32_t &hi) {
    const uint32_t x = w ^ 0x80808080u;
    uint32_t a = __byte_perm(x, 0x64646464u, 0x4140);
    uint32_t b = __byte_perm(x, 0x64646464u, 0x4342);
    const __half2 k1152 = __half2half2(__ushort_as_half((unsigned short)0x6480));
    __half2 ha = __hsub2(*reinterpret_cast<__half2 *>(&a), k1152);
    __half2 hb = __hsub2(*reinterpret_cast<__half2 *>(&b), k1152);
    lo = *reinterpret_cast<uint32_t *>(&ha);
    hi = *reinterpret_cast<uint32_t *>(&hb);
}

// Shared memory per pipeline stage: fp16 A (128 rows x 128 B, swizzled; written by the converter
// warps from the int8 staging rows, or by TMA directly when A arrives as fp16), fp16 W (BN rows x
// 128 B, swizzled by TMA; absent when the CTA's weights are resident), int8 A staging (128 rows x
// 64 B, written by TMA; absent for fp16 A).  Resident weights (WRES) keep every K block of the
// CTA's BN rows of W after the stages.
template <int BN, bool AF16 = false, bool WRES = false>
struct Smem {
    static constexpr int kA16 = BM * 128;
    static constexpr int kW = WRES ? 0 : BN * 128;
    static constexpr int kA8 = AF16 ? 0 : BM * 64;
    static constexpr int kStage = kA16 + kW + kA8;
    static constexpr int kWtile = BN * 128;  // one K block of W
};

// Output kinds: one compact epilogue per kernel instantiation.
// F16OUT: RQ8 values as fp16; GELU_F16: GELU8 values as fp16
enum { KIND_RQ8 = 0, KIND_RQ16 = 1, KIND_RAW32 = 2, KIND_GELU8 = 3, KIND_F16OUT = 4, KIND_GELU_F16 = 5 };
constexpr bool gelu_kind(int kind) { return kind == KIND_GELU8 || kind == KIND_GELU_F16; }

// 16 consecutive int32 of shared memory (16-byte aligned) into registers: four 128-bit loads
__device__ __forceinline__ void lds16(const int32_t *p, int32_t (&o)[16]) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
#pragma unroll
    for (int j = 0; j < 4; ++j)
        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                     : "=r"(o[4 * j]), "=r"(o[4 * j + 1]), "=r"(o[4 * j + 2]), "=r"(o[4 * j + 3])
                     : "r"(a + 16 * j));
}

// The fused epilogue of 16 consecutive columns of one row, computed stage by stage so that the
// 16 independent elements overlap.  FAST (uniform across the warp, decided per tile) says every
// shift of the warp's columns is >= 33; ss then holds s - 32 and sr 2^(s-33) (rq_hi), else ss
// holds s.  RFAST: the residual's shift s_r is >= 17.  gtab points at entry 0 of the SD-ShiftGELU output table (index -32767 .. 32767).
template <int KIND, bool FAST, bool RFAST>
__device__ __forceinline__ void epi_chunk(const EpiParams &ep, bool has_res, const uint32_t (&rp)[8],
                                          const int32_t (&acc)[16], const int32_t (&sb)[16],
                                          const int32_t (&sm)[16], const int32_t (&ss)[16],
                                          const int32_t (&sr)[16], const int8_t *gtab, int32_t (&out)[16]) {
    if (KIND == KIND_RAW32) {
#pragma unroll
        for (int i = 0; i < 16; ++i) out[i] = acc[i] + sb[i];
        return;
    }
    int32_t r[16];
    if (FAST) {
#pragma unroll
        for (int i = 0; i < 16; ++i) r[i] = rq_hi(acc[i] + sb[i], sm[i], sr[i], ss[i]);  // |r| < 2^29
    } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int64_t t = rq((int64_t)acc[i] + sb[i], sm[i], ss[i]);
            r[i] = (int32_t)(t < -(1 << 30) ? -(1 << 30) : (t > (1 << 30) ? (1 << 30) : t));  // saturates the same
        }
    }
    if (KIND == KIND_GELU8 || KIND == KIND_GELU_F16) {
        // g = sat16(r); the table holds sat8(rq(g * I_div(g); m_g, s_g)) for every int16 g
#pragma unroll
        for (int i = 0; i < 16; ++i) out[i] = gtab[clamp16(r[i])];
        return;
    }
    if (has_res) {
        // rp holds the 16 int16 residuals in pairs; x * 2^16 is the pair word masked or shifted
        // (RFAST: rq(x; m_r, s_r) = rq(x * 2^16; m_r, s_r + 16) with s_r + 16 >= 33)
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int32_t xs = (i & 1) ? (int32_t)(rp[i >> 1] & 0xFFFF0000u) : (int32_t)(rp[i >> 1] << 16);
            r[i] += RFAST ? rq_hi(xs, ep.m_r, 1 << (ep.s_r - 17), ep.s_r - 16) : (int32_t)rq((int64_t)(xs >> 16), ep.m_r, ep.s_r);
        }
    }
#pragma unroll
    for (int i = 0; i < 16; ++i) out[i] = (KIND == KIND_RQ8 || KIND == KIND_F16OUT) ? clamp8(r[i]) : clamp16(r[i]);
}

// Stores 16 epilogue outputs of one row (out[i] for columns c0 + i) at dst: 16-byte vector stores
// when all 16 columns exist and dst is 16-byte aligned, else element by element (ncol columns).
template <int KIND>
__device__ __forceinline__ void store16(char *dst, const int32_t (&out)[16], int ncol, bool vec) {
    constexpr int bits = (KIND == KIND_RQ16 || KIND == KIND_F16OUT || KIND == KIND_GELU_F16) ? 16 : (KIND == KIND_RAW32 ? 32 : 8);
    if constexpr (KIND == KIND_F16OUT || KIND == KIND_GELU_F16) {
        // |v| <= 127: the fp16 bits of 1152 + v are 0x6480 + v; one half2 subtract of 1152 leaves v exactly
        const __half2 k1152 = __half2half2(__ushort_as_half((unsigned short)0x6480));
        uint32_t hw[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            uint32_t x = (uint32_t)(0x6480 + out[2 * j]) | ((uint32_t)(0x6480 + out[2 * j + 1]) << 16);
            __half2 h = __hsub2(*reinterpret_cast<__half2 *>(&x), k1152);
            hw[j] = *reinterpret_cast<uint32_t *>(&h);
        }
        if (vec) {
            ((uint4 *)dst)[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            ((uint4 *)dst)[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (i < ncol) ((uint16_t *)dst)[i] = (uint16_t)((i & 1) ? hw[i >> 1] >> 16 : hw[i >> 1]);
        }
    } else if constexpr (bits == 8) {
        if (vec) {
            uint32_t w[4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
                w[u] = (uint32_t)(uint8_t)out[4 * u] | ((uint32_t)(uint8_t)out[4 * u + 1] << 8) |
                       ((uint32_t)(uint8_t)out[4 * u + 2] << 16) | ((uint32_t)(uint8_t)out[4 * u + 3] << 24);
            *(uint4 *)dst = make_uint4(w[0], w[1], w[2], w[3]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (i < ncol) ((int8_t *)dst)[i] = (int8_t)out[i];
        }
    } else if constexpr (bits == 16) {
        if (vec) {
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                uint32_t w[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    w[u] = (uint32_t)(uint16_t)out[8 * j + 2 * u] | ((uint32_t)(uint16_t)out[8 * j + 2 * u + 1] << 16);
                ((uint4 *)dst)[j] = make_uint4(w[0], w[1], w[2], w[3]);
            }
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (i < ncol) ((int16_t *)dst)[i] = (int16_t)out[i];
        }
    } else {
        if (vec) {
#pragma unroll
            for (int j = 0; j < 4; ++j) ((int4 *)dst)[j] = make_int4(out[4 * j], out[4 * j + 1], out[4 * j + 2], out[4 * j + 3]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (i < ncol) ((int32_t *)dst)[i] = out[i];
        }
    }
}

// 16 epilogue outputs of one row into row `lane` of the warp's 32 x 16 TMA-store box: 2-byte outputs
// (fp16-carried int8, int16) as two 16-byte halves in the 32-byte swizzle the tensor map declares
// (half j of row r at ((j ^ ((r >> 2) & 1)) << 4): no bank conflicts), 1-byte outputs as one 16-byte row.
template <int KIND>
__device__ __forceinline__ void box_row16(uint8_t *box, int lane, const int32_t (&out)[16]) {
    if constexpr (KIND == KIND_F16OUT || KIND == KIND_GELU_F16) {
        const __half2 k1152 = __half2half2(__ushort_as_half((unsigned short)0x6480));
        uint32_t hw[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            uint32_t x = (uint32_t)(0x6480 + out[2 * j]) | ((uint32_t)(0x6480 + out[2 * j + 1]) << 16);
            __half2 h = __hsub2(*reinterpret_cast<__half2 *>(&x), k1152);
            hw[j] = *reinterpret_cast<uint32_t *>(&h);
        }
        const int sw = (lane >> 2) & 1;
        *(uint4 *)(box + lane * 32 + (sw << 4)) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *(uint4 *)(box + lane * 32 + ((sw ^ 1) << 4)) = make_uint4(hw[4], hw[5], hw[6], hw[7]);
    } else if constexpr (KIND == KIND_RQ16) {
        uint32_t w[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) w[j] = (uint32_t)(uint16_t)out[2 * j] | ((uint32_t)(uint16_t)out[2 * j + 1] << 16);
        const int sw = (lane >> 2) & 1;
        *(uint4 *)(box + lane * 32 + (sw << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
        *(uint4 *)(box + lane * 32 + ((sw ^ 1) << 4)) = make_uint4(w[4], w[5], w[6], w[7]);
    } else {
        uint32_t w[4];
#pragma unroll
        for (int u = 0; u < 4; ++u)
            w[u] = (uint32_t)(uint8_t)out[4 * u] | ((uint32_t)(uint8_t)out[4 * u + 1] << 8) |
                   ((uint32_t)(uint8_t)out[4 * u + 2] << 16) | ((uint32_t)(uint8_t)out[4 * u + 3] << 24);
        *(uint4 *)(box + lane * 16) = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// Waits for this thread's TMEM loads; every register of v is marked as written by the wait.
template <int NSEG>
__device__ __forceinline__ void tmem_wait_all(uint32_t (&v)[NSEG][16]) {
    tmem_wait_ld16(v[0]);
#pragma unroll
    for (int sg = 1; sg < NSEG; ++sg)
        asm volatile(""
                     : "+r"(v[sg][0]), "+r"(v[sg][1]), "+r"(v[sg][2]), "+r"(v[sg][3]), "+r"(v[sg][4]), "+r"(v[sg][5]),
                       "+r"(v[sg][6]), "+r"(v[sg][7]), "+r"(v[sg][8]), "+r"(v[sg][9]), "+r"(v[sg][10]), "+r"(v[sg][11]),
                       "+r"(v[sg][12]), "+r"(v[sg][13]), "+r"(v[sg][14]), "+r"(v[sg][15])::"memory");
}

// The epilogue of one warp's part of a tile (its 32 rows x HALF columns) in the common case: a
// plain GEMM whose K is split into NSEG accumulators (compile-time), and one dyadic shift s >= 33
// shared by all the part's columns (checked per tile by the caller), so rq(v; m, s) =
// mad.hi(v, m, 2^(s-33)) >> (s - 32) with a scalar rounding constant and shift.  The part's
// accumulators are read from TMEM in 32-column groups (all of them at once for one segment), so the
// accumulator set is released to the MMA warp after the first wait, and the requantisation of the
// 16-column chunks that follows has no TMEM latency left in it.  RES: the two-term residual form
// (s_r >= 17); rp holds the residual pairs of group 0 (fetched by the caller while the MMAs ran), and
// each later group's pairs are fetched before its TMEM loads.
// The residual pairs (x[2j] | x[2j+1] << 16) of 32 columns of a row starting at rrow + c0 (columns
// at or past ncol read as 0; rvec: 16-byte aligned and all 32 present).
__device__ __forceinline__ void res_group(const int16_t *rrow, int c0, int ncol, bool rvec, uint32_t (&rp)[16]) {
    if (rrow && rvec && c0 + 32 <= ncol) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint4 a = __ldg((const uint4 *)(rrow + c0) + j);
            rp[4 * j] = a.x; rp[4 * j + 1] = a.y; rp[4 * j + 2] = a.z; rp[4 * j + 3] = a.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            const int cl = c0 + 2 * j;
            const uint32_t lo = (rrow && cl < ncol) ? (uint16_t)rrow[cl] : 0u;
            const uint32_t hi = (rrow && cl + 1 < ncol) ? (uint16_t)rrow[cl + 1] : 0u;
            rp[j] = lo | (hi << 16);
        }
    }
}

// box: this warp's TMA-store box (nullptr: plain stores at dst), written out at column x0 + 16 c, row
// y0 of cmap by lane 0 once every lane has written its row; the box is rewritten only after the
// previous store has read it (that wait comes after the next chunk's arithmetic).
template <int KIND, int BN, int HALF, int NSEG, bool RES>
__device__ __forceinline__ void epi_fast(const EpiParams &ep, uint32_t tbase, const int32_t *s_bias,
                                         const int32_t *s_mult, int32_t rnd, int32_t sh, uint32_t (&rp)[16],
                                         const int16_t *rrow, bool rvec, char *dst, int ncol_row, bool vec_ok,
                                         const int8_t *gt, uint32_t empty_bar, int lane, uint8_t *box,
                                         const CUtensorMap *cmap, int x0, int y0) {
    static_assert(HALF % 32 == 0, "32-column groups");
    constexpr int NG = HALF / 32;                    // 32-column groups of the part
    // groups read per TMEM pass (32 registers per group and segment): the whole part for one segment
    // without a residual, one group otherwise (the residual's pairs take 32 registers)
    constexpr int GPASS = (NSEG == 1 && !RES) ? NG : 1;
    constexpr int esz = (KIND == KIND_RQ16 || KIND == KIND_F16OUT || KIND == KIND_GELU_F16) ? 2 : (KIND == KIND_RAW32 ? 4 : 1);
    const int32_t r_rnd = RES ? 1 << (ep.s_r - 17) : 0, r_sh = RES ? ep.s_r - 16 : 0;
#pragma unroll
    for (int g0 = 0; g0 < NG; g0 += GPASS) {
        if constexpr (RES) {  // this group's residual pairs (group 0's came with the call), in flight during the TMEM wait
            if (g0 > 0) res_group(rrow, 32 * g0, ncol_row, rvec, rp);
        }
        uint32_t v[NSEG][GPASS * 32];
#pragma unroll
        for (int gg = 0; gg < GPASS; ++gg)
#pragma unroll
            for (int sg = 0; sg < NSEG; ++sg) tmem_ld32(tbase + (uint32_t)(sg * BN + 32 * (g0 + gg)), v[sg] + 32 * gg);
        tmem_wait_only();
#pragma unroll
        for (int gg = 0; gg < GPASS; ++gg)
#pragma unroll
            for (int sg = 0; sg < NSEG; ++sg) tmem_mark32(v[sg] + 32 * gg);
        if (g0 + GPASS >= NG) {  // every TMEM read of this warp in this accumulator set is done
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(empty_bar);
        }
        // the integer accumulators (exact: every partial sum is below 2^24), in place
#pragma unroll
        for (int i = 0; i < GPASS * 32; ++i) {
            int32_t a = __float2int_rn(__uint_as_float(v[0][i]));
#pragma unroll
            for (int sg = 1; sg < NSEG; ++sg) a += __float2int_rn(__uint_as_float(v[sg][i]));
            v[0][i] = (uint32_t)a;
        }
#pragma unroll
        for (int cc = 0; cc < GPASS * 2; ++cc) {
            const int c = 2 * g0 + cc;  // 16-column chunk of the part
            int32_t cb[16], cm[16];
            lds16(s_bias + 16 * c, cb);
            lds16(s_mult + 16 * c, cm);
            int32_t out[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                int32_t r = rq_hi((int32_t)v[0][16 * cc + i] + cb[i], cm[i], rnd, sh);  // |r| < 2^29
                if constexpr (KIND == KIND_GELU8 || KIND == KIND_GELU_F16) {
                    out[i] = gt[clamp16(r)];
                } else {
                    if constexpr (RES) {
                        const uint32_t w = rp[8 * cc + (i >> 1)];
                        const int32_t xs = (i & 1) ? (int32_t)(w & 0xFFFF0000u) : (int32_t)(w << 16);
                        r += rq_hi(xs, ep.m_r, r_rnd, r_sh);
                    }
                    out[i] = (KIND == KIND_RQ8 || KIND == KIND_F16OUT) ? clamp8(r) : clamp16(r);
                }
            }
            if (box) {
                if (lane == 0) tma_store_wait_read();  // the previous chunk's box has been read
                __syncwarp();
                box_row16<KIND>(box, lane, out);
                fence_async_smem_g();
                __syncwarp();
                if (lane == 0 && 16 * c < ncol_row) tma_store_2d(cmap, x0 + 16 * c, y0, smem_u32(box));
            } else if (dst) {
                const int ncol = ncol_row - 16 * c;
                if (ncol > 0) store16<KIND>(dst + 16 * c * esz, out, ncol, vec_ok && ncol >= 16);
            }
        }
        __syncwarp();  // reconverge before the next warp-synchronous tcgen05 instruction
    }
}

template <int BN, int STAGES, int KIND, int NB, bool AF16, bool WRES>
__global__ void __launch_bounds__(kThreads, 1) gemm_tc_kernel(const __grid_constant__ TcParams<NB> p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    using SM = Smem<BN, AF16, WRES>;
    constexpr int kStage = SM::kStage;
    // Epilogue warps: 8 (warps 6-13, two column parts per TMEM lane quarter), or, when A arrives in
    // fp16 and the tile is 192 wide, the converters' warps too: 12 (warps 2-13, three parts of 64).
    constexpr int NP = (AF16 && BN == 192) ? 3 : 2;
    constexpr int EPI0 = NP == 3 ? 2 : 6;
    constexpr int NWE = 4 * NP;
    uint8_t *wres = smem + STAGES * kStage;  // resident weights (WRES)
    uint64_t *bars = (uint64_t *)(wres + (WRES ? p.wres_bytes : 0));
    // barriers: full[S], a_ready[S], empty[S], acc_full[2], acc_empty[2], wfull[kMaxWk] (one per K block
    // of the resident weights, so the first MMAs start as soon as their own block has landed)
    uint32_t *tmem_slot = (uint32_t *)(bars + 3 * STAGES + 5 + kMaxWk);
    volatile int *abort = (volatile int *)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t bar0 = smem_u32(bars);
    auto full = [&](int s) { return bar0 + 8u * s; };
    auto a_ready = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto empty = [&](int s) { return bar0 + 8u * (2 * STAGES + s); };
    auto acc_full = [&](int b) { return bar0 + 8u * (3 * STAGES + b); };
    auto acc_empty = [&](int b) { return bar0 + 8u * (3 * STAGES + 2 + b); };
    auto wfull = [&](int kk) { return bar0 + 8u * (3 * STAGES + 4 + kk); };
    const uint32_t drain = bar0 + 8u * (3 * STAGES + 4 + kMaxWk);  // every MMA issued has completed

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(full(s), 1);
            mbar_init(a_ready(s), 4);
            mbar_init(empty(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(acc_full(b), 1);
            mbar_init(acc_empty(b), NWE);
        }
        for (int kk = 0; kk < kMaxWk; ++kk) mbar_init(wfull(kk), 1);
        mbar_init(drain, 1);
        *abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(p.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // SD-ShiftGELU and its output requantisation depend on the int16 value g alone: the table of
    // sat8(rq(g * I_div(g); m_g, s_g)) (built once per parameter set by gelu_table_kernel) is
    // copied into shared memory here.
    int8_t *gtab = (int8_t *)((int32_t *)(((uintptr_t)(tmem_slot + 4) + 15) & ~(uintptr_t)15) + 16 * BN);
    if ((KIND == KIND_GELU8 || KIND == KIND_GELU_F16) && warp >= EPI0) {
        for (int i = threadIdx.x - 32 * EPI0; i < 65536 / 16; i += 32 * NWE)
            ((uint4 *)gtab)[i] = __ldg((const uint4 *)p.gelu_tab + i);
        asm volatile("bar.sync 1, %0;" ::"r"(32 * NWE) : "memory");  // the epilogue warps only
    }
    const int acc_cols = p.nseg * BN;  // columns of one accumulator set
    // the epilogue warps' TMA-store boxes (1024-byte aligned, after the parameters and the GELU table)
    uint8_t *stg = (uint8_t *)(((uintptr_t)gtab + (gelu_kind(KIND) ? 65536 : 0) + 1023) & ~(uintptr_t)1023);

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0) {
            int it = 0;  // global K-block counter (ring position)
            int wk = 0;  // K blocks of the resident weights issued
            bool ok = true;
            for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x) {
                const int m0 = (t / p.tiles_n) * BM, n0 = (t % p.tiles_n) * BN;
                for (int sg = 0; sg < p.nseg && ok; ++sg) {
                    const Seg &S = p.seg[sg];
                    const int nk = (S.klen + BK - 1) / BK;
                    for (int kk = 0; kk < nk; ++kk, ++it) {
                        const int s = it % STAGES;
                        const uint32_t ph = (it / STAGES) & 1;
                        if (WRES && t == (int)blockIdx.x && kk < STAGES) {
                            // the CTA's BN rows of W, resident for all of its tiles (the grid is a
                            // multiple of tiles_n, so every tile of the CTA has the same n block): the
                            // first K blocks travel with the first tile's activations of the same K block,
                            // the rest follow at once (they have shared memory of their own)
                            const int last = kk == (STAGES < nk ? STAGES : nk) - 1 ? nk - 1 : kk;
                            for (int j = kk; j <= last; ++j) {
                                mbar_expect_tx(wfull(j), (uint32_t)SM::kWtile);
                                tma_load_2d(smem_u32(wres + j * SM::kWtile), &p.wmap[0], p.seg[0].k0 + j * BK, n0,
                                            wfull(j));
                            }
                            wk = last + 1;
                        }
                        if (!mbar_wait(empty(s), ph ^ 1, abort, p.status, kStatusTimeoutFree, p.wait_cycles)) {
                            ok = false;
                            break;
                        }
                        uint8_t *st = smem + s * kStage;
                        if (it == p.dbg_skip) continue;  // test hook: this stage's barrier never completes
                        mbar_expect_tx(full(s), (AF16 ? SM::kA16 : SM::kA8) + SM::kW);
                        tma_load_2d(smem_u32(AF16 ? st : st + SM::kA16 + SM::kW), &p.amap[S.map], S.k0 + kk * BK, m0,
                                    full(s));
                        if (!WRES) tma_load_2d(smem_u32(st + SM::kA16), &p.wmap[S.map], S.k0 + kk * BK, n0, full(s));
                    }
                }
            }
            if (!ok || *abort) {  // drain the loads still in flight (bounded) before the CTA can exit
                long long t0 = clock64();
                for (int kk = 0; kk < wk; ++kk)
                    while (!mbar_try(wfull(kk), 0) && clock64() - t0 < p.wait_cycles) {
                    }
                for (int j = (it > STAGES ? it - STAGES : 0); j < it; ++j)
                    while (j != p.dbg_skip && !mbar_try(full(j % STAGES), (j / STAGES) & 1) &&
                           clock64() - t0 < p.wait_cycles) {
                    }
            }
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
            // operand descriptors from two precomputed bases: a 16-byte step of the address is 1 in
            // the descriptor's low word (shared-memory offsets stay below 256 KB, so nothing carries)
            const uint64_t a_desc0 = sw128_desc(smem_u32(smem)), w_desc0 = sw128_desc(smem_u32(wres));
            int it = 0, tl = 0, s = 0;
            uint32_t ph = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++tl) {
                const int b = tl % p.nbuf;
                const uint32_t use = (uint32_t)(tl / p.nbuf);
                if (!mbar_wait(acc_empty(b), (use & 1) ^ 1, abort, p.status, kStatusTimeoutMma, p.wait_cycles)) break;
                tc_fence_after();
                for (int sg = 0; sg < p.nseg && ok; ++sg) {
                    const Seg &S = p.seg[sg];
                    const int nk = (S.klen + BK - 1) / BK;
                    const uint32_t dt = tmem + (uint32_t)(b * acc_cols + sg * BN);
                    for (int kk = 0; kk < nk; ++kk, ++it) {
                        if (!mbar_wait(AF16 ? full(s) : a_ready(s), ph, abort, p.status,
                                       AF16 ? kStatusTimeoutTma : kStatusTimeoutOperand, p.wait_cycles) ||
                            (WRES && tl == 0 && !mbar_wait(wfull(kk), 0, abort, p.status, kStatusTimeoutTma, p.wait_cycles))) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t da = a_desc0 + (uint64_t)((s * kStage) >> 4);
                        const uint64_t dw = WRES ? w_desc0 + (uint64_t)((kk * SM::kWtile) >> 4) : da + (uint64_t)(SM::kA16 >> 4);
#pragma unroll
                        for (int k16 = 0; k16 < BK / 16; ++k16)
                            tc_mma(dt, da + 2 * k16, dw + 2 * k16, idesc, (kk > 0 || k16 > 0) ? 1u : 0u);
                        tc_commit(empty(s));
                        if (++s == STAGES) {
                            s = 0;
                            ph ^= 1u;
                        }
                    }
                }
                tc_commit(acc_full(b));  // arrives once every MMA of this tile has completed
            }
            // every MMA issued has completed before the CTA can reach the TMEM release (also after an
            // abort, when the epilogue no longer waits for the accumulators)
            tc_commit(drain);
            const long long t0 = clock64();
            while (!mbar_try(drain, 0) && clock64() - t0 < p.wait_cycles) {
            }
        }
    } else if (warp < EPI0) {
        // ---------------------------------------------------------------- operand converters
        if constexpr (!AF16) {  // fp16 A arrives in the MMA's operand layout: nothing to convert
            const int r = (warp - 2) * 32 + lane;  // row of the 128-row A tile
            const int sw = (r >> 1) & 3;           // TMA's 64-byte swizzle of the int8 staging rows
            int it = 0;
            for (int t = blockIdx.x; t < p.tiles; t += gridDim.x) {
                for (int sg = 0; sg < p.nseg; ++sg) {
                    const int nk = (p.seg[sg].klen + BK - 1) / BK;
                    for (int kk = 0; kk < nk; ++kk, ++it) {
                        const int s = it % STAGES;
                        const uint32_t ph = (it / STAGES) & 1;
                        if (!mbar_wait(full(s), ph, abort, p.status, kStatusTimeoutTma, p.wait_cycles)) goto conv_done;
                        uint8_t *st = smem + s * kStage;
                        const uint8_t *a8 = st + SM::kA16 + SM::kW + r * 64;
                        uint8_t *a16 = st + r * 128;
    #pragma unroll
                        for (int j = 0; j < 4; ++j) {  // 16 int8 = K elements 16j .. 16j+15
                            const uint4 v = *(const uint4 *)(a8 + 16 * (j ^ sw));
                            uint4 o0, o1;
                            i8x4_to_f16x4(v.x, o0.x, o0.y);
                            i8x4_to_f16x4(v.y, o0.z, o0.w);
                            i8x4_to_f16x4(v.z, o1.x, o1.y);
                            i8x4_to_f16x4(v.w, o1.z, o1.w);
                            *(uint4 *)(a16 + (((2 * j) ^ (r & 7)) << 4)) = o0;
                            *(uint4 *)(a16 + (((2 * j + 1) ^ (r & 7)) << 4)) = o1;
                        }
                        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                        __syncwarp();
                        if (lane == 0) mbar_arrive(a_ready(s));
                    }
                }
            }
        conv_done:;
        }
    } else {
        // ---------------------------------------------------------------- epilogue
        // NWE warps: warp w reads TMEM lanes 32q..32q+31 (q = w % 4) and owns part h of the columns
        constexpr int HALF = BN / NP;  // columns of this warp in a tile
        const int q = warp & 3, h = (warp - EPI0) >> 2;
        const EpiParams &ep = p.ep;
        int32_t *s_bias = (int32_t *)(((uintptr_t)(tmem_slot + 4) + 15) & ~(uintptr_t)15) + (warp - EPI0) * 4 * HALF;  // this warp's copy of
        int32_t *s_mult = s_bias + HALF;                                       // the tile's per-column
        int32_t *s_shift = s_mult + HALF;                                      // epilogue parameters
        int32_t *s_rnd = s_shift + HALF;                                       // (rq_hi rounding constants)
        constexpr int bits = (KIND == KIND_RQ16 || KIND == KIND_F16OUT || KIND == KIND_GELU_F16) ? 16
                             : (KIND == KIND_RAW32 ? 32 : 8);
        constexpr int PPL = HALF / 32;  // parameters per lane and per array
        constexpr bool kFastKind = KIND == KIND_RQ8 || KIND == KIND_RQ16 || KIND == KIND_F16OUT || gelu_kind(KIND);
        constexpr bool kResKind = KIND == KIND_RQ8 || KIND == KIND_RQ16;  // kinds with a residual
        // The next tile's parameters are fetched into registers while the current tile is processed.
        int32_t pb[PPL], pm[PPL], ps[PPL];
        auto fetch = [&](int t) {
            const int nn = (t % p.tiles_n) * BN + h * HALF;
#pragma unroll
            for (int k = 0; k < PPL; ++k) {
                const int col = nn + lane + 32 * k;
                const bool ok = col < p.N;
                pb[k] = (ok && ep.bias) ? __ldg(ep.bias + col) : 0;
                pm[k] = (ok && ep.mult) ? __ldg(ep.mult + col) : 0;
                ps[k] = (ok && ep.shift) ? __ldg(ep.shift + col) : 33;
            }
        };
        if (blockIdx.x < p.tiles) fetch(blockIdx.x);
        const int nseg = p.nseg, nld = (HALF / 16) * nseg;  // TMEM loads per tile
        int tl = 0;
        for (int t = blockIdx.x; t < p.tiles; t += gridDim.x, ++tl) {
            const int b = tl % p.nbuf;
            const uint32_t use = (uint32_t)(tl / p.nbuf);
            const int m0 = (t / p.tiles_n) * BM, n0 = (t % p.tiles_n) * BN + h * HALF;
            __syncwarp();  // this warp is done with the previous tile's parameters
            bool fast_lane = true, same_lane = true;
            const int32_t s_0 = __shfl_sync(0xffffffffu, ps[0], 0);
#pragma unroll
            for (int k = 0; k < PPL; ++k) {
                fast_lane &= ps[k] >= 33;
                same_lane &= ps[k] == s_0;
            }
            const bool fastw = __all_sync(0xffffffffu, fast_lane);  // shifts stored as s - 32 if so
            // the common case (epi_fast): one shift >= 33 for all of this warp's columns, 1 or 2 segments
            const bool ush = kFastKind && NB == 1 && !p.branch_rq && p.nseg <= 2 && fastw &&
                             __all_sync(0xffffffffu, same_lane);
#pragma unroll
            for (int k = 0; k < PPL; ++k) {
                s_bias[lane + 32 * k] = pb[k];
                s_mult[lane + 32 * k] = pm[k];
                s_shift[lane + 32 * k] = fastw ? ps[k] - 32 : ps[k];
                s_rnd[lane + 32 * k] = fastw ? 1 << (ps[k] - 33) : 0;
            }
            __syncwarp();
            if (t + (int)gridDim.x < p.tiles) fetch(t + gridDim.x);
            const int64_t row = (int64_t)m0 + 32 * q + lane;
            const bool row_ok = row < p.M;
            // this row's residual (row modulo res_rows broadcasts a [res_rows, N] table)
            const int16_t *rrow = (ep.res && row_ok) ? ep.res + (row % ep.res_rows) * ep.ldr + n0 : nullptr;
            const bool rvec = ((uintptr_t)rrow & 15) == 0;
            const bool has_res = ep.res != nullptr;
            const bool rfast = has_res && ep.s_r >= 17;
            const uint32_t tbase = tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(b * acc_cols + h * HALF);
            if constexpr (kFastKind && NB == 1) {
                if (ush && (!has_res || rfast)) {
                    // the residuals of the first 32 columns are fetched while the MMAs run
                    uint32_t rpa[16];
#pragma unroll
                    for (int j = 0; j < 16; ++j) rpa[j] = 0;
                    if (kResKind && has_res) res_group(rrow, 0, p.N - n0, rvec, rpa);
                    if (!mbar_wait(acc_full(b), use & 1, abort, p.status, kStatusTimeoutMma, p.wait_cycles)) break;
                    tc_fence_after();
                    char *dst = row_ok ? (char *)ep.C + (row * ep.ldc + n0) * (bits / 8) : nullptr;
                    const bool vec_ok = ((uintptr_t)dst & 15) == 0;
                    const int ncol_row = p.N - n0;
                    const int32_t rnd = 1 << (s_0 - 33), sh = s_0 - 32;
                    const int8_t *gt = gtab + 32767;
                    const uint32_t eb = acc_empty(b);
                    uint8_t *box = p.tma_store ? stg + (warp - EPI0) * kStageBytes : nullptr;
                    if (p.nseg == 1) {
                        if (kResKind && has_res)
                            epi_fast<KIND, BN, HALF, 1, kResKind>(ep, tbase, s_bias, s_mult, rnd, sh, rpa, rrow, rvec, dst,
                                                                   ncol_row, vec_ok, gt, eb, lane, box, &p.cmap, n0,
                                                                   m0 + 32 * q);
                        else
                            epi_fast<KIND, BN, HALF, 1, false>(ep, tbase, s_bias, s_mult, rnd, sh, rpa, rrow, rvec, dst,
                                                               ncol_row, vec_ok, gt, eb, lane, box, &p.cmap, n0,
                                                               m0 + 32 * q);
                    } else {
                        if (kResKind && has_res)
                            epi_fast<KIND, BN, HALF, 2, kResKind>(ep, tbase, s_bias, s_mult, rnd, sh, rpa, rrow, rvec, dst,
                                                                   ncol_row, vec_ok, gt, eb, lane, box, &p.cmap, n0,
                                                                   m0 + 32 * q);
                        else
                            epi_fast<KIND, BN, HALF, 2, false>(ep, tbase, s_bias, s_mult, rnd, sh, rpa, rrow, rvec, dst,
                                                               ncol_row, vec_ok, gt, eb, lane, box, &p.cmap, n0,
                                                               m0 + 32 * q);
                    }
                    continue;
                }
            }
            if (!mbar_wait(acc_full(b), use & 1, abort, p.status, kStatusTimeoutMma, p.wait_cycles)) break;
            tc_fence_after();
            uint32_t rp[8];
            // The tile's chunks, with the requantisation forms fixed for the whole tile (a branch per
            // tile instead of both forms predicated per element).  TMEM load i reads segment i % nseg
            // of chunk i / nseg; load i+1 is in flight while the epilogue of load i's chunk runs.
            auto chunks = [&](auto fast_c, auto rfast_c) {
                constexpr bool FAST = decltype(fast_c)::value, RFAST = decltype(rfast_c)::value;
                uint32_t v[16];
                tmem_ld16(tbase, v);
                int32_t acc[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) acc[i] = 0;
                for (int li = 0; li < nld; ++li) {
                    const int c0 = (li / nseg) * 16, sg = li - (li / nseg) * nseg;
                    if (has_res && sg == 0) {  // this chunk's residuals, in flight during the TMEM wait
                        if (rrow && rvec && n0 + c0 + 16 <= p.N) {
                            const uint4 a = __ldg((const uint4 *)(rrow + c0)), b = __ldg((const uint4 *)(rrow + c0) + 1);
                            rp[0] = a.x; rp[1] = a.y; rp[2] = a.z; rp[3] = a.w;
                            rp[4] = b.x; rp[5] = b.y; rp[6] = b.z; rp[7] = b.w;
                        } else {
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                const int cl = n0 + c0 + 2 * j;
                                const uint32_t lo = (rrow && cl < p.N) ? (uint16_t)rrow[c0 + 2 * j] : 0u;
                                const uint32_t hi = (rrow && cl + 1 < p.N) ? (uint16_t)rrow[c0 + 2 * j + 1] : 0u;
                                rp[j] = lo | (hi << 16);
                            }
                        }
                    }
                    tmem_wait_ld16(v);
                    if (p.branch_rq) {
                        const int32_t mb = p.seg[sg].m_b, sbb = p.seg[sg].s_b;
#pragma unroll
                        for (int i = 0; i < 16; ++i) acc[i] += (int32_t)rq(__float2int_rn(__uint_as_float(v[i])), mb, sbb);
                    } else {
#pragma unroll
                        for (int i = 0; i < 16; ++i) acc[i] += __float2int_rn(__uint_as_float(v[i]));  // exact: < 2^24
                    }
                    if (li + 1 < nld) {
                        const int c1 = ((li + 1) / nseg) * 16, sg1 = (li + 1) - ((li + 1) / nseg) * nseg;
                        tmem_ld16(tbase + (uint32_t)(sg1 * BN + c1), v);
                    } else {  // every TMEM read of this warp in this accumulator set is done
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(acc_empty(b));
                    }
                    if (sg != nseg - 1) continue;
                    int32_t cb[16], cm[16], cs[16], cr[16];  // this chunk's per-column parameters
                    lds16(s_bias + c0, cb);
                    lds16(s_mult + c0, cm);
                    lds16(s_shift + c0, cs);
                    if (FAST) lds16(s_rnd + c0, cr);
                    const int ncol = min(16, p.N - (n0 + c0));
                    if (row_ok && ncol > 0) {
                        int32_t out[16];
                        const int8_t *gt = gtab + 32767;
                        epi_chunk<KIND, FAST, RFAST>(ep, has_res, rp, acc, cb, cm, cs, cr, gt, out);
                        char *dst = (char *)ep.C + (row * ep.ldc + n0 + c0) * (bits / 8);
                        const bool vec = ncol == 16 && (((uintptr_t)dst & 15) == 0);
                        if constexpr (KIND == KIND_F16OUT || KIND == KIND_GELU_F16) {
                            // |v| <= 127: the fp16 bits of 1152 + v are 0x6480 + v; one half2 subtract of
                            // 1152 leaves v exactly
                            const __half2 k1152 = __half2half2(__ushort_as_half((unsigned short)0x6480));
                            uint32_t hw[8];
#pragma unroll
                            for (int j = 0; j < 8; ++j) {
                                uint32_t x = (uint32_t)(0x6480 + out[2 * j]) | ((uint32_t)(0x6480 + out[2 * j + 1]) << 16);
                                __half2 h = __hsub2(*reinterpret_cast<__half2 *>(&x), k1152);
                                hw[j] = *reinterpret_cast<uint32_t *>(&h);
                            }
                            if (vec) {
                                ((uint4 *)dst)[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
                                ((uint4 *)dst)[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
                            } else {
#pragma unroll
                                for (int i = 0; i < 16; ++i)
                                    if (i < ncol) ((uint16_t *)dst)[i] = (uint16_t)((i & 1) ? hw[i >> 1] >> 16 : hw[i >> 1]);
                            }
                        } else if constexpr (bits == 8) {
                            if (vec) {
                                uint32_t w[4];
#pragma unroll
                                for (int u = 0; u < 4; ++u)
                                    w[u] = (uint32_t)(uint8_t)out[4 * u] | ((uint32_t)(uint8_t)out[4 * u + 1] << 8) |
                                           ((uint32_t)(uint8_t)out[4 * u + 2] << 16) | ((uint32_t)(uint8_t)out[4 * u + 3] << 24);
                                *(uint4 *)dst = make_uint4(w[0], w[1], w[2], w[3]);
                            } else {
#pragma unroll
                                for (int i = 0; i < 16; ++i)
                                    if (i < ncol) ((int8_t *)dst)[i] = (int8_t)out[i];
                            }
                        } else if constexpr (bits == 16) {
                            if (vec) {
#pragma unroll
                                for (int j = 0; j < 2; ++j) {
                                    uint32_t w[4];
#pragma unroll
                                    for (int u = 0; u < 4; ++u)
                                        w[u] = (uint32_t)(uint16_t)out[8 * j + 2 * u] | ((uint32_t)(uint16_t)out[8 * j + 2 * u + 1] << 16);
                                    ((uint4 *)dst)[j] = make_uint4(w[0], w[1], w[2], w[3]);
                                }
                            } else {
#pragma unroll
                                for (int i = 0; i < 16; ++i)
                                    if (i < ncol) ((int16_t *)dst)[i] = (int16_t)out[i];
                            }
                        } else {
                            if (vec) {
#pragma unroll
                                for (int j = 0; j < 4; ++j)
                                    ((int4 *)dst)[j] = make_int4(out[4 * j], out[4 * j + 1], out[4 * j + 2], out[4 * j + 3]);
                            } else {
#pragma unroll
                                for (int i = 0; i < 16; ++i)
                                    if (i < ncol) ((int32_t *)dst)[i] = out[i];
                            }
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc[i] = 0;
                    __syncwarp();  // reconverge before the next warp-synchronous tcgen05 instruction
                }
            };
            constexpr bool kRes = KIND == KIND_RQ8 || KIND == KIND_RQ16;  // kinds with a residual
            using T_ = std::true_type;
            using F_ = std::false_type;
            using R_ = std::integral_constant<bool, kRes>;
            auto go = [&](auto f, auto r) { chunks(f, r); };
            if (fastw) {
                if (kRes && rfast) go(T_{}, R_{});
                else go(T_{}, F_{});
            } else {
                if (kRes && rfast) go(F_{}, R_{});
                else go(F_{}, F_{});
            }
        }
        if (p.tma_store && lane == 0) tma_store_wait_all();  // this warp's stores are complete
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(p.tmem_cols) : "memory");
    }
}

inline int num_sms() { return sm_count(); }

// Dynamic shared memory of one instantiation (wres: resident weight bytes).
// stg: the epilogue warps' TMA-store boxes (0 without TMA stores).
template <int BN, int STAGES, int KIND, bool AF16, bool WRES>
size_t smem_bytes(int wres, int stg = 0) {
    return 1024 + (size_t)STAGES * Smem<BN, AF16, WRES>::kStage + (WRES ? wres : 0) + 8 * (3 * STAGES + 5 + kMaxWk) +
           32 + 4 * 4 * BN * 4 + (gelu_kind(KIND) ? 65536 : 0) + (stg ? 1024 + stg : 0);
}
template <int BN, bool AF16>
constexpr int epi_warps() { return 4 * ((AF16 && BN == 192) ? 3 : 2); }
constexpr size_t kSmemMax = 227 * 1024;

template <int BN, int STAGES, int KIND, int NB, bool AF16, bool WRES>
cudaError_t launch_tc(TcParams<NB> &tp, cudaStream_t s) {
    // TMA stores when the output allows them (set up by run) and their boxes fit next to the rest
    constexpr int stg = epi_warps<BN, AF16>() * kStageBytes;
    if (tp.tma_store && smem_bytes<BN, STAGES, KIND, AF16, WRES>(tp.wres_bytes, stg) > kSmemMax) tp.tma_store = 0;
    const size_t smem = smem_bytes<BN, STAGES, KIND, AF16, WRES>(tp.wres_bytes, tp.tma_store ? stg : 0);
    if (smem > kSmemMax) return cudaErrorInvalidValue;
    static SmemLimit limit;
    const cudaError_t attr_err =
        raise_smem_limit(limit, (const void *)gemm_tc_kernel<BN, STAGES, KIND, NB, AF16, WRES>, (int)kSmemMax);
    if (attr_err != cudaSuccess) return attr_err;
    int grid = tp.tiles < num_sms() ? tp.tiles : num_sms();
    if (WRES) {  // a multiple of tiles_n: every CTA keeps one n block of W
        const int tiles_m = tp.tiles / tp.tiles_n;
        int per_n = num_sms() / tp.tiles_n;
        per_n = per_n < 1 ? 1 : (per_n > tiles_m ? tiles_m : per_n);
        grid = per_n * tp.tiles_n;
    }
    gemm_tc_kernel<BN, STAGES, KIND, NB, AF16, WRES><<<grid, kThreads, smem, s>>>(tp);
    return cudaGetLastError();
}

// One launch shape: the tile width, pipeline depth, tensor-map slots, A form and weight residency;
// GELU selects the SD-ShiftGELU output kinds, otherwise the requantising / raw kinds are built.
template <int BN, int STAGES, int NB, bool AF16, bool WRES, bool GELU>
cudaError_t run(const GemmProblem &gp, const EpiParams &ep, cudaStream_t s) {
    if (gp.nb > NB || (ep.kind == EPI_GELU) != GELU) return cudaErrorInvalidValue;
    TcParams<NB> tp;
    memset(&tp, 0, sizeof(tp));
    tp.M = gp.M;
    tp.N = gp.N;
    tp.branch_rq = gp.branch_rq ? 1 : 0;
    tp.ep = ep;
    tp.status = status_word_ptr();
    int nseg = 0;
    for (int b = 0; b < gp.nb; ++b) {
        const GemmBranch &br = gp.br[b];
        const bool amap_ok =
            AF16 ? gemm_make_map(&tp.amap[b], br.A, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, gp.M, br.K, br.lda, BK, BM,
                            CU_TENSOR_MAP_SWIZZLE_128B)
                 : gemm_make_map(&tp.amap[b], br.A, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, gp.M, br.K, br.lda, BK, BM,
                            CU_TENSOR_MAP_SWIZZLE_64B);
        if (!amap_ok ||
            !gemm_make_map(&tp.wmap[b], br.Wp, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, gp.N, br.K, br.K, BK, BN,
                      CU_TENSOR_MAP_SWIZZLE_128B))
            return cudaErrorInvalidValue;
        // cut K into near-equal segments of at most kSegK (multiples of 64)
        const int parts = (br.K + kSegK - 1) / kSegK;
        if (gp.branch_rq && parts != 1) return cudaErrorInvalidValue;
        const int per = ((br.K + parts - 1) / parts + BK - 1) / BK * BK;
        for (int k0 = 0; k0 < br.K; k0 += per) {
            if (nseg >= kMaxSeg) return cudaErrorInvalidValue;
            Seg &S = tp.seg[nseg++];
            S.k0 = k0;
            S.klen = min(per, br.K - k0);
            S.map = b;
            S.m_b = br.m_b;
            S.s_b = br.s_b;
        }
    }
    tp.nseg = nseg;
    tp.tiles_n = (gp.N + BN - 1) / BN;
    tp.tiles = ((gp.M + BM - 1) / BM) * tp.tiles_n;
    const int one = nseg * BN;
    tp.nbuf = 2 * one <= 512 ? 2 : 1;
    int alloc = 32;
    while (alloc < tp.nbuf * one) alloc <<= 1;
    if (alloc > 512) return cudaErrorInvalidValue;
    tp.tmem_cols = alloc;
    gemm_debug_wait(&tp.dbg_skip, &tp.wait_cycles);
    // TMA tensor stores of the outputs: 16 x 32 boxes of C (1-byte outputs: 16-byte box rows; 2-byte
    // outputs: 32-byte rows in the 32-byte swizzle), for a C whose rows start on 16-byte boundaries
    tp.tma_store = 0;
    if (NB == 1 && ep.out_bits != 32) {
        const int esz = ep.out_bits == 8 ? 1 : 2;  // int8, or int16 / fp16-carried int8
        if (((uintptr_t)ep.C % 16) == 0 && (ep.ldc * esz) % 16 == 0 && gp.N * esz >= 16)
            tp.tma_store = gemm_make_map(&tp.cmap, ep.C, esz == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_UINT16,
                                         esz, gp.M, gp.N, ep.ldc, 16, 32,
                                         esz == 1 ? CU_TENSOR_MAP_SWIZZLE_NONE : CU_TENSOR_MAP_SWIZZLE_32B)
                               ? 1
                               : 0;
    }
    if (WRES) {
        if (nseg != 1) return cudaErrorInvalidValue;
        tp.wres_bytes = ((tp.seg[0].klen + BK - 1) / BK) * Smem<BN, AF16, WRES>::kWtile;
    }
    if (ep.kind == EPI_GELU) {
        cudaError_t e = cudaSuccess;
        tp.gelu_tab = gemm_gelu_table(ep.gelu, ep.m_g, ep.s_g, s, &e);
        if (!tp.gelu_tab) return e != cudaSuccess ? e : cudaErrorUnknown;
    }
    if constexpr (GELU) {
        if constexpr (NB == 1)
            return ep.out_bits == kOutI8InF16 ? launch_tc<BN, STAGES, KIND_GELU_F16, NB, AF16, WRES>(tp, s)
                                              : launch_tc<BN, STAGES, KIND_GELU8, NB, AF16, WRES>(tp, s);
        else
            return cudaErrorInvalidValue;  // split convolutions requantise only
    } else {
        if (ep.out_bits == kOutI8InF16) {
            if constexpr (NB == 1) return launch_tc<BN, STAGES, KIND_F16OUT, NB, AF16, WRES>(tp, s);
            else return cudaErrorInvalidValue;
        }
        if (ep.out_bits == 8) return launch_tc<BN, STAGES, KIND_RQ8, NB, AF16, WRES>(tp, s);
        if (ep.out_bits == 16) return launch_tc<BN, STAGES, KIND_RQ16, NB, AF16, WRES>(tp, s);
        return launch_tc<BN, STAGES, KIND_RAW32, NB, AF16, WRES>(tp, s);
    }
}

}  // namespace
}  // namespace ilw
