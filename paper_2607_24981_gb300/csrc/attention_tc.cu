// attention_tc.cu -- fused integer attention on the 5th-generation tensor cores: scores = q k^T
// (tcgen05, fp32 accumulators in TMEM), Constrained Shiftmax (Algorithm 2) on the scores read back
// from TMEM, O = P V (tcgen05, accumulated in TMEM), requantisation (Sec. 3.2.1, 3.3.2).
//
// ShiftExp floors its input, so the row maximum must be known before any exponential: the keys
// of the attention group are streamed three times (pass 1: exact row max, pass 2: exact int64
// sum of ShiftExp, which fixes s_d and F; pass 3: P and P V).  Every score |q.k| <= 64 * 127^2 <
// 2^20 and every partial sum of P V (<= 256 * 127 in magnitude) is an integer below 2^24, so the
// fp32 accumulation of the fp16-carried integers is exact.
//
// One CTA = 128 queries of one (image, head, group), 12 warps, two CTAs per SM:
//   warp 0      TMEM allocation; MMA issuer (one thread): per key block of 128, 4 MMAs
//               128 x 128 x 16 into a score buffer (passes 2 and 3: plus one K = 16 MMA that adds
//               each row's constant term), and in pass 3 8 MMAs O += P V (P from shared memory in
//               two 64-key sub-tiles, v as an N-major operand, exactly the rows it was loaded with),
//               issued after the scores of the next block.  Passes 1 and 2 alternate between two
//               score buffers; pass 3 has one, O taking the second one's columns
//   warps 1-3   the CTA's 128 q rows once (cp.async, in the tensor cores' 128-byte swizzled
//               layout); then one thread of warp 1 streams the key blocks as TMA pieces into a
//               3-slot ring, in the order the MMA consumes them (k blocks in passes 1 and 2; then
//               k0, k1, v0, k2, v1, ...).  A key block is 128 consecutive tokens (global attention:
//               a 2-D box of the q|k|v matrix) or R whole rows of a ws x ws window,
//               R = min(floor(128 / ws), ws) (a 3-D box over (channel, x, y)); the slot rows a window
//               block leaves unwritten stay zero
//   warps 4-11  softmax: warp 4 + w reads TMEM lanes 32 (w % 4) .. + 31 (one query row per
//               thread) and score columns 64 (w / 4) .. + 63 of each block (two 32-column loads);
//               the two halves of a row combine their max and sum once per pass through shared
//               memory; P rows go to shared memory as fp16 operands (P < 1024 written as its own
//               bits, the subnormal P 2^-24; O is scaled back by 2^24).  A score buffer is released
//               as soon as the last load of a block has landed, so the next block's MMAs run
//               while the softmax works.  Warps whose rows all lie past the group, and 32-key
//               loads past its keys, skip the arithmetic (their P is written as zero)
// The CTAs holding the last (possibly partial, hence shorter) query tile of each group come after
// all the others, so they fill the last wave; paired last tiles (below) come before all the others.  Global attention whose last tile has at most 64
// queries puts the last tiles of two (image, head) units in one CTA (rows 0-63 and 64-127): a key
// block is then 64 keys of each unit (two N = 64 score MMAs, each unit's rows reading their own
// half of the columns), and each unit has its own O.  At 1600 tokens this turns 8 x 6 x 13 = 624
// CTAs (2.05 waves of two per SM) into 600 (two waves).
// The softmax warps' loop is compiled per pass, per launch form (with or without paired tiles) and,
// for global attention, separately for full key blocks, so the hot loop carries no branch for the
// cases it cannot meet.  In pass 3, P is one high-word product umulhi(I_b, F 2^(32 - sh0)) >> q when
// every row of the warp allows it.
// Every mbarrier wait is bounded (about one second); on expiry the kernel latches the device status
// word, every role stops, the loaders drain their copies and the TMEM is freed after every MMA
// issued has completed.
#include <cuda.h>

#include <cstdint>
#include <mutex>

#include "ilw_kernels.h"

namespace ilw {
namespace {

// The CTA form seen by the softmax warps: fixed at compile time (launches without paired tiles) or
// read at run time (launches with them, where one code path serves both forms: two specialised
// copies measured slower there, the SMs running both).
template <bool B> struct FixedForm {
    __device__ constexpr bool operator()() const { return B; }
};
template <int P> struct PassTag { static constexpr int value = P; };
template <bool B> struct BoolTag { static constexpr bool value = B; };
struct RuntimeForm {
    bool pair;
    __device__ bool operator()() const { return pair; }
};
constexpr int TQ = 128;      // queries per CTA
constexpr int TKB = 128;     // keys per block (global attention)
constexpr int NP = 3;        // ring slots of TKB x 128 bytes (one k or v block)
// score buffers (TMEM, TKB columns each): two in passes 1 and 2, when O is not yet accumulated and
// the second buffer takes its columns; one in pass 3, with O in the columns after it
constexpr int NS = 2;
constexpr int NPB = 1;       // P buffers (shared memory, TQ x TKB fp16)
constexpr int NCQ = 2;       // softmax warps per TMEM lane quarter, each on CPW columns of a block
constexpr int CPW = TKB / NCQ;
constexpr int CW = 32;          // columns per TMEM load (one softmax chunk)
constexpr int NCH = CPW / CW;   // chunks per block and thread
constexpr int OPW = 64 / NCQ;  // output columns per softmax thread
constexpr int kSlotB = TKB * 128;
constexpr int kPB = TQ * TKB * 2;  // bytes of one P buffer: TKB / 64 sub-tiles of 128 rows x 128 bytes
constexpr int kTmemCols = 256;  // S[0] | S[1] or O (64 columns; paired tiles: 128)
constexpr int kMinBlocks = 2;
static_assert(NS * TKB <= kTmemCols && TKB + 128 <= kTmemCols, "TMEM columns");
constexpr int NLOAD = 96;        // q loader threads (warps 1-3)
constexpr int NSMX = 128 * NCQ;  // softmax threads (warps 4 ..)
constexpr int kThreadsTc = 128 + NSMX;
constexpr long long kWaitTc = 2000000000ll;  // ~1 s at 2 GHz

struct TcSmem {  // offsets from the 1024-aligned base
    static constexpr int kQ = 0;
    static constexpr int kRing = kQ + TQ * 128;
    static constexpr int kP = kRing + NP * kSlotB;
    // the constant-term operands of passes 2 and 3 (K = 16, 32-byte rows, 32-byte swizzle):
    // A: -(2^23 + max + 1) of each query row as fp16 terms, B: the matching weights for every key
    static constexpr int kAugA = kP + NPB * kPB;
    static constexpr int kAugB = kAugA + TQ * 32;
    static constexpr int kRedMax = kAugB + TKB * 32;       // float [NCQ][128]
    static constexpr int kRedSum = kRedMax + NCQ * TQ * 4; // uint64 [NCQ][128]
    static constexpr int kBar = kRedSum + NCQ * TQ * 8;
    // barriers: q_full, full[NP], empty[NP], s_full[NS], s_free[NS], p_full[NPB], p_free[NPB], o_full, drain,
    // xchg, aug_full
    static constexpr int kNBar = 1 + 2 * NP + 2 * NS + 2 * NPB + 4;
    static constexpr int kSlot = kBar + 8 * kNBar;  // TMEM address, abort flag
    static constexpr int kBytes = kSlot + 16;
};

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ void bar_init(uint32_t b, uint32_t n) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(b), "r"(n) : "memory");
}
__device__ __forceinline__ void bar_arrive(uint32_t b) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(b) : "memory");
}
__device__ __forceinline__ bool bar_try(uint32_t b, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred P;\n mbarrier.try_wait.parity.shared::cta.b64 P, [%1], %2, %3;\n selp.b32 %0, 1, 0, P;\n}\n"
        : "=r"(ok)
        : "r"(b), "r"(parity), "r"(20000)
        : "memory");
    return ok != 0;
}
// Bounded wait: false (after latching `code` and raising the abort flag) when it ran out, or when
// another role already aborted.
__device__ __forceinline__ bool bar_wait(uint32_t b, uint32_t parity, volatile int *abort, int *status, int code) {
    if (bar_try(b, parity)) return true;
    const long long t0 = clock64();
    for (uint32_t i = 0;; ++i) {
        if (bar_try(b, parity)) return true;
        if ((i & 63) == 63) {
            if (*abort) return false;
            if (clock64() - t0 > kWaitTc) {
                if (status) atomicExch(status, code);
                *abort = 1;
                return false;
            }
        }
    }
}
__device__ __forceinline__ void fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void commit(uint32_t b) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(b) : "memory");
}
// 128-byte swizzled operand: 8-row groups 1024 bytes apart (K-major rows of 128 B, or, for the
// N-major V operand, rows of 128 B along N with 8-row groups along K)
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
// 32-byte swizzled K-major operand of K = 16: rows of 32 bytes, 8-row groups 256 bytes apart
__device__ __forceinline__ uint64_t desc_sw32(uint32_t saddr) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1 << 16;
    d |= (uint64_t)(256 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)6 << 61;
    return d;
}
__device__ __forceinline__ void mma(uint32_t dt, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(dt),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// TMEM load of N = 16 or 32 consecutive 32-bit columns of this thread's lane.
template <int N>
__device__ __forceinline__ void tld(uint32_t taddr, uint32_t (&v)[N]) {
    if constexpr (N == 32) {
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
            "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
              "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]),
              "=r"(v[17]), "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
              "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
            : "r"(taddr));
    } else {
        static_assert(N == 16, "16 or 32 columns");
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]), "=r"(v[7]), "=r"(v[8]),
              "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
            : "r"(taddr));
    }
}
// Waits for this thread's TMEM loads; the destination registers are marked as written by the
// wait so that no use is scheduled before it.
template <int N>
__device__ __forceinline__ void twait(uint32_t (&a)[N]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(a[0]), "+r"(a[1]), "+r"(a[2]), "+r"(a[3]), "+r"(a[4]), "+r"(a[5]), "+r"(a[6]), "+r"(a[7]),
                   "+r"(a[8]), "+r"(a[9]), "+r"(a[10]), "+r"(a[11]), "+r"(a[12]), "+r"(a[13]), "+r"(a[14]), "+r"(a[15])
                 :
                 : "memory");
    if constexpr (N == 32)
        asm volatile(""
                     : "+r"(a[16]), "+r"(a[17]), "+r"(a[18]), "+r"(a[19]), "+r"(a[20]), "+r"(a[21]), "+r"(a[22]),
                       "+r"(a[23]), "+r"(a[24]), "+r"(a[25]), "+r"(a[26]), "+r"(a[27]), "+r"(a[28]), "+r"(a[29]),
                       "+r"(a[30]), "+r"(a[31])::"memory");
}
__device__ __forceinline__ void cpa16(uint32_t dst, const void *src, uint32_t n) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(n) : "memory");
}
__device__ __forceinline__ void cpa_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void bar_expect_tx(uint32_t b, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(b), "r"(bytes) : "memory");
}
__device__ __forceinline__ void tma_2d(uint32_t dst, const CUtensorMap *m, int32_t x, int32_t y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"((uint64_t)m), "r"(x), "r"(y), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void tma_3d(uint32_t dst, const CUtensorMap *m, int32_t x, int32_t y, int32_t z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"((uint64_t)m), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}

// Kernel arguments: the attention problem and the tensor maps of its k and v columns.
struct TcArgs {
    CUtensorMap kmap, vmap;      // 2-D {64 H, B T} (global) or 3-D {64 H, gs, B gs} (windows), 128-byte swizzle
    CUtensorMap kmap64, vmap64;  // global, paired last tiles: the same with 64-row boxes
    AttnParams p;
    int32_t kbk;   // keys per block: 128 (global) or R ws (windows)
    int32_t rpb;   // window rows per block R (windows)
    int32_t win;   // 1: 3-D window boxes
    int32_t nq;    // query tiles per group
    int32_t pair;  // 1: the last tiles (<= 64 queries each) of two (image, head) units share a CTA
};
__device__ __forceinline__ uint32_t shr_clamp(uint32_t v, uint32_t n) {
    uint32_t r;
    asm("shr.u32 %0, %1, %2;" : "=r"(r) : "r"(v), "r"(n));
    return r;
}
// Constrained Shiftmax output from ShiftExp's parts (see attention.cu): floor(I_b F / 2^(sh0 + q)),
// w = bits of the fp32 value s - (2^23 + max + 1) that the score MMA of passes 2 and 3 leaves in TMEM
template <bool FASTQ>
__device__ __forceinline__ uint32_t p_direct(uint32_t w, const ShiftExpC &c, uint32_t F, uint32_t sh0) {
    uint32_t n = exp_arg_from_neg_bits(w);
    n = min(n, (uint32_t)c.kI0);
    const uint32_t q = FASTQ ? __umulhi(n, c.m32) : (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    const uint32_t Ib = ((q + 2u) * (uint32_t)c.I0 - n) >> 1;
    return shr_clamp(Ib * F, sh0 + q);
}

// The same P as one high-word product: floor(I_b F / 2^(sh0 + q)) = umulhi(I_b, G) >> q with
// G = F 2^(32 - sh0) when sh0 <= 32 and F < 2^sh0 (floors compose), and G = 0 when sh0 > 32 (then
// I_b F < 2^32 <= 2^sh0 and every P is 0).  q <= k_inter < 32.
template <bool FASTQ>
__device__ __forceinline__ uint32_t p_direct_hi(uint32_t w, const ShiftExpC &c, uint32_t G) {
    uint32_t n = exp_arg_from_neg_bits(w);
    n = min(n, (uint32_t)c.kI0);
    const uint32_t q = FASTQ ? __umulhi(n, c.m32) : (__umulhi(n, c.m_lo) + n * c.m_hi) >> 8;
    const uint32_t Ib = ((q + 2u) * (uint32_t)c.I0 - n) >> 1;
    return __umulhi(Ib, G) >> q;
}

struct GroupTc {
    int64_t base;
    int32_t Tg, nw, ws, gs, wy, wx;
    __device__ __forceinline__ int64_t token(int32_t t) const {
        if (nw <= 1) return base + t;
        return base + (int64_t)(wy * ws + t / ws) * gs + wx * ws + t % ws;
    }
};

// P of one score: (I_exp F) >> sh, or its direct form from ShiftExp's parts (DIRECT)
template <bool FASTQ, bool DIRECT>
__device__ __forceinline__ uint32_t p_of(uint32_t w, const ShiftExpC &se, const RowNorm &rn, uint32_t sh0) {
    return DIRECT ? p_direct<FASTQ>(w, se, rn.F, sh0) : shiftmax_out(shift_exp_nbits<FASTQ>(w, se), rn);
}

// DIRECT: per-row s_d with I_b F < 2^32 (the host's condition), so P comes straight from ShiftExp's
// parts; otherwise P = (I_exp F) >> sh from the 64-bit product.  SUM4: every ShiftExp value is below
// 2^30 (I0 2^k_inter < 2^30, the host's condition), so four of them add up in 32 bits.
// MAYPAIR: the launch may hold paired last tiles (args.pair).  MAYFULL: key blocks of 128 tokens
// (global attention), whose full blocks are compiled without the masking of partial ones.
template <bool FASTQ, bool DIRECT, bool SUM4, bool MAYPAIR, bool MAYFULL>
__global__ void __launch_bounds__(kThreadsTc, kMinBlocks) attn_tc_kernel(const __grid_constant__ TcArgs args) {
    const AttnParams &p = args.p;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = (uint8_t *)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    const uint32_t sbase = su32(sm);
    const uint32_t bq_full = sbase + TcSmem::kBar;
    auto full = [&](int s) { return bq_full + 8u * (1 + s); };
    auto empty = [&](int s) { return bq_full + 8u * (1 + NP + s); };
    auto s_full = [&](int b) { return bq_full + 8u * (1 + 2 * NP + b); };
    auto s_free = [&](int b) { return bq_full + 8u * (1 + 2 * NP + NS + b); };
    auto p_full = [&](int b) { return bq_full + 8u * (1 + 2 * NP + 2 * NS + b); };
    auto p_free = [&](int b) { return bq_full + 8u * (1 + 2 * NP + 2 * NS + NPB + b); };
    const uint32_t o_full = bq_full + 8u * (1 + 2 * NP + 2 * NS + 2 * NPB), drain = o_full + 8u, xchg = o_full + 16u,
                   aug_full = o_full + 24u;
    uint32_t *tmem_slot = (uint32_t *)(sm + TcSmem::kSlot);
    volatile int *abort = (volatile int *)(sm + TcSmem::kSlot + 4);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // CTA -> (query tile, head, group): the tiles of every group but its last come first, the last
    // (possibly partial, hence shorter) tiles of all groups at the end, so they fill the last wave
    // (pair: the CTA holds the last tiles of units 2 j and 2 j + 1, unit = (image, head), rows
    // 0-63 for the first and 64-127 for the second; a key block is then 64 keys of each unit)
    int qt, head, z, head1 = 0, z1 = 0;
    bool pair = false, has1 = false;
    {
        // paired CTAs (the longest: every block twice the MMA and key traffic) come first, so they
        // do not form the tail of the last wave; the unpaired last tiles (shorter) come last
        const int Z = p.B * p.nw * p.nw, F = (args.nq - 1) * p.H * Z;
        const int NPR = (MAYPAIR && args.pair) ? (p.H * Z + 1) / 2 : 0;
        const int L = (int)blockIdx.x < NPR ? F + (int)blockIdx.x : (int)blockIdx.x - NPR;
        if (L < F) {
            qt = L % (args.nq - 1);
            head = (L / (args.nq - 1)) % p.H;
            z = L / ((args.nq - 1) * p.H);
        } else if (!MAYPAIR || !args.pair) {
            qt = args.nq - 1;
            head = (L - F) % p.H;
            z = (L - F) / p.H;
        } else {
            const int u0 = 2 * (L - F), u1 = u0 + 1;
            pair = true;
            qt = args.nq - 1;
            head = u0 % p.H;
            z = u0 / p.H;
            has1 = u1 < p.H * Z;
            head1 = has1 ? u1 % p.H : head;
            z1 = has1 ? u1 / p.H : z;
        }
    }
    GroupTc gr;
    {
        const int G2 = p.nw * p.nw, b = z / G2, w = z % G2;
        gr.base = (int64_t)b * p.T;
        gr.nw = p.nw;
        gr.gs = p.grid_side;
        gr.ws = p.nw > 1 ? p.grid_side / p.nw : 0;
        gr.wy = w / p.nw;
        gr.wx = w % p.nw;
        gr.Tg = p.nw > 1 ? gr.ws * gr.ws : p.T;
    }
    const int Tg = gr.Tg, q0 = qt * TQ, hoff = head * 64, kbk = pair ? 64 : args.kbk;
    const int nkb = (Tg + kbk - 1) / kbk;
    // pair: the second unit's first token (global attention: image z1) and head offset
    const int64_t base1 = (int64_t)z1 * p.T;
    const int hoff1 = head1 * 64;

    if (threadIdx.x == 0) {
        bar_init(bq_full, NLOAD);
        for (int s = 0; s < NP; ++s) {
            bar_init(full(s), 1);
            bar_init(empty(s), 1);
        }
        for (int b = 0; b < NS; ++b) {
            bar_init(s_full(b), 1);
            bar_init(s_free(b), NSMX / 32);
        }
        for (int b = 0; b < NPB; ++b) {
            bar_init(p_full(b), NSMX / 32);
            bar_init(p_free(b), 1);
        }
        bar_init(o_full, 1);
        bar_init(drain, 1);
        bar_init(xchg, NSMX / 32);
        bar_init(aug_full, 4);  // the four warps of the first column group write the constant-term rows
        *abort = 0;
        if (kbk < TKB)  // slot rows no window box writes: zero k rows give masked scores, zero v rows add nothing
            for (int sl = 0; sl < NP; ++sl)
                for (int o = kbk * 128; o < kSlotB; o += 16)
                    *(uint4 *)(sm + TcSmem::kRing + sl * kSlotB + o) = make_uint4(0, 0, 0, 0);
        fence_async_smem();
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(tmem_slot)), "n"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    fence_before();
    __syncthreads();
    fence_after();
    const uint32_t tmem = *tmem_slot;  // columns: S[b] at TKB b; O at TKB (pass 3)
    constexpr uint32_t kOcol = (uint32_t)TKB;  // O shares its columns with S[1], used before pass 3 only

    // Piece sequence: pieces 0 .. 2 nkb - 1 are the k blocks of passes 1 and 2; pass 3 streams
    // k0, k1, v0, k2, v1, ..., k(nkb - 1), v(nkb - 2), v(nkb - 1), the order in which the MMA uses them.
    if (warp == 0) {
        // ------------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            // D f32, A/B f16, both K-major, M = 128, N = TKB (scores) or 64 (O, B = v N-major)
            const uint32_t id_s = (1u << 4) | ((uint32_t)(TKB >> 3) << 17) | ((128u >> 4) << 24);
            const uint32_t id_s64 = (1u << 4) | ((64u >> 3) << 17) | ((128u >> 4) << 24);
            const uint32_t id_o = (1u << 4) | (1u << 16) | ((64u >> 3) << 17) | ((128u >> 4) << 24);
            // descriptors: an address step of 16 bytes is 1 in the low word (addresses < 256 KB, no carry)
            const uint64_t dq = desc_sw128(sbase + TcSmem::kQ), dring = desc_sw128(sbase + TcSmem::kRing),
                           dp = desc_sw128(sbase + TcSmem::kP), daa = desc_sw32(sbase + TcSmem::kAugA),
                           dab = desc_sw32(sbase + TcSmem::kAugB);
            // consumption state: the S buffer, the ring slot of the next piece and the P buffer, each
            // with its phase bit
            int sb = 0, ks = 0, pb = 0;
            uint32_t sph = 0, kph = 0, pph = 0;
            auto adv = [](int &slot, uint32_t &ph, int by) {
                slot += by;
                while (slot >= NP) {
                    slot -= NP;
                    ph ^= 1u;
                }
            };
            // scores of the next key block into S[sb] (aug: plus the constant term -(2^23 + max + 1) of
            // each row, passes 2 and 3); the k piece is released when they complete.  Passes 1 and 2
            // alternate between the two buffers (ring), pass 3 uses S[0] alone
            auto issue_s = [&](bool aug, bool ring) -> bool {
                if (!bar_wait(full(ks), kph, abort, p.status, kStatusTimeoutTma)) return false;
                if (!bar_wait(s_free(sb), sph ^ 1u, abort, p.status, kStatusTimeoutOperand)) return false;
                fence_after();
                const uint64_t dk = dring + (uint64_t)(ks * (kSlotB / 16));
                const uint32_t dt = tmem + (uint32_t)(TKB * sb);
                if (!pair) {
                    mma(dt, dq, dk, id_s, 0u);
                    mma(dt, dq + 2, dk + 2, id_s, 1u);
                    mma(dt, dq + 4, dk + 4, id_s, 1u);
                    mma(dt, dq + 6, dk + 6, id_s, 1u);
                } else {
                    // columns 0-63: every q row against the first unit's 64 keys (slot rows 0-63),
                    // columns 64-127: against the second unit's (slot rows 64-127, 8 KB on)
#pragma unroll
                    for (int u = 0; u < 2; ++u)
#pragma unroll
                        for (int t = 0; t < 4; ++t)
                            mma(dt + 64u * u, dq + 2 * t, dk + (uint64_t)(u * 512 + 2 * t), id_s64, t ? 1u : 0u);
                }
                if (aug) mma(dt, daa, dab, id_s, 1u);
                commit(s_full(sb));
                commit(empty(ks));
                if (!ring) sph ^= 1u;
                else if (++sb == NS) {
                    sb = 0;
                    sph ^= 1u;
                }
                return true;
            };
            // O += P V for the next key block of pass 3 (TKB / 16 steps; P sub-tile t / 4 holds keys
            // 64 (t / 4) ..); releases P[pb] and the v piece
            auto issue_pv = [&](bool first) -> bool {
                if (!bar_wait(full(ks), kph, abort, p.status, kStatusTimeoutTma)) return false;
                if (!bar_wait(p_full(pb), pph, abort, p.status, kStatusTimeoutOperand)) return false;
                fence_after();
                const uint64_t da = dp + (uint64_t)(pb * (kPB / 16)), dv = dring + (uint64_t)(ks * (kSlotB / 16));
                if (!pair) {
#pragma unroll
                    for (int t = 0; t < TKB / 16; ++t)
                        mma(tmem + kOcol, da + (uint64_t)((t >> 2) * (TQ * 128 / 16) + 2 * (t & 3)), dv + (uint64_t)(128 * t),
                            id_o, (first && t == 0) ? 0u : 1u);
                } else {
                    // P holds 64 keys per row (sub-tile 0); O of unit u (TMEM columns kOcol + 64 u) takes
                    // the P rows against that unit's v rows; only its own q rows are read back
#pragma unroll
                    for (int u = 0; u < 2; ++u)
#pragma unroll
                        for (int t = 0; t < 4; ++t)
                            mma(tmem + kOcol + 64u * u, da + (uint64_t)(2 * t), dv + (uint64_t)(u * 512 + 128 * t), id_o,
                                (first && t == 0) ? 0u : 1u);
                }
                commit(p_free(pb));
                commit(empty(ks));
                adv(ks, kph, 1);
                if (++pb == NPB) {
                    pb = 0;
                    pph ^= 1u;
                }
                return true;
            };
            bool ok = bar_wait(bq_full, 0, abort, p.status, kStatusTimeoutTma);
            fence_after();
            // passes 1 and 2: the k pieces in order; pass 2 waits for the rows' constant terms
            for (int j = 0; j < 2 * nkb && ok; ++j) {
                if (j == nkb) ok = bar_wait(aug_full, 0, abort, p.status, kStatusTimeoutOperand);
                if (ok) ok = issue_s(j >= nkb, true);
                adv(ks, kph, 1);
            }
            // pass 3: the scores of block kb + 1 are issued before the P V of block kb, so the softmax
            // warps always have the next scores waiting; the loaders stream the pieces in exactly this
            // order (k0, k1, v0, k2, v1, ..., v(n-1)), so a slot is refilled as soon as it is consumed
            // (after 2 nkb blocks the ring is back at S[0], whose phase bit sph now holds)
            if (ok) ok = issue_s(true, false);
            adv(ks, kph, 1);
            for (int kb = 0; kb + 1 < nkb && ok; ++kb) {
                ok = issue_s(true, false);
                adv(ks, kph, 1);
                if (ok) ok = issue_pv(kb == 0);
            }
            if (ok) ok = issue_pv(nkb == 1);
            if (ok) commit(o_full);
            // every MMA issued has completed before the TMEM is released
            commit(drain);
            const long long t0 = clock64();
            while (!bar_try(drain, 0) && clock64() - t0 < kWaitTc) {
            }
        }
    } else if (warp < 4) {
        // ------------------------------------------------------------------ loaders
        const int tl = threadIdx.x - 32;  // 0 .. 95
        const int64_t ld = p.ld_qkv;      // elements (fp16)
        const __half *Qg = (const __half *)p.Q;
        // one 16-byte chunk c of a 128-byte row r per item, swizzled: chunk c of row r at c ^ (r & 7)
        for (int it = tl; it < TQ * 8; it += NLOAD) {
            const int r = it >> 3, c = it & 7, u = pair ? r >> 6 : 0, tok = q0 + (pair ? r & 63 : r);
            const bool okr = tok < Tg && (u == 0 || has1);
            const int64_t t = !okr ? 0 : u ? base1 + tok : gr.token(tok);
            cpa16(sbase + TcSmem::kQ + r * 128 + ((c ^ (r & 7)) << 4), Qg + t * ld + (u ? hoff1 : hoff) + 8 * c,
                  okr ? 16u : 0u);
        }
        cpa_commit();
        asm volatile("cp.async.wait_all;" ::: "memory");
        fence_async_smem();
        bar_arrive(bq_full);
        if (tl == 0) {
            // the key-block stream: piece i into slot i % NP once the piece before it there is consumed.
            // Pieces 0 .. 2 nkb - 1 are the k blocks of passes 1 and 2; pass 3 follows the MMA's order:
            // k0, then k(j + 1), v(j) for j = 0 .. nkb - 2, then v(nkb - 1)
            const uint32_t bytes = pair ? 2u * 64u * 128u : (uint32_t)kbk * 128u;
            const int bimg = gr.base / p.T, npiece = 4 * nkb;
            int issued = 0, slot = 0;
            uint32_t ph = 0;
            for (int i = 0; i < npiece; ++i) {
                if (!bar_wait(empty(slot), ph ^ 1u, abort, p.status, kStatusTimeoutFree)) break;
                bool isv = false;
                int kb;
                if (i < 2 * nkb) {
                    kb = i < nkb ? i : i - nkb;
                } else {
                    const int j = i - 2 * nkb;
                    if (j == 0) kb = 0;
                    else if (j == 2 * nkb - 1) { kb = nkb - 1; isv = true; }
                    else if (j & 1) kb = (j + 1) >> 1;
                    else { kb = (j - 2) >> 1; isv = true; }
                }
                const CUtensorMap *m = isv ? &args.vmap : &args.kmap;
                const uint32_t dst = sbase + TcSmem::kRing + slot * kSlotB;
                bar_expect_tx(full(slot), bytes);
                if (pair) {
                    // 64 keys of each unit: rows 0-63 and 64-127 of the slot (the second unit's rows
                    // repeat the first's when there is none; nothing reads them then)
                    const CUtensorMap *m64 = isv ? &args.vmap64 : &args.kmap64;
                    tma_2d(dst, m64, hoff, (int32_t)(gr.base + kb * 64), full(slot));
                    tma_2d(dst + 8192u, m64, has1 ? hoff1 : hoff, (int32_t)((has1 ? base1 : gr.base) + kb * 64), full(slot));
                } else if (args.win)
                    tma_3d(dst, m, hoff, gr.wx * gr.ws, bimg * gr.gs + gr.wy * gr.ws + kb * args.rpb, full(slot));
                else
                    tma_2d(dst, m, hoff, bimg * p.T + kb * TKB, full(slot));
                issued = i + 1;
                if (++slot == NP) {
                    slot = 0;
                    ph ^= 1u;
                }
            }
            // after an abort, the pieces still in flight land before the CTA exits
            if (*abort)
                for (int i = issued - NP > 0 ? issued - NP : 0; i < issued; ++i) {
                    const long long t0 = clock64();
                    while (!bar_try(full(i % NP), (i / NP) & 1) && clock64() - t0 < kWaitTc) {
                    }
                }
        }
    } else {
        // the softmax warps' work for the CTA's form (one unit, or two paired last tiles)
        auto softmax = [&](auto form) {
            const bool PAIR = form();
            // ------------------------------------------------------------------ softmax, one row per thread
            // pair: rows 64-127 are the second unit's, row & 63 the query's place in its unit's tile
            const int qw = warp & 3, cq = (warp - 4) >> 2, row = 32 * qw + lane, unit = PAIR ? qw >> 1 : 0;
            const int urow = PAIR ? row & 63 : row, tok = q0 + urow;
            // some row of this warp is a query of the group
            const bool live = q0 + (urow & ~31) < Tg && (!PAIR || unit == 0 || has1);
            const uint32_t tlane = tmem + ((uint32_t)(32 * qw) << 16);
            float *red_max = (float *)(sm + TcSmem::kRedMax);
            uint64_t *red_sum = (uint64_t *)(sm + TcSmem::kRedSum);
            const ShiftExpC se = p.smx.se;
            bool ok = true;
            float mx = -3.0e38f;
            uint64_t sum = 0;
            RowNorm rn{};
            uint32_t sh0 = 0, hiG = 0;
            bool hi_form = false;
            // the other column groups' contributions to the row, through shared memory and the xchg barrier
            auto exchange = [&](int phase) -> bool {
                __syncwarp();
                if (lane == 0) bar_arrive(xchg);
                return __all_sync(0xffffffffu, bar_wait(xchg, phase, abort, p.status, kStatusTimeoutOperand));
            };
            int b = 0, pb = 0;  // S and P buffers of the next block, with their phase bits
            uint32_t sph = 0, pph = 0;
            // the three passes over the key blocks, each compiled for its own pass
            auto run_pass = [&](auto pass_tag) {
                constexpr int pass = decltype(pass_tag)::value;
                // one key block; FULL: the warp is live and every chunk of the block is whole (compiled
                // without the masking)
                auto block = [&](int kb, auto full_tag) -> bool {
                    constexpr bool FULL = decltype(full_tag)::value;
                        // warp-uniform outcome: the TMEM loads below need the whole warp
                        ok = __all_sync(0xffffffffu, bar_wait(s_full(b), sph, abort, p.status, kStatusTimeoutMma));
                        if (!ok) return false;
                        fence_after();
                        // pass 3 writes P into the buffer the previous block's P V reads: that MMA must have
                        // completed, which is waited for just before the first store, after the arithmetic
                        bool p_ready = pass != 2;
                        const int kvalid = min(kbk, Tg - kb * kbk);
                        // pair: 32 columns per block, from the unit's half of the score columns
                        const int nch = PAIR ? 32 / CW : NCH;
#pragma unroll 1
                        for (int h = 0; h < nch; ++h) {
                            const int kc = (PAIR ? 32 * cq : CPW * cq) + CW * h;  // first key of this load in the block
                            const int c0 = PAIR ? 64 * unit + kc : kc;           // its first score column
                            const int nvalid = kvalid - kc;  // valid columns of this load (may be <= 0 or > CW)
                            // warp-uniform: a warp whose rows all lie past the group, or a load past the group's
                            // keys, has nothing to compute (its P is zero, its other values unused)
                            const bool work = FULL || (live && nvalid > 0);
                            uint32_t s[CW];
                            tld<CW>(tlane + (uint32_t)(TKB * b + c0), s);
                            twait<CW>(s);
                            if (h == nch - 1) {  // the scores are in registers: the buffer is free
                                fence_before();
                                __syncwarp();
                                if (lane == 0) bar_arrive(s_free(b));
                            }
                            if (!work) {
                                if (pass == 2 && live) {
                                    if (!p_ready) {
                                        p_ready = true;
                                        ok = __all_sync(0xffffffffu, bar_wait(p_free(pb), pph ^ 1u, abort, p.status, kStatusTimeoutMma));
                                        if (!ok) break;
                                    }
                                    uint8_t *prow = sm + TcSmem::kP + pb * kPB + (kc >> 6) * (TQ * 128) + row * 128;
                                    const int k0 = (kc & 63) >> 3;
#pragma unroll
                                    for (int cc = 0; cc < CW / 8; ++cc) *(uint4 *)(prow + (((k0 + cc) ^ (row & 7)) << 4)) = make_uint4(0, 0, 0, 0);
                                }
                                continue;
                            }
                            const bool whole = FULL || nvalid >= CW;
                            if (pass == 0) {
                                float m = __uint_as_float(s[0]);
#pragma unroll
                                for (int c = 1; c < CW; ++c) m = fmaxf(m, __uint_as_float(s[c]));
                                if (!whole) {
                                    m = -3.0e38f;
#pragma unroll
                                    for (int c = 0; c < CW; ++c) m = c < nvalid ? fmaxf(m, __uint_as_float(s[c])) : m;
                                }
                                mx = fmaxf(mx, m);
                            } else if (pass == 1) {
                                uint32_t e[CW];
#pragma unroll
                                for (int c = 0; c < CW; ++c) e[c] = shift_exp_nbits<FASTQ>(s[c], se);
                                if (!whole) {
#pragma unroll
                                    for (int c = 0; c < CW; ++c) e[c] = c < nvalid ? e[c] : 0u;
                                }
                                // I0 2^k < 2^31 (checked by the host), so a pair of ShiftExp values fits in 32 bits;
                                // with SUM4 (I0 2^k < 2^30) four do
                                uint64_t part = 0;
                                if constexpr (SUM4) {
#pragma unroll
                                    for (int c = 0; c < CW; c += 4) part += (uint64_t)(e[c] + e[c + 1] + e[c + 2] + e[c + 3]);
                                } else {
#pragma unroll
                                    for (int c = 0; c < CW; c += 2) part += (uint64_t)(e[c] + e[c + 1]);
                                }
                                sum += part;
                            } else {
                                // P of the CW keys as fp16 operands: P < 1024, so its own bits are the fp16
                                // subnormal P 2^-24, exact; O then accumulates 2^-24 P V (also exact) and is
                                // scaled back by 2^24 when read
                                uint32_t pw[CW];
                                if (DIRECT && hi_form) {
#pragma unroll
                                    for (int c = 0; c < CW; ++c) pw[c] = p_direct_hi<FASTQ>(s[c], se, hiG);
                                } else {
#pragma unroll
                                    for (int c = 0; c < CW; ++c) pw[c] = p_of<FASTQ, DIRECT>(s[c], se, rn, sh0);
                                }
                                if (!whole) {
#pragma unroll
                                    for (int c = 0; c < CW; ++c) pw[c] = c < nvalid ? pw[c] : 0u;
                                }
                                uint32_t w[CW / 2];
#pragma unroll
                                for (int c = 0; c < CW / 2; ++c) w[c] = __byte_perm(pw[2 * c], pw[2 * c + 1], 0x5410);
                                if (!p_ready) {
                                    p_ready = true;
                                    ok = __all_sync(0xffffffffu, bar_wait(p_free(pb), pph ^ 1u, abort, p.status, kStatusTimeoutMma));
                                    if (!ok) break;
                                }
                                // keys kc .. kc + CW - 1 sit in sub-tile kc / 64, chunks (kc % 64) / 8 .. of the row;
                                // 16-byte chunk k of a row sits at k ^ (row & 7)
                                uint8_t *prow = sm + TcSmem::kP + pb * kPB + (kc >> 6) * (TQ * 128) + row * 128;
                                const int k0 = (kc & 63) >> 3;
#pragma unroll
                                for (int cc = 0; cc < CW / 8; ++cc)
                                    *(uint4 *)(prow + (((k0 + cc) ^ (row & 7)) << 4)) =
                                        make_uint4(w[4 * cc], w[4 * cc + 1], w[4 * cc + 2], w[4 * cc + 3]);
                            }
                        }
                        if (pass == 2) sph ^= 1u;  // pass 3: S[0] alone
                        else if (++b == NS) {
                            b = 0;
                            sph ^= 1u;
                        }
                        if (pass == 2) {
                            // every warp (also one that stored nothing) arrives for this block only after the
                            // previous block's P V completed, so arrivals never run a phase ahead
                            if (!p_ready) {
                                p_ready = true;
                                ok = __all_sync(0xffffffffu, bar_wait(p_free(pb), pph ^ 1u, abort, p.status, kStatusTimeoutMma));
                                if (!ok) return false;
                            }
                            fence_async_smem();
                            __syncwarp();
                            if (lane == 0) bar_arrive(p_full(pb));
                            if (++pb == NPB) {
                                pb = 0;
                                pph ^= 1u;
                            }
                        }
                                        return true;
                };
                if constexpr (MAYFULL) {
                    const int nfull = live && kbk % CW == 0 ? Tg / kbk : 0;
                    for (int kb = 0; kb < nkb; ++kb)
                        if (!(kb < nfull ? block(kb, BoolTag<true>{}) : block(kb, BoolTag<false>{}))) break;
                } else {
                    for (int kb = 0; kb < nkb; ++kb)
                        if (!block(kb, BoolTag<false>{})) break;
                }
            };
            run_pass(PassTag<0>{});
            do {  // pass 2 prologue: the row maxima meet; the constant-term rows
                if (!ok) break;
                    red_max[cq * TQ + row] = mx;
                    if (!(ok = exchange(0))) break;
#pragma unroll
                    for (int o = 1; o < NCQ; ++o) mx = fmaxf(mx, red_max[((cq + o) % NCQ) * TQ + row]);
                    if (cq == 0) {
                        // this row's constant term -(2^23 + max + 1) as fp16 terms against the key weights
                        // (1, 2048, 2048, 2048): max + 1 = 2048 a3 + a0 with a0 in [0, 2047], |a3| <= 512,
                        // every term exact in fp16 and every partial sum of the MMA an integer below 2^24.
                        // Both 16-byte halves of the row hold the same terms and the key rows carry their
                        // weights in one half only, so the product does not depend on which half the
                        // swizzle puts where.  Rows past the group get zeros.
                        const int m1 = live && tok < Tg ? __float2int_rn(mx) + 1 : 0;
                        const int a3 = m1 >> 11, a0 = m1 - (a3 << 11);
                        const uint32_t h0 = (uint32_t)__half_as_ushort(__int2half_rn(-a0)),
                                       h3 = (uint32_t)__half_as_ushort(__int2half_rn(-a3));
                        const uint32_t n2048 = live && tok < Tg ? 0xE800u : 0u;  // -2048
                        const uint4 ra = make_uint4(h0 | (n2048 << 16), n2048 | (h3 << 16), 0u, 0u);
                        *(uint4 *)(sm + TcSmem::kAugA + row * 32) = ra;
                        *(uint4 *)(sm + TcSmem::kAugA + row * 32 + 16) = ra;
                        // key row `row`: (1, 2048, 2048, 2048) in the first half, zeros in the second
                        *(uint4 *)(sm + TcSmem::kAugB + row * 32) = make_uint4(0x3C00u | (0x6800u << 16), 0x6800u | (0x6800u << 16), 0u, 0u);
                        *(uint4 *)(sm + TcSmem::kAugB + row * 32 + 16) = make_uint4(0u, 0u, 0u, 0u);
                        fence_async_smem();
                        __syncwarp();
                        if (lane == 0) bar_arrive(aug_full);
                    }
            } while (0);
            if (ok) run_pass(PassTag<1>{});
            do {  // pass 3 prologue: the row sums meet; s_d and F
                if (!ok) break;
                    red_sum[cq * TQ + row] = sum;
                    if (!(ok = exchange(1))) break;
#pragma unroll
                    for (int o = 1; o < NCQ; ++o) sum += red_sum[((cq + o) % NCQ) * TQ + row];
                    rn = shiftmax_norm(sum ? sum : 1, p.smx.s_d, p.smx.m_p, p.smx.M_hw, p.smx.k_out);
                    sh0 = (uint32_t)(rn.sh - se.k);
                    {
                        // the high-word form when every row of the warp allows it
                        const bool row_ok = sh0 >= 32 || (rn.F >> sh0) == 0u;
                        hiG = sh0 > 32 ? 0u : sh0 == 32 ? rn.F : rn.F << (32 - sh0);
                        hi_form = __all_sync(0xffffffffu, row_ok);
                    }
            } while (0);
            if (ok) run_pass(PassTag<2>{});
            // ---- O = P V from TMEM: sat8(rq(O; m_o, s_o)) at the token's own position (OPW columns)
            if (ok) ok = __all_sync(0xffffffffu, bar_wait(o_full, 0, abort, p.status, kStatusTimeoutMma));
            if (ok) {
                fence_after();
                uint32_t o[OPW];
                tld<OPW>(tlane + kOcol + (uint32_t)(64 * unit + OPW * cq), o);
                twait<OPW>(o);
                if (live && tok < Tg) {
                    int32_t r[OPW];
#pragma unroll
                    for (int c = 0; c < OPW; ++c)
                        r[c] = sat8(rq(__float2int_rn(__uint_as_float(o[c]) * 16777216.0f), p.m_o, p.s_o));  // O = 2^24 acc
                    const int64_t t = unit ? base1 + tok : gr.token(tok);
                    const int ho = unit ? hoff1 : hoff;
                    if (p.o_f16) {
                        // 1152 + r (|r| <= 127) has the fp16 bits 0x6480 + r; subtracting 1152 leaves r
                        const __half2 h1152 = __half2half2(__ushort_as_half((unsigned short)0x6480));
                        uint32_t hw[OPW / 2];
#pragma unroll
                        for (int c = 0; c < OPW / 2; ++c) {
                            uint32_t x = (uint32_t)(0x6480 + r[2 * c]) | ((uint32_t)(0x6480 + r[2 * c + 1]) << 16);
                            __half2 hh = __hsub2(*reinterpret_cast<__half2 *>(&x), h1152);
                            hw[c] = *reinterpret_cast<uint32_t *>(&hh);
                        }
                        uint4 *dst = (uint4 *)((__half *)p.O + t * p.ld_o + ho + OPW * cq);
#pragma unroll
                        for (int c = 0; c < OPW / 8; ++c) dst[c] = make_uint4(hw[4 * c], hw[4 * c + 1], hw[4 * c + 2], hw[4 * c + 3]);
                    } else {
                        uint32_t bw[OPW / 4];
#pragma unroll
                        for (int c = 0; c < OPW / 4; ++c)
                            bw[c] = (uint32_t)(uint8_t)r[4 * c] | ((uint32_t)(uint8_t)r[4 * c + 1] << 8) |
                                    ((uint32_t)(uint8_t)r[4 * c + 2] << 16) | ((uint32_t)(uint8_t)r[4 * c + 3] << 24);
                        uint4 *dst = (uint4 *)((int8_t *)p.O + t * p.ld_o + ho + OPW * cq);
#pragma unroll
                        for (int c = 0; c < OPW / 16; ++c) dst[c] = make_uint4(bw[4 * c], bw[4 * c + 1], bw[4 * c + 2], bw[4 * c + 3]);
                    }
                }
            }
        };
        if constexpr (MAYPAIR) softmax(RuntimeForm{pair});
        else softmax(FixedForm<false>{});
    }

    fence_before();
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "n"(kTmemCols) : "memory");
    }
}

typedef CUresult (*EncodeTiledTc)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledTc encode_tc() {
    static std::once_flag once;
    static EncodeTiledTc fn = nullptr;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledTc)f;
    });
    return fn;
}

// Tensor map over the 64 H fp16 columns of k (or v) starting at `base`: 2-D {64 H, B T} with
// 64 x `rows` boxes, or (win) 3-D {64 H, gs, B gs} with 64 x ws x R boxes; 128-byte swizzle, zero fill.
bool kv_map(CUtensorMap *m, const void *base, const AttnParams &p, bool win, int ws, int R, int rows = TKB) {
    EncodeTiledTc fn = encode_tc();
    if (!fn) return false;
    const cuuint64_t row = (cuuint64_t)p.ld_qkv * 2;
    if (!win) {
        cuuint64_t dims[2] = {(cuuint64_t)p.H * 64, (cuuint64_t)p.B * p.T};
        cuuint64_t str[1] = {row};
        cuuint32_t box[2] = {64, (cuuint32_t)rows};
        cuuint32_t es[2] = {1, 1};
        return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(base), dims, str, box, es,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
    }
    const int gs = p.grid_side;
    cuuint64_t dims[3] = {(cuuint64_t)p.H * 64, (cuuint64_t)gs, (cuuint64_t)p.B * gs};
    cuuint64_t str[2] = {row, row * (cuuint64_t)gs};
    cuuint32_t box[3] = {64, (cuuint32_t)ws, (cuuint32_t)R};
    cuuint32_t es[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 3, const_cast<void *>(base), dims, str, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// One instantiation's launch; its shared-memory limit (the same for every launch) is raised once
// per device.
template <bool FASTQ, bool DIRECT, bool SUM4, bool MAYPAIR, bool MAYFULL>
cudaError_t launch_tc_one(const TcArgs &a, dim3 grid, size_t smem, cudaStream_t s) {
    static SmemLimit limit;
    const cudaError_t attr =
        raise_smem_limit(limit, (const void *)attn_tc_kernel<FASTQ, DIRECT, SUM4, MAYPAIR, MAYFULL>, (int)smem);
    if (attr != cudaSuccess) return attr;
    attn_tc_kernel<FASTQ, DIRECT, SUM4, MAYPAIR, MAYFULL><<<grid, kThreadsTc, smem, s>>>(a);
    return cudaGetLastError();
}
// windows: one form; global attention: full blocks compiled apart, and paired last tiles when the
// last tile has at most 64 queries
template <bool FASTQ, bool DIRECT, bool SUM4>
cudaError_t launch_tc_kernel(const TcArgs &a, dim3 grid, size_t smem, cudaStream_t s) {
    if (a.win) return launch_tc_one<FASTQ, DIRECT, SUM4, false, false>(a, grid, smem, s);
    return a.pair ? launch_tc_one<FASTQ, DIRECT, SUM4, true, true>(a, grid, smem, s)
                  : launch_tc_one<FASTQ, DIRECT, SUM4, false, true>(a, grid, smem, s);
}

}  // namespace

// The tensor-memory attention for dh = 64 with fp16-carried q|k|v whose rows are 16-byte aligned,
// an O whose rows of 64 outputs are 16-byte aligned, and windows of side <= 128;
// cudaErrorNotSupported otherwise (the caller then uses the warp-MMA kernel).
cudaError_t launch_attention_tc(const AttnParams &p, cudaStream_t s) {
    const int esz_o = p.o_f16 ? 2 : 1;
    if (p.dh != 64 || !p.qkv_f16 || (p.ld_qkv * 2) % 16 || (p.ld_o * esz_o) % 16 ||
        (((uintptr_t)p.Q | (uintptr_t)p.K | (uintptr_t)p.V) % 16) || ((uintptr_t)p.O % 16))
        return cudaErrorNotSupported;
    const bool win = p.nw > 1;
    const int ws = win ? p.grid_side / p.nw : 0;
    if (win && (ws > TKB || ws * p.nw != p.grid_side)) return cudaErrorNotSupported;
    const int G2 = win ? p.nw * p.nw : 1;
    const int Tg = win ? ws * ws : p.T;
    if (p.B == 0 || Tg == 0) return cudaSuccess;
    TcArgs a;
    a.p = p;
    a.win = win ? 1 : 0;
    a.rpb = win ? (TKB / ws < ws ? TKB / ws : ws) : 0;
    a.kbk = win ? a.rpb * ws : TKB;
    if (!kv_map(&a.kmap, p.K, p, win, ws, a.rpb) || !kv_map(&a.vmap, p.V, p, win, ws, a.rpb))
        return cudaErrorNotSupported;
    const bool fastq = p.smx.se.m32 != 0;
    const bool direct = p.smx.s_d < 0 && p.smx.m_p + 15 <= p.smx.M_hw && 32 - p.smx.k_out >= p.smx.se.k;
    const size_t smem = 1024 + TcSmem::kBytes;
    a.nq = (Tg + TQ - 1) / TQ;
    // global attention whose last query tile has at most 64 rows: two units' last tiles per CTA
    // (T = 1600: 48 half tiles become 24 CTAs, so 8 x 6 units fill two waves of two CTAs per SM)
    a.pair = !win && Tg - (a.nq - 1) * TQ <= 64 ? 1 : 0;
    if (a.pair && (!kv_map(&a.kmap64, p.K, p, false, 0, 0, 64) || !kv_map(&a.vmap64, p.V, p, false, 0, 0, 64)))
        return cudaErrorNotSupported;
    const int units = p.H * p.B * G2;
    const dim3 grid((unsigned)((a.nq - 1) * units + (a.pair ? (units + 1) / 2 : units)));
    const bool sum4 = ((int64_t)p.smx.se.I0 << p.smx.se.k) < ((int64_t)1 << 30);
    if (fastq && direct)
        return sum4 ? launch_tc_kernel<true, true, true>(a, grid, smem, s) : launch_tc_kernel<true, true, false>(a, grid, smem, s);
    if (fastq) return launch_tc_kernel<true, false, false>(a, grid, smem, s);
    if (direct) return launch_tc_kernel<false, true, false>(a, grid, smem, s);
    return launch_tc_kernel<false, false, false>(a, grid, smem, s);
}

}  // namespace ilw
