// gemm_tc.cu -- host side of the tensor-core integer GEMM (tensor maps, SD-ShiftGELU output tables,
// weight packing, launch-shape choice) and its fp16-A launch shapes; the kernel is in gemm_tc.cuh,
// the int8-A launch shapes in gemm_tc_i8.cu.
#include <atomic>

#include "gemm_tc.cuh"

namespace ilw {
namespace {

// SD-ShiftGELU output tables, one slot per parameter set (I0, k_inter, k_out, m_g, s_g): entry
// g + 32767 is sat8(rq(g * I_div(g); m_g, s_g)) for every int16 value g (Algorithm 1 followed by the
// output requantisation), a pure function of g.  A slot, once given to a parameter set, keeps it
// for the life of the process: kernels in flight on other streams and captured graphs hold its
// address, so it is never rebuilt for another set.  A parameter set beyond the last slot is refused.
constexpr int kGeluSlots = 256;  // 16 MiB per device
constexpr int kGeluTabBytes = 65536;  // 65535 entries, padded to 16 bytes
__device__ __align__(16) int8_t g_gelu_tab[kGeluSlots][kGeluTabBytes];

__global__ void gelu_table_kernel(int8_t *tab, GeluC c, int32_t m_g, int32_t s_g) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < kGeluTabBytes) {
        const int32_t g = min(i, 65534) - 32767;
        tab[i] = (int8_t)sat8(rq((int64_t)g * gelu_idiv(g, c), m_g, s_g));
    }
}

// The table slot of (device, GELU constants, m_g, s_g), built on first use.  The first build of a
// slot is waited for (unless the stream is being captured), so a slot marked built is complete for
// every stream; a build recorded into a graph is repeated by each replay until an eager call builds it
// (every replay writes the same bytes, since the slot never changes hands).  With every slot taken,
// a new parameter set gets cudaErrorMemoryAllocation and nothing is launched.
const int8_t *gelu_table_impl(const GeluC &c, int32_t m_g, int32_t s_g, cudaStream_t s, cudaError_t *err) {
    struct Key {
        int dev;
        int32_t I0, k, out_sh, m_g, s_g;
        bool operator==(const Key &o) const {
            return dev == o.dev && I0 == o.I0 && k == o.k && out_sh == o.out_sh && m_g == o.m_g && s_g == o.s_g;
        }
    };
    static std::mutex mu;
    static Key keys[64][kGeluSlots];
    static bool built[64][kGeluSlots] = {};
    static int nused[64] = {};
    static int8_t *base[64] = {};
    *err = cudaSuccess;
    int dev = 0;
    if ((*err = cudaGetDevice(&dev)) != cudaSuccess) return nullptr;
    if (dev < 0 || dev >= 64) {
        *err = cudaErrorInvalidDevice;
        return nullptr;
    }
    std::lock_guard<std::mutex> lock(mu);
    if (!base[dev]) {
        void *b = nullptr;
        if ((*err = cudaGetSymbolAddress(&b, g_gelu_tab)) != cudaSuccess) return nullptr;
        base[dev] = (int8_t *)b;
    }
    const Key key{dev, c.se.I0, c.se.k, c.out_sh, m_g, s_g};
    int slot = -1;
    for (int i = 0; i < nused[dev]; ++i)
        if (keys[dev][i] == key) slot = i;
    if (slot < 0) {
        if (nused[dev] >= kGeluSlots) {
            *err = cudaErrorMemoryAllocation;
            return nullptr;
        }
        slot = nused[dev]++;
        keys[dev][slot] = key;
        built[dev][slot] = false;
    }
    int8_t *tab = base[dev] + (size_t)slot * kGeluTabBytes;
    if (!built[dev][slot]) {
        gelu_table_kernel<<<kGeluTabBytes / 256, 256, 0, s>>>(tab, c, m_g, s_g);
        if ((*err = cudaGetLastError()) != cudaSuccess) return nullptr;
        cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
        if ((*err = cudaStreamIsCapturing(s, &cs)) != cudaSuccess) return nullptr;
        if (cs == cudaStreamCaptureStatusNone) {
            if ((*err = cudaStreamSynchronize(s)) != cudaSuccess) return nullptr;
            built[dev][slot] = true;
        }
    }
    return tab;
}

// int8 weight -> fp16 operand copy (|w| <= 127: exact)
__global__ void pack_weight_kernel(const int8_t *W, int64_t n, __half *w16) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) w16[i] = __int2half_rn((int)W[i]);
}

// ------------------------------------------------------------------ host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static std::once_flag once;
    static EncodeTiledFn fn = nullptr;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)f;
    });
    return fn;
}

// Recently encoded tensor maps of this host thread.  A map is a pure function of its key, so a hit
// is the same 128 bytes cuTensorMapEncodeTiled would write; the cache only saves the encoding.
struct MapKey {
    const void *base;
    int64_t rows, cols, ld;
    int32_t dt, box_cols, box_rows, sw;
    bool operator==(const MapKey &o) const {
        return base == o.base && rows == o.rows && cols == o.cols && ld == o.ld && dt == o.dt &&
               box_cols == o.box_cols && box_rows == o.box_rows && sw == o.sw;
    }
};
struct MapCache {
    static constexpr int kSlots = 64;
    MapKey key[kSlots];
    CUtensorMap map[kSlots];
    bool used[kSlots] = {};
    int next = 0;
};

// 2-D tensor map over a row-major [rows, cols] matrix (cols contiguous), boxes of box_cols x box_rows
bool make_map_impl(CUtensorMap *m, const void *base, CUtensorMapDataType dt, int esize, int64_t rows, int64_t cols,
              int64_t ld, int box_cols, int box_rows, CUtensorMapSwizzle sw) {
    thread_local MapCache cache;
    const MapKey k{base, rows, cols, ld, (int32_t)dt, box_cols, box_rows, (int32_t)sw};
    for (int i = 0; i < MapCache::kSlots; ++i)
        if (cache.used[i] && cache.key[i] == k) {
            *m = cache.map[i];
            return true;
        }
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(ld * esize)};
    cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    if (fn(m, dt, 2, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return false;
    const int slot = cache.next;
    cache.next = (cache.next + 1) % MapCache::kSlots;
    cache.key[slot] = k;
    cache.map[slot] = *m;
    cache.used[slot] = true;
    return true;
}

}  // namespace

bool gemm_make_map(CUtensorMap *m, const void *base, CUtensorMapDataType dt, int esize, int64_t rows, int64_t cols,
                   int64_t ld, int box_cols, int box_rows, CUtensorMapSwizzle sw) {
    return make_map_impl(m, base, dt, esize, rows, cols, ld, box_cols, box_rows, sw);
}
const int8_t *gemm_gelu_table(const GeluC &c, int32_t m_g, int32_t s_g, cudaStream_t s, cudaError_t *err) {
    return gelu_table_impl(c, m_g, s_g, s, err);
}

namespace {
std::atomic<int32_t> g_dbg_skip{-1};
std::atomic<long long> g_dbg_cycles{0};
}  // namespace
void gemm_debug_wait(int32_t *skip, long long *cycles) {
    *skip = g_dbg_skip.load(std::memory_order_relaxed);
    const long long c = g_dbg_cycles.load(std::memory_order_relaxed);
    *cycles = c > 0 ? c : kWaitCycles;
}
void gemm_set_debug_wait(int32_t skip, long long cycles) {
    g_dbg_skip.store(skip, std::memory_order_relaxed);
    g_dbg_cycles.store(cycles, std::memory_order_relaxed);
}

cudaError_t launch_pack_weight(const int8_t *W, int32_t N, int32_t K, void *packed, cudaStream_t s) {
    const int64_t n = (int64_t)N * K;
    pack_weight_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(W, n, (__half *)packed);
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmProblem &gp, const EpiParams &ep, cudaStream_t s) {
    if (gp.M == 0 || gp.N == 0) return cudaSuccess;
    const bool gelu = ep.kind == EPI_GELU;
    // 192-wide tiles when N splits evenly into them (fewer re-reads of A per flop), else 128
    if (gp.nb > 1) return run_i8<128, 5, kMaxBranches, false>(gp, ep, s);
    if (gp.a_f16) {
        // fp16 A: no conversion stage, so 192-wide tiles get 12 epilogue warps.  Weights resident
        // in shared memory when the CTA's BN rows of W fit next to the A stages (K <= 1024).
        // GELU keeps its 64 KB table in shared memory, so its 192-wide tiles stream the weights.
        // K > 1024 needs two accumulators per tile: 128-wide tiles keep two TMEM sets (overlap).
        // Without GELU, among the shapes that fit, the one whose busiest CTA has the fewest output
        // columns to produce wins (tiles are uniform work, so wave quantisation decides; ties go to
        // the wider tile, which re-reads A less).
        const int K = gp.br[0].K, nkb = (K + BK - 1) / BK;
        const bool n192 = gp.N % 192 == 0 && gp.N >= 384;
        const int64_t tiles_m = (gp.M + BM - 1) / BM;
        auto cost = [&](int bn, bool wres) -> int64_t {  // output columns of the busiest CTA, per row block
            const int64_t tiles_n = (gp.N + bn - 1) / bn, sms = num_sms();
            if (wres) {
                int64_t per_n = sms / tiles_n;
                per_n = per_n < 1 ? 1 : (per_n > tiles_m ? tiles_m : per_n);
                return (tiles_m + per_n - 1) / per_n * bn;
            }
            const int64_t tiles = tiles_m * tiles_n, grid = tiles < sms ? tiles : sms;
            return (tiles + grid - 1) / grid * bn;
        };
        if (gelu) {  // 192-wide measured faster inside the encoder step even at 6 vs 8 rounds (FC1)
            if (n192) return run<192, 3, 1, true, false, true>(gp, ep, s);
            if (K <= kSegK && smem_bytes<128, 3, KIND_GELU8, true, true>(nkb * 128 * 128) <= kSmemMax)
                return run<128, 3, 1, true, true, true>(gp, ep, s);
            return run<128, 3, 1, true, false, true>(gp, ep, s);
        }
        if (K <= kSegK) {
            const bool w192 = n192 && smem_bytes<192, 3, KIND_RQ8, true, true>(nkb * 192 * 128) <= kSmemMax;
            const bool w128 = smem_bytes<128, 3, KIND_RQ8, true, true>(nkb * 128 * 128) <= kSmemMax;
            const int64_t c192w = w192 ? cost(192, true) : INT64_MAX, c128w = w128 ? cost(128, true) : INT64_MAX,
                          c192 = n192 ? cost(192, false) : INT64_MAX, c128 = cost(128, false);
            const int64_t best = std::min(std::min(c192w, c128w), std::min(c192, c128));
            if (c192w == best) return run<192, 3, 1, true, true, false>(gp, ep, s);
            if (c192 == best) return run<192, 4, 1, true, false, false>(gp, ep, s);
            if (c128w == best) return run<128, 3, 1, true, true, false>(gp, ep, s);
            return run<128, 5, 1, true, false, false>(gp, ep, s);
        }
        return run<128, 5, 1, true, false, false>(gp, ep, s);
    }
    // int8 A (converted to the fp16 operand in shared memory by the converter warps)
    if (gp.N % 192 == 0 && gp.N >= 768)
        return gelu ? run_i8<192, 3, 1, true>(gp, ep, s) : run_i8<192, 4, 1, false>(gp, ep, s);
    return gelu ? run_i8<128, 3, 1, true>(gp, ep, s) : run_i8<128, 5, 1, false>(gp, ep, s);
}

}  // namespace ilw
