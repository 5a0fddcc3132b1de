// noalloc.cu -- ilwdetr_patch_embed_noalloc: the patch embedding without any workspace
// argument and without any device allocation.
//
// Some callers cannot hand this library a workspace or let it allocate: a host runtime that owns
// the whole device-memory budget and forbids allocations inside its inference loop, or a
// latency-critical loop where cudaMalloc/cudaFree would add their implicit device-wide
// synchronisation.  For them the gathered patch matrix lives in a fixed device array compiled
// into the library: every GPU that loads the library reserves kNoAllocScratchBytes for it until
// the process exits.
#include <cstdint>
#include <mutex>

#include "ilw_kernels.h"
#include "ilwdetr.h"

namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)8 << 20;  // 8 MiB: 6 images of 3 x 640 x 640
constexpr int kMaxDevices = 64;

// The scratch array.  In host code this name is only a stand-in for the device symbol, never a
// device address: host code must use the address cudaGetSymbolAddress returns for the device.
static __device__ __align__(256) int8_t g_patch_scratch[kNoAllocScratchBytes];

std::mutex g_mu;
int8_t *g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device; looked up once per device (the
// first call on each device), with that device current, and kept for the life of the process: a
// cudaDeviceReset ends the context the address belongs to, so the entry point is not to be used
// across one.
int scratch_on_current_device(int8_t **out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return ilw::report_error(ILW_ERR_CUDA, cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices) return ilw::report_error(ILW_ERR_UNSUPPORTED, "device index too large");
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_patch_scratch);
        if (e != cudaSuccess || !p)
            return ilw::report_error(ILW_ERR_CUDA, "cudaGetSymbolAddress of the patch scratch array failed");
        g_scratch_addr[dev] = (int8_t *)p;
    }
    *out = g_scratch_addr[dev];
    return ILW_OK;
}

}  // namespace

extern "C" size_t ilwdetr_patch_embed_noalloc_max_bytes(void) { return kNoAllocScratchBytes; }

extern "C" int ilwdetr_patch_embed_noalloc(const int8_t *img, int32_t B, int32_t Cin, int32_t Hh, int32_t Ww,
                                           int32_t p, const void *Wp, const int32_t *bias, const int32_t *mult,
                                           const int32_t *shift, int32_t d, const int16_t *pos, int32_t m_pos,
                                           int32_t s_pos, int16_t *x0, ilw_stream_t stream) {
    // every argument is checked before anything is launched
    if (B < 0 || Cin < 1 || p < 16 || p % 16 || Hh < p || Ww < p || Hh % p || Ww % p || Ww % 16 || d < 1)
        return ilw::report_error(ILW_ERR_UNSUPPORTED, "patch_embed_noalloc: needs p % 16 == 0, p | H, p | W");
    if (B == 0) return ILW_OK;
    if (!img || ((uintptr_t)img % 16) != 0 || !x0)
        return ilw::report_error(ILW_ERR_INVALID_ARG, "patch_embed_noalloc: NULL or misaligned image, or NULL x0");
    if (!Wp || ((uintptr_t)Wp % 256) != 0)
        return ilw::report_error(ILW_ERR_INVALID_ARG, "patch_embed_noalloc: packed weight NULL or not 256-byte aligned");
    if (!mult || !shift) return ilw::report_error(ILW_ERR_INVALID_ARG, "patch_embed_noalloc: mult/shift are NULL");
    if (pos && (s_pos < 1 || s_pos > 62))
        return ilw::report_error(ILW_ERR_INVALID_ARG, "patch_embed_noalloc: position shift outside [1, 62]");
    // the gathered patch matrix, int8 (B*T rows of Cin*p*p)
    const size_t need = (size_t)B * (Hh / p) * (Ww / p) * Cin * p * p;
    if (need > kNoAllocScratchBytes)
        return ilw::report_error(ILW_ERR_UNSUPPORTED,
                                 "patch_embed_noalloc: this batch needs more scratch than the fixed 8 MiB "
                                 "(B * (H/p) * (W/p) * Cin * p * p bytes); split the batch or use "
                                 "ilwdetr_patch_embed with a workspace");
    const int32_t T = (Hh / p) * (Ww / p), K = Cin * p * p;
    ilw_residual_t r{pos, d, T, m_pos, s_pos};
    if (ilw::validate_only())  // the GEMM's own checks; Wp (256-byte aligned) stands in for the scratch
        return ilwdetr_gemm_requant((const int8_t *)Wp, K, Wp, bias, mult, shift, B * T, d, K, 16, x0, d,
                                    pos ? &r : nullptr, stream);
    int8_t *scratch = nullptr;
    int rc = scratch_on_current_device(&scratch);
    if (rc) return rc;
    // every byte the GEMM reads is written by the gather first: nothing needs clearing
    cudaError_t e = ilw::launch_patchify(img, B, Cin, Hh, Ww, p, scratch, (cudaStream_t)stream);
    if (e != cudaSuccess) return ilw::report_error(ILW_ERR_CUDA, cudaGetErrorString(e));
    return ilwdetr_gemm_requant(scratch, K, Wp, bias, mult, shift, B * T, d, K, 16, x0, d, pos ? &r : nullptr, stream);
}
