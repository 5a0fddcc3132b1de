// status.cu -- the device status word that kernels with bounded waits latch when a wait runs
// out, and the host side that reads and clears it (ilwdetr_device_status).
#include <atomic>
#include <cstdint>
#include <mutex>

#include "ilw_kernels.h"

namespace ilw {
namespace {

__device__ int g_status_word;

constexpr int kMaxDev = 64;
std::mutex g_mu;
int *g_addr[kMaxDev] = {};

}  // namespace

int *status_word_ptr() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return nullptr;
    thread_local int last_dev = -1;
    thread_local int *last_ptr = nullptr;
    if (dev == last_dev) return last_ptr;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
        g_addr[dev] = (int *)p;
    }
    last_dev = dev;
    last_ptr = g_addr[dev];
    return g_addr[dev];
}

int sm_count() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return 1;
    static std::atomic<int> count[kMaxDev];  // 0 until read; every writer stores the same value
    int v = count[dev].load(std::memory_order_relaxed);
    if (!v) {
        if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1) return 1;
        count[dev].store(v, std::memory_order_relaxed);
    }
    return v;
}

cudaError_t read_and_clear_status(int *value) {
    *value = 0;
    int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(value, g_status_word, sizeof(int));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_status_word, &zero, sizeof(int));
}

}  // namespace ilw
