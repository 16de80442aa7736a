// fxpq_host.cu -- device status word, launch accounting and status strings of libfxpq.so.
#include <atomic>
#include <mutex>

#include "fxpq_common.cuh"

namespace {
// Latched device status: the first error code a kernel reports (0 = none).  A file-scope
// __device__ word exists once per device that loads the library.
__device__ int g_status_word;

std::atomic<long long> g_launches{0};
std::mutex g_mu;
int* g_status_addr[64] = {nullptr};
}  // namespace

namespace fxpq {

int* status_ptr() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_status_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
        g_status_addr[dev] = static_cast<int*>(p);
    }
    return g_status_addr[dev];
}

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

fxpq_status after_launch(const char* what) {
    (void)what;
    note_launch();
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? FXPQ_OK : FXPQ_ERR_CUDA;
}

}  // namespace fxpq

extern "C" fxpq_status fxpq_get_device_status(void* stream) {
    if (cudaStreamSynchronize(fxpq::as_stream(stream)) != cudaSuccess) return FXPQ_ERR_CUDA;
    int* p = fxpq::status_ptr();
    if (!p) return FXPQ_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return FXPQ_ERR_CUDA;
    if (v != 0) {
        int z = 0;
        if (cudaMemcpy(p, &z, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess) return FXPQ_ERR_CUDA;
    }
    return static_cast<fxpq_status>(v);
}

extern "C" const char* fxpq_status_string(fxpq_status s) {
    switch (s) {
        case FXPQ_OK: return "ok";
        case FXPQ_ERR_INVALID_ARG: return "invalid argument";
        case FXPQ_ERR_UNSUPPORTED: return "unsupported request";
        case FXPQ_ERR_NONFINITE: return "non-finite input";
        case FXPQ_ERR_TIMEOUT: return "bounded device wait timed out";
        case FXPQ_ERR_CUDA: return "CUDA runtime error";
        case FXPQ_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
        case FXPQ_ERR_RANGE: return "integer range of the exact arithmetic exceeded";
        default: return "unknown status";
    }
}

extern "C" int64_t fxpq_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }
