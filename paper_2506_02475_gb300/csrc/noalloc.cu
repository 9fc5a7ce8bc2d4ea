// Chunk forward for callers that may not allocate device memory.
//
// Some callers cannot hand the library a workspace: code that runs inside a
// host framework's execute step where device allocation is forbidden (an
// inference-engine or serving plugin, for instance), or a latency-critical
// loop that must never reach an allocator.  For them the forward's scratch
// lives in a fixed, file-scope device array instead of a caller workspace.
//
// The array is COMBA_STATIC_SCRATCH_BYTES (32 MiB) and exists on every GPU
// that loads this library, for the life of the process.  Its device address
// is looked up once per device (cudaGetSymbolAddress, with that device
// current) on the first call made there.  All calls share the one array and
// it keeps whatever the last call left: the forward writes every scratch byte
// before reading it, so nothing needs clearing, but two calls whose kernels
// overlap on the GPU (different streams, or different host threads) race on
// it and must be serialised by the caller.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/comba.h"

namespace {

static __device__ __align__(256) unsigned char g_static_scratch[COMBA_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the static scratch on the current device (looked up once).
comba_status_t static_scratch(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return COMBA_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return COMBA_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) return COMBA_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return COMBA_OK;
}

}  // namespace

extern "C" comba_status_t comba_chunk_fwd_noalloc(const comba_shape_t* shape, const void* q, const void* k,
                                                  const void* v, const float* alpha, const float* beta,
                                                  const float* b, const float* d, const float* h0, void* o,
                                                  float* hT, void* stream) {
    const size_t need = comba_workspace_size(shape, 0);
    if (need > (size_t)COMBA_STATIC_SCRATCH_BYTES) return COMBA_ERR_WORKSPACE;
    void* scratch = nullptr;
    if (need > 0) {
        const comba_status_t st = static_scratch(&scratch);
        if (st != COMBA_OK) return st;
    }
    // need == 0 means an invalid shape: the regular entry point reports why before launching anything.
    return comba_chunk_fwd(shape, q, k, v, alpha, beta, b, d, h0, o, hT, scratch, (size_t)COMBA_STATIC_SCRATCH_BYTES,
                           stream);
}
