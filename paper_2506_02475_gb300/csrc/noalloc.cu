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
// is looked up on every call (cudaGetSymbolAddress, with the caller's device
// current): the lookup is cheap and cannot go stale when a context is torn
// down and re-created.  All calls share the one array and
// it keeps whatever the last call left: the forward writes every scratch byte
// before reading it, so nothing needs clearing, but two calls whose kernels
// overlap on the GPU (different streams, or different host threads) race on
// it and must be serialised by the caller.
#include <cuda_runtime.h>

#include "../../include/comba.h"
#include "params.cuh"

namespace {

static __device__ __align__(256) unsigned char g_static_scratch[COMBA_STATIC_SCRATCH_BYTES];

}  // namespace

namespace comba {

// Device address of the static scratch on the current device.  In host code
// the array's name is only a host-side stand-in, so the address is asked of
// the runtime each time.
cudaError_t static_scratch_address(void** out) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess) return e;
    if (!p) return cudaErrorInvalidSymbol;
    *out = p;
    return cudaSuccess;
}

}  // namespace comba

extern "C" comba_status_t comba_chunk_fwd_noalloc(const comba_shape_t* shape, const void* q, const void* k,
                                                  const void* v, const float* alpha, const float* beta,
                                                  const float* b, const float* d, const float* h0, void* o,
                                                  float* hT, comba_stream_t stream) {
    // Only the plain and iplr forms run here: saved factors would land in the shared array where no
    // caller can reach them, and the gated and pk forms have entry points of their own.
    if (shape && (shape->flags & ~COMBA_IPLR)) return COMBA_ERR_INVALID_ARG;
    const size_t need = comba_workspace_size(shape, 0);
    if (need > (size_t)COMBA_STATIC_SCRATCH_BYTES) return COMBA_ERR_WORKSPACE;
    void* scratch = nullptr;
    if (need > 0) {
        if (comba::static_scratch_address(&scratch) != cudaSuccess) return COMBA_ERR_CUDA;
    }
    // need == 0 means an invalid shape: the regular entry point reports why before launching anything.
    return comba_chunk_fwd(shape, q, k, v, alpha, beta, b, d, h0, o, hT, scratch, (size_t)COMBA_STATIC_SCRATCH_BYTES,
                           stream);
}
