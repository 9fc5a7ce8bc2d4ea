// Comba-pk output correction (appendix B.3, the "p" form): the chunk kernels of the pk form
// run on q~ = q - d_h p with d = 0, so the correction is applied here, once per call:
//     qt[t, h, :] = q[t, h, :] - d_h p[t, h, :].
// Elementwise and HBM-bound: 16-byte vectors, four per thread in flight.
#include "params.cuh"

namespace comba {

template <typename T>
__global__ void __launch_bounds__(256) k_pk_qtilde(const T* __restrict__ q, const T* __restrict__ p,
                                                   const float* __restrict__ d, T* __restrict__ qt, long long nvec,
                                                   int vec_per_row, int H) {
    constexpr int V = 16 / (int)sizeof(T), U = 4;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long base = (long long)blockIdx.x * blockDim.x + threadIdx.x; base < nvec; base += stride * U) {
        uint4 qa[U], pa[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const long long i = base + u * stride;
            if (i < nvec) {
                qa[u] = *reinterpret_cast<const uint4*>(q + i * V);
                pa[u] = *reinterpret_cast<const uint4*>(p + i * V);
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const long long i = base + u * stride;
            if (i < nvec) {
                const float dh = d[(i / vec_per_row) % H];
                T* qe = reinterpret_cast<T*>(&qa[u]);
                const T* pe = reinterpret_cast<const T*>(&pa[u]);
#pragma unroll
                for (int e = 0; e < V; ++e) qe[e] = from_f<T>(to_f(qe[e]) - dh * to_f(pe[e]));
                *reinterpret_cast<uint4*>(qt + i * V) = qa[u];
            }
        }
    }
}

cudaError_t launch_pk_qtilde(const void* q, const void* p, const float* d, void* qt, long long rows, int H, int dk,
                             bool is_bf16, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    int dev = 0, nsm = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) || (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev))) return e;
    const int es = is_bf16 ? 2 : 4;
    const int vec_per_row = dk * es / 16;
    const long long nvec = rows * vec_per_row;
    long long grid = (nvec + 256LL * 4 - 1) / (256LL * 4);
    if (grid > 8LL * nsm) grid = 8LL * nsm;
    if (is_bf16)
        k_pk_qtilde<bf16><<<(unsigned)grid, 256, 0, s>>>((const bf16*)q, (const bf16*)p, d, (bf16*)qt, nvec,
                                                         vec_per_row, H);
    else
        k_pk_qtilde<float><<<(unsigned)grid, 256, 0, s>>>((const float*)q, (const float*)p, d, (float*)qt, nvec,
                                                          vec_per_row, H);
    return cudaGetLastError();
}

}  // namespace comba
