// One-token Comba recurrence (appendix B.1, recurrent form) for a batch of
// independent decode rows.  Per (row, head) with H = S^T (dk x dv) and feedback
// vector f (f = k; the Comba-pk vector p of appendix B.3 when given):
//   x = H^T f, y = H^T q~ (q~ = q - d f), e = beta v - b beta x,
//   o = alpha y + e (k . q~),  H <- alpha H + k e^T.
// Columns of H are independent, so a block owns one (row, head, 32-column
// tile): it reads its 32 columns of the state once with 16-byte streaming
// loads, keeps them in registers, and writes them back once.  The kernel is
// bound by HBM bandwidth on the state (2 * dk * dv * 4 bytes per row-head).
#include "params.cuh"

namespace comba {

template <typename T, int DK, int DV>
__global__ void __launch_bounds__(128) k_step(int H, const T* __restrict__ q, const T* __restrict__ k,
                                              const T* __restrict__ v, const T* __restrict__ pf,
                                              const float* __restrict__ alpha,
                                              const float* __restrict__ beta, const float* __restrict__ b,
                                              const float* __restrict__ d, float* __restrict__ state,
                                              T* __restrict__ o, int iplr) {
    constexpr int NT = DV / 32;   // column tiles per (row, head)
    constexpr int RPT = DK / 16;  // state rows per thread
    const int tile = blockIdx.x % NT;
    const long long u = blockIdx.x / NT;  // row * H + head
    const int h = (int)(u % H);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int c4 = tid & 7;              // which 4 columns of the tile
    const int rg = tid >> 3;             // row group 0..15
    const int col0 = tile * 32;

    __shared__ float sk[DK], sq[DK], sf[DK];
    __shared__ float rx[4][32], ry[4][32];
    __shared__ float se[32];
    __shared__ float skq;

    float4* st = reinterpret_cast<float4*>(state + u * DK * DV + col0) + c4;
    float4 hv[RPT];
#pragma unroll
    for (int r = 0; r < RPT; ++r) hv[r] = __ldcs(st + (long long)(rg + 16 * r) * (DV / 4));

    const float dh = d[h];
    for (int i = tid; i < DK; i += 128) {
        const float kk = to_f(k[u * DK + i]);
        const float ff = pf ? to_f(pf[u * DK + i]) : kk;
        sk[i] = kk;
        sf[i] = ff;
        sq[i] = to_f(q[u * DK + i]) - dh * ff;
    }
    __syncthreads();
    if (warp == 0) {
        float s = 0.f;
        for (int i = lane; i < DK; i += 32) s += sk[i] * sq[i];
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o2);
        if (lane == 0) skq = s;
    }
    float x[4] = {0.f, 0.f, 0.f, 0.f}, y[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        const float kr = sf[rg + 16 * r], qr = sq[rg + 16 * r];   // feedback read through f
        x[0] += hv[r].x * kr; x[1] += hv[r].y * kr; x[2] += hv[r].z * kr; x[3] += hv[r].w * kr;
        y[0] += hv[r].x * qr; y[1] += hv[r].y * qr; y[2] += hv[r].z * qr; y[3] += hv[r].w * qr;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        x[j] += __shfl_xor_sync(0xffffffffu, x[j], 8);
        x[j] += __shfl_xor_sync(0xffffffffu, x[j], 16);
        y[j] += __shfl_xor_sync(0xffffffffu, y[j], 8);
        y[j] += __shfl_xor_sync(0xffffffffu, y[j], 16);
    }
    if (lane < 8) {
#pragma unroll
        for (int j = 0; j < 4; ++j) { rx[warp][4 * c4 + j] = x[j]; ry[warp][4 * c4 + j] = y[j]; }
    }
    __syncthreads();
    const float a = alpha[u], be = beta[u];
    if (tid < 32) {
        const float xs = rx[0][tid] + rx[1][tid] + rx[2][tid] + rx[3][tid];
        const float ys = ry[0][tid] + ry[1][tid] + ry[2][tid] + ry[3][tid];
        const float e = be * to_f(v[u * DV + col0 + tid]) - (b ? b[h] : 1.f) * be * feedback_scale(iplr, a) * xs;
        se[tid] = e;
        o[u * DV + col0 + tid] = from_f<T>(a * ys + e * skq);
    }
    __syncthreads();
    const float e0 = se[4 * c4], e1 = se[4 * c4 + 1], e2 = se[4 * c4 + 2], e3 = se[4 * c4 + 3];
#pragma unroll
    for (int r = 0; r < RPT; ++r) {
        const float kr = sk[rg + 16 * r];
        float4 nv;
        nv.x = a * hv[r].x + kr * e0;
        nv.y = a * hv[r].y + kr * e1;
        nv.z = a * hv[r].z + kr * e2;
        nv.w = a * hv[r].w + kr * e3;
        __stcs(st + (long long)(rg + 16 * r) * (DV / 4), nv);
    }
}

template <typename T, int DK, int DV>
static cudaError_t run_step(int Bd, int H, const void* q, const void* k, const void* v, const void* pf,
                            const float* alpha,
                            const float* beta, const float* b, const float* d, float* state, void* o,
                            bool iplr, cudaStream_t s) {
    const long long blocks = (long long)Bd * H * (DV / 32);
    k_step<T, DK, DV><<<(unsigned)blocks, 128, 0, s>>>(H, (const T*)q, (const T*)k, (const T*)v, (const T*)pf, alpha,
                                                       beta, b, d, state, (T*)o, iplr ? 1 : 0);
    return cudaGetLastError();
}

cudaError_t launch_recurrent_step(int Bd, int H, int dk, int dv, bool is_bf16, const void* q, const void* k,
                                  const void* v, const void* p, const float* alpha, const float* beta,
                                  const float* b, const float* d, float* state, void* o, bool iplr, cudaStream_t s) {
#define COMBA_STEP(T, DK, DV) \
    if (dk == DK && dv == DV) return run_step<T, DK, DV>(Bd, H, q, k, v, p, alpha, beta, b, d, state, o, iplr, s);
    if (is_bf16) {
        COMBA_STEP(bf16, 128, 128) COMBA_STEP(bf16, 128, 64) COMBA_STEP(bf16, 64, 128) COMBA_STEP(bf16, 64, 64)
        COMBA_STEP(bf16, 128, 256) COMBA_STEP(bf16, 256, 64) COMBA_STEP(bf16, 256, 128) COMBA_STEP(bf16, 256, 256)
    } else {
        COMBA_STEP(float, 128, 128) COMBA_STEP(float, 128, 64) COMBA_STEP(float, 64, 128) COMBA_STEP(float, 64, 64)
        COMBA_STEP(float, 128, 256) COMBA_STEP(float, 256, 64) COMBA_STEP(float, 256, 128) COMBA_STEP(float, 256, 256)
    }
#undef COMBA_STEP
    return cudaErrorInvalidValue;
}

}  // namespace comba
