// Gate and normalisation prologue / epilogue around the chunk recurrence.
//
// Forward prologue over (token, head) rows, in one pass over the raw inputs (section 3.1
// gates; L2-normalised q and k of the neural-architecture section):
//     q_hat = q / sqrt(|q|^2 + eps),  k_hat = k / sqrt(|k|^2 + eps),
//     alpha = exp(-a_h softplus(g_alpha + c_h)),  beta = sigmoid(g_beta),
// and b = sigmoid(b_raw) per head.  The chunk kernels then run on (q_hat, k_hat, alpha,
// beta, b).  Backward epilogue, same rows: the chunk backward's gradients w.r.t. q_hat,
// k_hat, alpha, beta map back to the raw inputs,
//     dx = (dx_hat - x_hat (x_hat . dx_hat)) / sqrt(|x|^2 + eps),
//     dg_alpha = -a_h alpha sigmoid(g_alpha + c_h) dalpha,   dg_beta = beta (1 - beta) dbeta,
// and each row's contributions to da_h (-alpha softplus(g_alpha + c_h) dalpha) and dc_h
// (dg_alpha) are written out and summed per head in a fixed order by two small reduction
// kernels (token blocks, then heads); db_raw = b (1 - b) db.
//
// Both elementwise passes are HBM-bound (the prologue moves 4 row-vectors per row, the
// epilogue 6).  A block streams 64-row stages of its inputs through a ring of shared-memory
// slots with cp.async, several stages ahead of its arithmetic, so that the bytes in flight
// per SM do not depend on how many registers a warp can spare.
#include "params.cuh"

namespace comba {

namespace {

__device__ __forceinline__ float softplus_f(float x) { return x > 20.f ? x : log1pf(expf(x)); }
__device__ __forceinline__ float sigmoid_f(float x) { return 1.f / (1.f + expf(-x)); }

// 16-byte global->shared copy of which only the first `bytes` (0..16) are read; the rest
// of the 16 shared bytes are zero-filled.
__device__ __forceinline__ void cp_async_part(void* s, const void* g, int bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(smem_u32(s)), "l"(g), "r"(bytes)
                 : "memory");
}

// Rows of one stage of a [rows, D] array (row r of the stage at smem + r * D).
template <typename T, int D>
__device__ __forceinline__ void stage_rows(T* smem, const T* g, long long row0, int nr, int tid, int nthr) {
    constexpr int CH = D * (int)sizeof(T) / 16;   // 16-byte chunks per row
    const char* src = reinterpret_cast<const char*>(g + row0 * D);
    char* dst = reinterpret_cast<char*>(smem);
    for (int i = tid; i < nr * CH; i += nthr) cp_async16(dst + 16 * i, src + 16 * i, true);
}
// A stage of a per-row float array (rows >= nr zero-filled); `tid` in [0, rows / 4) picks the chunk.
__device__ __forceinline__ void stage_scalars(float* smem, const float* g, long long row0, int nr, int tid) {
    const int bytes = 4 * (nr - 4 * tid);
    if (bytes > 0) cp_async_part(smem + 4 * tid, g + row0 + 4 * tid, bytes < 16 ? bytes : 16);
}

// A row split over a group of 8 lanes: lane l of the group owns the 16-byte chunks
// c * 8 + l (c < C) of the row, E elements in all, so that one warp instruction covers
// four rows and each 8-lane store writes a full 128-byte line.
template <typename T, int D>
struct Part {
    static constexpr int V = 16 / (int)sizeof(T);            // elements per chunk
    static constexpr int C = D * (int)sizeof(T) / 16 / 8;    // chunks per lane
    static constexpr int E = C * V;                          // elements per lane
};

template <typename T, int D>
__device__ __forceinline__ void load_part(const T* row, float (&x)[Part<T, D>::E], int l) {
    using P = Part<T, D>;
#pragma unroll
    for (int c = 0; c < P::C; ++c) {
        union { uint4 v; T e[P::V]; } u;
        u.v = *reinterpret_cast<const uint4*>(row + (c * 8 + l) * P::V);
#pragma unroll
        for (int i = 0; i < P::V; ++i) x[c * P::V + i] = to_f(u.e[i]);
    }
}
template <typename T, int D>
__device__ __forceinline__ void store_part(T* row, const float (&x)[Part<T, D>::E], int l) {
    using P = Part<T, D>;
#pragma unroll
    for (int c = 0; c < P::C; ++c) {
        union { uint4 v; T e[P::V]; } u;
#pragma unroll
        for (int i = 0; i < P::V; ++i) u.e[i] = from_f<T>(x[c * P::V + i]);
        *reinterpret_cast<uint4*>(row + (c * 8 + l) * P::V) = u.v;
    }
}
__device__ __forceinline__ float group_sum(float s) {   // over the 8 lanes of a group
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 4);
    return s;
}

// one 8-lane group per row: dx = (dx_hat - x_hat (x_hat . dx_hat)) / n,  n = sqrt(|x|^2 + eps)
template <typename T, int D>
__device__ __forceinline__ void unnormalise_part(const T* xs, const T* gs, T* dx, bool store, float eps, int l) {
    constexpr int E = Part<T, D>::E;
    float x[E], g[E];
    load_part<T, D>(xs, x, l);
    load_part<T, D>(gs, g, l);
    float s = 0.f, dot = 0.f;
#pragma unroll
    for (int i = 0; i < E; ++i) { s = fmaf(x[i], x[i], s); dot = fmaf(x[i], g[i], dot); }
    const float inv = rsqrtf(group_sum(s) + eps);
    dot = group_sum(dot) * inv;   // x_hat . dx_hat
#pragma unroll
    for (int i = 0; i < E; ++i) g[i] = (g[i] - x[i] * inv * dot) * inv;
    if (store) store_part<T, D>(dx, g, l);
}

constexpr int kGateThreads = 512;   // 16 warps, four rows of a stage each (one per 8-lane group)
constexpr int kStageRows = kGateThreads / 8;
constexpr int kRingBytes = 200 * 1024;

// Ring depth: as many stages as fit in kRingBytes, 2..8.
template <int STAGE_BYTES>
struct Ring {
    static constexpr int fit = kRingBytes / STAGE_BYTES;
    static constexpr int n = fit > 8 ? 8 : (fit < 2 ? 2 : fit);
    static constexpr int bytes = n * STAGE_BYTES;
};

template <typename T, int DK>
struct ProStage {   // one slot of the prologue ring
    T q[kStageRows * DK], k[kStageRows * DK];
    float ga[kStageRows], gb[kStageRows];
};
template <typename T, int DK, int NP>
struct EpiStage {   // one slot of the epilogue ring: NP (x, dx_hat) pairs, q then k
    T x[NP][kStageRows * DK], dx[NP][kStageRows * DK];
    float ga[kStageRows], al[kStageRows], dal[kStageRows], be[kStageRows], dbe[kStageRows];
};

}  // namespace

// Stages s = blockIdx.x + i * gridDim.x of kStageRows rows; the ring runs Ring::n - 1 stages ahead.
template <typename T, int DK>
__global__ void __launch_bounds__(kGateThreads) k_gate_prologue(GateParams g) {
    using S = ProStage<T, DK>;
    constexpr int NS = Ring<(int)sizeof(S)>::n;
    extern __shared__ __align__(128) unsigned char gate_smem[];
    S* ring = reinterpret_cast<S*>(gate_smem);
    const int tid = threadIdx.x;
    if (blockIdx.x == 0)
        for (int h = tid; h < g.H; h += kGateThreads) g.bgate[h] = sigmoid_f(g.b_raw[h]);
    const long long nstages = (g.rows + kStageRows - 1) / kStageRows;
    const long long mine = nstages > blockIdx.x ? (nstages - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
    auto issue = [&](long long i) {
        if (i < mine) {
            const long long row0 = (blockIdx.x + i * gridDim.x) * kStageRows;
            const int nr = (int)(g.rows - row0 < kStageRows ? g.rows - row0 : kStageRows);
            S& st = ring[i % NS];
            stage_rows<T, DK>(st.q, (const T*)g.q, row0, nr, tid, kGateThreads);
            stage_rows<T, DK>(st.k, (const T*)g.k, row0, nr, tid, kGateThreads);
            constexpr int SC = kStageRows / 4;   // 16-byte chunks of a stage's per-row floats
            if (tid < SC) stage_scalars(st.ga, g.g_alpha, row0, nr, tid);
            else if (tid < 2 * SC) stage_scalars(st.gb, g.g_beta, row0, nr, tid - SC);
        }
        cp_async_commit();
    };
    for (int i = 0; i < NS - 1; ++i) issue(i);
    for (long long i = 0; i < mine; ++i) {
        cp_async_wait<NS - 2>();
        __syncthreads();            // stage i landed; every warp is done with slot (i - 1) % NS
        issue(i + NS - 1);
        const S& st = ring[i % NS];
        const long long row0 = (blockIdx.x + i * gridDim.x) * kStageRows;
        const int nr = (int)(g.rows - row0 < kStageRows ? g.rows - row0 : kStageRows);
        const int sr = tid - (kGateThreads - kStageRows);   // the last warps' threads: one row's gates each
        if (sr >= 0 && sr < nr) {
            const long long row = row0 + sr;
            const int h = (int)(row % g.H);
            g.alpha[row] = expf(-g.a[h] * softplus_f(st.ga[sr] + g.c[h]));
            g.beta[row] = sigmoid_f(st.gb[sr]);
        }
        {
            constexpr int E = Part<T, DK>::E;
            const int r = tid >> 3, l = tid & 7;
            float xq[E], xk[E];
            load_part<T, DK>(st.q + r * DK, xq, l);
            load_part<T, DK>(st.k + r * DK, xk, l);
            float sq = 0.f, sk = 0.f;
#pragma unroll
            for (int e = 0; e < E; ++e) { sq = fmaf(xq[e], xq[e], sq); sk = fmaf(xk[e], xk[e], sk); }
            const float iq = rsqrtf(group_sum(sq) + g.eps), ik = rsqrtf(group_sum(sk) + g.eps);
#pragma unroll
            for (int e = 0; e < E; ++e) { xq[e] *= iq; xk[e] *= ik; }
            if (r < nr) {
                store_part<T, DK>((T*)g.qh + (row0 + r) * DK, xq, l);
                store_part<T, DK>((T*)g.kh + (row0 + r) * DK, xk, l);
            }
        }
    }
    cp_async_wait<0>();
}

// NP = 2: q and k in one pass.  NP = 1 (head dim 256, whose four [64][256] tiles would not fit
// two ring slots): pass 0 takes q and the gates, pass 1 k.
template <typename T, int DK, int NP>
__global__ void __launch_bounds__(kGateThreads) k_gate_epilogue(GateParams g, int pass) {
    using S = EpiStage<T, DK, NP>;
    const bool gates = pass == 0;
    // pair j's raw input, chunk-backward gradient and output
    auto src = [&](int j) { return (NP == 2 ? j : pass) == 0 ? (const T*)g.q : (const T*)g.k; };
    auto dsrc = [&](int j) { return (NP == 2 ? j : pass) == 0 ? (const T*)g.dqh : (const T*)g.dkh; };
    auto dst = [&](int j) { return (NP == 2 ? j : pass) == 0 ? (T*)g.dq : (T*)g.dk; };
    constexpr int NS = Ring<(int)sizeof(S)>::n;
    extern __shared__ __align__(128) unsigned char gate_smem[];
    S* ring = reinterpret_cast<S*>(gate_smem);
    const int tid = threadIdx.x;
    const long long nstages = (g.rows + kStageRows - 1) / kStageRows;
    const long long mine = nstages > blockIdx.x ? (nstages - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
    auto issue = [&](long long i) {
        if (i < mine) {
            const long long row0 = (blockIdx.x + i * gridDim.x) * kStageRows;
            const int nr = (int)(g.rows - row0 < kStageRows ? g.rows - row0 : kStageRows);
            S& st = ring[i % NS];
#pragma unroll
            for (int j = 0; j < NP; ++j) {
                stage_rows<T, DK>(st.x[j], src(j), row0, nr, tid, kGateThreads);
                stage_rows<T, DK>(st.dx[j], dsrc(j), row0, nr, tid, kGateThreads);
            }
            constexpr int SC = kStageRows / 4;   // 16-byte chunks of a stage's per-row floats
            if (gates) {
                if (tid < SC) stage_scalars(st.ga, g.g_alpha, row0, nr, tid);
                else if (tid < 2 * SC) stage_scalars(st.al, g.alpha, row0, nr, tid - SC);
                else if (tid < 3 * SC) stage_scalars(st.dal, g.dalpha, row0, nr, tid - 2 * SC);
                else if (tid < 4 * SC) stage_scalars(st.be, g.beta, row0, nr, tid - 3 * SC);
                else if (tid < 5 * SC) stage_scalars(st.dbe, g.dbeta, row0, nr, tid - 4 * SC);
            }
        }
        cp_async_commit();
    };
    for (int i = 0; i < NS - 1; ++i) issue(i);
    for (long long i = 0; i < mine; ++i) {
        cp_async_wait<NS - 2>();
        __syncthreads();            // stage i landed; every warp is done with slot (i - 1) % NS
        issue(i + NS - 1);
        const S& st = ring[i % NS];
        const long long row0 = (blockIdx.x + i * gridDim.x) * kStageRows;
        const int nr = (int)(g.rows - row0 < kStageRows ? g.rows - row0 : kStageRows);
        const int sr = tid - (kGateThreads - kStageRows);   // the last warps' threads: one row's gates each
        if (gates && sr >= 0 && sr < nr) {
            const long long row = row0 + sr;
            const int h = (int)(row % g.H);
            const float z = st.ga[sr] + g.c[h], al = st.al[sr], dal = st.dal[sr], be = st.be[sr];
            const float dga = dal * (-g.a[h] * al * sigmoid_f(z));
            g.dg_alpha[row] = dga;
            g.dg_beta[row] = st.dbe[sr] * be * (1.f - be);
            g.da_rows[row] = dal * (-al * softplus_f(z));
            g.dc_rows[row] = dga;
        }
        {
            const int r = tid >> 3, l = tid & 7;
#pragma unroll
            for (int j = 0; j < NP; ++j)
                unnormalise_part<T, DK>(st.x[j] + r * DK, st.dx[j] + r * DK, dst(j) + (row0 + r) * DK, r < nr, g.eps, l);
        }
    }
    cp_async_wait<0>();
}

// da, dc: per-row contributions summed per head in a fixed order.  First level: block
// (c, head group) sums tokens [kRedTokens c, kRedTokens (c + 1)) of 32 heads (lane = head,
// warp w takes tokens w, w + 8, ...) into part[h * C + c].
constexpr int kRedTokens = 64;

__global__ void __launch_bounds__(256) k_gate_reduce_tokens(GateParams g, int C) {
    __shared__ float sa[8][32], sc[8][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int h = blockIdx.y * 32 + lane;
    const long long tokens = g.rows / g.H;
    float a = 0.f, c = 0.f;
    if (h < g.H) {
        float va[kRedTokens / 8], vc[kRedTokens / 8];
#pragma unroll
        for (int i = 0; i < kRedTokens / 8; ++i) {
            const long long t = (long long)blockIdx.x * kRedTokens + warp + 8 * i;
            va[i] = t < tokens ? g.da_rows[t * g.H + h] : 0.f;
            vc[i] = t < tokens ? g.dc_rows[t * g.H + h] : 0.f;
        }
#pragma unroll
        for (int i = 0; i < kRedTokens / 8; ++i) { a += va[i]; c += vc[i]; }
    }
    sa[warp][lane] = a;
    sc[warp][lane] = c;
    __syncthreads();
    if (warp == 0 && h < g.H) {
        float ta = 0.f, tc = 0.f;
        for (int w = 0; w < 8; ++w) { ta += sa[w][lane]; tc += sc[w][lane]; }
        g.da_part[(long long)h * C + blockIdx.x] = ta;
        g.dc_part[(long long)h * C + blockIdx.x] = tc;
    }
}

// Second level, one block per head: da, dc = fixed-order sums of the head's C partials;
// db_raw = b (1 - b) db.
__global__ void __launch_bounds__(256) k_gate_reduce(GateParams g, int nblk) {
    __shared__ float sa[256], sc[256];
    const int h = blockIdx.x, tid = threadIdx.x;
    float a = 0.f, c = 0.f;
    for (int t = tid; t < nblk; t += 256) {
        a += g.da_part[(long long)h * nblk + t];
        c += g.dc_part[(long long)h * nblk + t];
    }
    sa[tid] = a;
    sc[tid] = c;
    __syncthreads();
    for (int s = 128; s > 0; s >>= 1) {
        if (tid < s) { sa[tid] += sa[tid + s]; sc[tid] += sc[tid + s]; }
        __syncthreads();
    }
    if (tid == 0) {
        g.da[h] = sa[0];
        g.dc[h] = sc[0];
        const float b = g.bgate[h];
        if (g.db_raw) g.db_raw[h] = g.db ? g.db[h] * b * (1.f - b) : 0.f;
    }
}

// Grid-stride launch over 64-row stages: one block per SM (the ring fills shared memory).
template <typename K, typename... A>
static cudaError_t launch_ring(K kernel, int smem, const GateParams& g, cudaStream_t s, A... args) {
    int dev = 0, nsm = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) || (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) ||
        (e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem)))
        return e;
    const long long nstages = (g.rows + kStageRows - 1) / kStageRows;
    const long long grid = nstages < nsm ? (nstages > 0 ? nstages : 1) : nsm;
    kernel<<<(unsigned)grid, kGateThreads, smem, s>>>(g, args...);
    return cudaGetLastError();
}

template <typename T, int DK>
static cudaError_t run_prologue(const GateParams& g, cudaStream_t s) {
    static_assert(Ring<(int)sizeof(ProStage<T, DK>)>::bytes <= 227 * 1024, "prologue ring exceeds shared memory");
    return launch_ring(k_gate_prologue<T, DK>, Ring<(int)sizeof(ProStage<T, DK>)>::bytes, g, s);
}
template <typename T, int DK>
static cudaError_t run_epilogue(const GateParams& g, cudaStream_t s) {
    constexpr int one = Ring<(int)sizeof(EpiStage<T, DK, 2>)>::bytes;
    if constexpr (one <= 227 * 1024) {
        return launch_ring(k_gate_epilogue<T, DK, 2>, one, g, s, 0);
    } else {
        constexpr int two = Ring<(int)sizeof(EpiStage<T, DK, 1>)>::bytes;
        static_assert(two <= 227 * 1024, "epilogue ring exceeds shared memory");
        cudaError_t e = launch_ring(k_gate_epilogue<T, DK, 1>, two, g, s, 0);
        return e ? e : launch_ring(k_gate_epilogue<T, DK, 1>, two, g, s, 1);
    }
}

cudaError_t launch_gate_prologue(const GateParams& g, bool is_bf16, int dk, cudaStream_t s) {
    if (is_bf16) {
        if (dk == 256) return run_prologue<bf16, 256>(g, s);
        return dk == 128 ? run_prologue<bf16, 128>(g, s) : run_prologue<bf16, 64>(g, s);
    }
    return dk == 128 ? run_prologue<float, 128>(g, s) : run_prologue<float, 64>(g, s);
}

cudaError_t launch_gate_epilogue(const GateParams& g, bool is_bf16, int dk, cudaStream_t s) {
    cudaError_t e;
    if (g.rows > 0) {
        if (is_bf16) e = dk == 256 ? run_epilogue<bf16, 256>(g, s)
                                   : (dk == 128 ? run_epilogue<bf16, 128>(g, s) : run_epilogue<bf16, 64>(g, s));
        else if (dk == 64) e = run_epilogue<float, 64>(g, s);   // the fp32 backward runs dk = dv = 64 only
        else return cudaErrorInvalidValue;
        if (e) return e;
    }
    const long long tokens = g.rows / g.H;
    const int C = (int)((tokens + kRedTokens - 1) / kRedTokens);
    if (C > 0) {
        k_gate_reduce_tokens<<<dim3(C, (g.H + 31) / 32), 256, 0, s>>>(g, C);
        if ((e = cudaGetLastError())) return e;
    }
    k_gate_reduce<<<g.H, 256, 0, s>>>(g, C);
    return cudaGetLastError();
}

}  // namespace comba
