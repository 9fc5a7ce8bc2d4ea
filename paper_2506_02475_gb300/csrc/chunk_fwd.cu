// Chunk-parallel Comba forward (section 3.3 of the paper):
//   k_chunk_map : chunk slots of (packed) sequences
//   k_prep      : per chunk, Gram matrix, UT inverse M by forward substitution,
//                 WY factors W = M Diag(btilde gamma_{r-1}) K, U = M Diag(beta) V
//                 (Eq. "prepare WY_M")
//   k_scan_fwd  : per (sequence, head, 64-column tile of dv), sequential over
//                 chunks: E = U - W H, H <- gamma_C H + Kbar^T E (inter-chunk
//                 state equation)
//   k_output    : per chunk, O = Diag(gamma) Q~ H + Tril(Q~ K^T * Gamma) E
//                 (output equation with Q~ = Q - d K)
#include "params.cuh"

namespace comba {

// ---------------------------------------------------------------- chunk map

// One block.  seq_first[n] = exclusive prefix of ceil(len_n / 64); slots past
// the last chunk get len = 0.  Invalid cu_seqlens are clamped (never read or
// write out of bounds); they only produce wrong results.
__global__ void __launch_bounds__(1024) k_chunk_map(ChunkParams p) {
    __shared__ int carry;
    __shared__ int wsum[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) carry = 0;
    __syncthreads();
    for (int base = 0; base < p.N; base += 1024) {
        const int n = base + tid;
        int nch = 0;
        if (n < p.N) {
            long long a = p.cu ? p.cu[n] : (long long)n * p.T;
            long long e = p.cu ? p.cu[n + 1] : (long long)(n + 1) * p.T;
            a = a < 0 ? 0 : (a > p.Ttot ? p.Ttot : a);
            e = e < a ? a : (e > p.Ttot ? p.Ttot : e);
            nch = (int)((e - a + kChunk - 1) / kChunk);
        }
        int x = nch;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) wsum[warp] = x;
        __syncthreads();
        if (warp == 0) {
            int w = wsum[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += y;
            }
            wsum[lane] = w;
        }
        __syncthreads();
        const int incl = x + (warp > 0 ? wsum[warp - 1] : 0) + carry;
        if (n < p.N) p.seq_first[n] = incl - nch;
        __syncthreads();
        if (tid == 1023) carry = incl;
        __syncthreads();
    }
    if (tid == 0) p.seq_first[p.N] = carry;
    __syncthreads();
    const int total = carry < p.slots ? carry : p.slots;
    for (int s = tid; s < p.slots; s += 1024) {
        SlotInfo si;
        si.start = 0; si.len = 0; si.seq = 0; si.idx = 0;
        if (s < total) {
            int lo = 0, hi = p.N - 1;  // last n with seq_first[n] <= s
            while (lo < hi) {
                const int mid = (lo + hi + 1) >> 1;
                if (p.seq_first[mid] <= s) lo = mid; else hi = mid - 1;
            }
            long long a = p.cu ? p.cu[lo] : (long long)lo * p.T;
            long long e = p.cu ? p.cu[lo + 1] : (long long)(lo + 1) * p.T;
            a = a < 0 ? 0 : (a > p.Ttot ? p.Ttot : a);
            e = e < a ? a : (e > p.Ttot ? p.Ttot : e);
            const int c = s - p.seq_first[lo];
            const long long st = a + (long long)c * kChunk;
            const long long l = e - st;
            si.start = (int)st;
            si.len = (int)(l > kChunk ? kChunk : (l < 0 ? 0 : l));
            si.seq = lo;
            si.idx = c;
        }
        p.slot_info[s] = si;
    }
}

// Store a fragment block to global memory (row-major, pitch ld), pairs of
// adjacent columns at a time; rows >= valid are skipped.
template <typename T, int NT>
__device__ __forceinline__ void frag_store_global(T* g, long long ld, int m0, int n0, const float (&acc)[NT][4],
                                                  int valid, float scale = 1.f) {
#pragma unroll
    for (int t = 0; t < NT; ++t)
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            const int r = m0 + frag_row(2 * hh);
            if (r >= valid) continue;
            const int c = n0 + frag_col(t, 0);
            T* dst = g + (long long)r * ld + c;
            dst[0] = from_f<T>(acc[t][2 * hh] * scale);
            dst[1] = from_f<T>(acc[t][2 * hh + 1] * scale);
        }
}

// ------------------------------------------------------------------ prep

template <typename T, int DK, int DV>
struct PrepSmem {
    static constexpr int PK = pitch<T>(DK), PV = pitch<T>(DV), PL = pitch<T>(64);
    static constexpr size_t bytes() {
        size_t o = 0;
        o = carve_bytes(o, sizeof(T) * 64 * PK);
        o = carve_bytes(o, sizeof(T) * 64 * PV);
        o = carve_bytes(o, sizeof(float) * 64 * 65);
        o = carve_bytes(o, sizeof(float) * 64 * 65);
        o = carve_bytes(o, sizeof(float) * 3 * 272);
        o = carve_bytes(o, sizeof(T) * 64 * PL);
        o = carve_bytes(o, sizeof(T) * 64 * PL);
        for (int i = 0; i < 4; ++i) o = carve_bytes(o, sizeof(float) * 64);
        return o;
    }
};

template <typename T, int DK, int DV>
__global__ void __launch_bounds__(128) k_prep(ChunkParams p) {
    using S = PrepSmem<T, DK, DV>;
    const int slot = blockIdx.x, h = blockIdx.y;
    const SlotInfo si = p.slot_info[slot];
    if (si.len <= 0) return;
    const int L = si.len;
    const long long t0 = si.start;
    const long long idx = (long long)slot * p.H + h;
    const int tid = threadIdx.x, warp = tid >> 5;

    extern __shared__ __align__(128) char smem[];
    SmemCarver sc(smem);
    T* sK = sc.take<T>(64 * S::PK);
    T* sV = sc.take<T>(64 * S::PV);
    float* sA = sc.take<float>(64 * 65);
    float* sM = sc.take<float>(64 * 65);
    float* sTmp = sc.take<float>(3 * 272);
    T* sMw = sc.take<T>(64 * S::PL);
    T* sMu = sc.take<T>(64 * S::PL);
    float* sG = sc.take<float>(64);
    float* sGm1 = sc.take<float>(64);
    float* sBt = sc.take<float>(64);
    float* sBe = sc.take<float>(64);

    load_tile_async<T>(sK, S::PK, (const T*)p.k + (t0 * p.H + h) * DK, (long long)p.H * DK, 64, DK, L, tid, 128);
    load_tile_async<T>(sV, S::PV, (const T*)p.v + (t0 * p.H + h) * DV, (long long)p.H * DV, 64, DV, L, tid, 128);
    cp_async_commit();
    if (warp == 0) chunk_log_cumsum(p.alpha + t0 * p.H + h, p.H, L, sG, sGm1);
    if (tid < 64) {
        const float be = tid < L ? p.beta[(t0 + tid) * p.H + h] : 0.f;
        sBe[tid] = be;
        sBt[tid] = (p.b ? p.b[h] : 1.f) * be;
    }
    cp_async_wait<0>();
    __syncthreads();

    // Strictly-lower A = Diag(btilde) (gamma_{r-1}/gamma_i * K K^T); exp taken only below the diagonal.
    {
        float acc[8][4];
        zero(acc);
        warp_gemm<true, true, 8>(acc, sK, S::PK, sK, S::PK, 16 * warp, 0, DK);
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = 16 * warp + frag_row(i), c = frag_col(t, i);
                float a = 0.f;
                if (c < r && r < L) a = sBt[r] * expf(sGm1[r] - sG[c]) * acc[t][i];
                sA[r * 65 + c] = a;
            }
    }
    // M = (I + A)^{-1} (the single UT inverse of the chunk), blocked forward substitution.
    unit_lower_inverse64(sA, sM, sTmp, tid);

    // Column-scaled copies for the two products: Mw = M Diag(btilde gamma_{r-1}), Mu = M Diag(beta).
    T* Mg = p.Mb ? (T*)p.Mb + idx * 4096 : nullptr;
    for (int e = tid; e < 64 * 64; e += 128) {
        const int r = e >> 6, c = e & 63;
        const float m = sM[r * 65 + c];
        sMw[r * S::PL + c] = from_f<T>(m * sBt[c] * expf(sGm1[c]));
        sMu[r * S::PL + c] = from_f<T>(m * sBe[c]);
        if (Mg) Mg[e] = from_f<T>(m);
    }
    if (tid < 64) p.Gb[idx * 64 + tid] = sG[tid];
    __syncthreads();

    {
        float acc[DK / 8][4];
        zero(acc);
        warp_gemm<true, false, DK / 8>(acc, sMw, S::PL, sK, S::PK, 16 * warp, 0, 64);
        frag_store_global<T, DK / 8>((T*)p.Wb + idx * 64 * DK, DK, 16 * warp, 0, acc, 64);
    }
    {
        float acc[DV / 8][4];
        zero(acc);
        warp_gemm<true, false, DV / 8>(acc, sMu, S::PL, sV, S::PV, 16 * warp, 0, 64);
        frag_store_global<T, DV / 8>((T*)p.Ub + idx * 64 * DV, DV, 16 * warp, 0, acc, 64);
    }
}

// ------------------------------------------------------------- state scan

template <typename T, int DK>
struct ScanSmem {
    static constexpr int PK = pitch<T>(DK), PT = pitch<T>(64);
    // per pipeline stage: W, K, U tile, G
    static constexpr size_t OW = 0;
    static constexpr size_t OK = align128(OW + sizeof(T) * 64 * PK);
    static constexpr size_t OU = align128(OK + sizeof(T) * 64 * PK);
    static constexpr size_t OG = align128(OU + sizeof(T) * 64 * PT);
    static constexpr size_t STAGE = align128(OG + sizeof(float) * 64);
    static constexpr size_t OH = 2 * STAGE;                                  // H tile (storage type)
    static constexpr size_t OE = align128(OH + sizeof(T) * DK * PT);         // scaled E tile
    static constexpr size_t bytes() { return OE + sizeof(T) * 64 * PT; }
};

__device__ __forceinline__ void seq_range(const ChunkParams& p, int n, long long& start, long long& len) {
    long long a = p.cu ? p.cu[n] : (long long)n * p.T;
    long long e = p.cu ? p.cu[n + 1] : (long long)(n + 1) * p.T;
    a = a < 0 ? 0 : (a > p.Ttot ? p.Ttot : a);
    e = e < a ? a : (e > p.Ttot ? p.Ttot : e);
    start = a;
    len = e - a;
}

// The sequential inter-chunk recurrence: E_n = U_n - W_n H_n, H_{n+1} = gamma_C H_n + Kbar_n^T E_n.
// One CTA owns a 64-column tile of H (fp32, in registers) for one (sequence, head); the
// next chunk's W, K, U tile and log-decays are prefetched while the current chunk computes.
template <typename T, int DK, int DV>
__global__ void __launch_bounds__(128) k_scan_fwd(ChunkParams p) {
    using S = ScanSmem<T, DK>;
    constexpr int MT = DK / 64;  // 16-row m-tiles per warp
    const int jt = blockIdx.x % (DV / 64), n = blockIdx.x / (DV / 64), h = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int c0 = jt * 64;

    extern __shared__ __align__(128) char smem[];
    auto sW = [&](int st) { return reinterpret_cast<T*>(smem + st * S::STAGE + S::OW); };
    auto sK = [&](int st) { return reinterpret_cast<T*>(smem + st * S::STAGE + S::OK); };
    auto sU = [&](int st) { return reinterpret_cast<T*>(smem + st * S::STAGE + S::OU); };
    auto sG = [&](int st) { return reinterpret_cast<float*>(smem + st * S::STAGE + S::OG); };
    T* sH = reinterpret_cast<T*>(smem + S::OH);
    T* sE = reinterpret_cast<T*>(smem + S::OE);

    float hs[MT][8][4];
    const float* h0 = p.h0 ? p.h0 + ((long long)n * p.H + h) * DK * DV : nullptr;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt)
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = (warp * MT + mt) * 16 + frag_row(i), c = c0 + frag_col(t, i);
                hs[mt][t][i] = h0 ? h0[(long long)r * DV + c] : 0.f;
            }

    long long start, len;
    seq_range(p, n, start, len);
    const int s0 = p.seq_first[n];
    int nch = (int)((len + kChunk - 1) / kChunk);
    if (s0 + nch > p.slots) nch = p.slots - s0 > 0 ? p.slots - s0 : 0;

    auto issue = [&](int c, int st) {
        const long long idx = (long long)(s0 + c) * p.H + h;
        const long long t0 = start + (long long)c * kChunk;
        const int L = (int)(len - (long long)c * kChunk < kChunk ? len - (long long)c * kChunk : kChunk);
        load_tile_async<T>(sW(st), S::PK, (const T*)p.Wb + idx * 64 * DK, DK, 64, DK, 64, tid, 128);
        load_tile_async<T>(sK(st), S::PK, (const T*)p.k + (t0 * p.H + h) * DK, (long long)p.H * DK, 64, DK, L, tid,
                           128);
        load_tile_async<T>(sU(st), S::PT, (const T*)p.Ub + idx * 64 * DV + c0, DV, 64, 64, 64, tid, 128);
        if (tid < 16) cp_async16(sG(st) + 4 * tid, p.Gb + idx * 64 + 4 * tid, true);
        cp_async_commit();
    };
    if (nch > 0) issue(0, 0);

    for (int c = 0; c < nch; ++c) {
        const int st = c & 1;
        const int L = (int)(len - (long long)c * kChunk < kChunk ? len - (long long)c * kChunk : kChunk);
        const long long idx = (long long)(s0 + c) * p.H + h;
        if (c + 1 < nch) {
            issue(c + 1, st ^ 1);
            cp_async_wait<1>();
        } else {
            cp_async_wait<0>();
        }
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
            const int m0 = (warp * MT + mt) * 16;
            frag_store<T, 8>(sH, S::PT, m0, 0, hs[mt]);
            frag_store_global<T, 8>((T*)p.Hb + idx * DK * DV + c0, DV, m0, 0, hs[mt], DK);
        }
        __syncthreads();

        const float* G = sG(st);
        const float gL = G[L - 1];
        {
            float e[8][4];
            zero(e);
            warp_gemm<true, false, 8>(e, sW(st), S::PK, sH, S::PT, 16 * warp, 0, DK);
            T* Eg = (T*)p.Eb + idx * 64 * DV + c0;
            const T* U = sU(st);
#pragma unroll
            for (int t = 0; t < 8; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = 16 * warp + frag_row(i), cc = frag_col(t, i);
                    const float ev = to_f(U[r * S::PT + cc]) - e[t][i];
                    Eg[(long long)r * DV + cc] = from_f<T>(ev);
                    sE[r * S::PT + cc] = from_f<T>(r < L ? ev * expf(gL - G[r]) : 0.f);
                }
        }
        __syncthreads();

        const float dec = expf(gL);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
            for (int t = 0; t < 8; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) hs[mt][t][i] *= dec;
            warp_gemm<false, false, 8>(hs[mt], sK(st), S::PK, sE, S::PT, (warp * MT + mt) * 16, 0, 64);
        }
        __syncthreads();
    }

    if (p.hT) {
        float* hT = p.hT + ((long long)n * p.H + h) * DK * DV;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt)
#pragma unroll
            for (int t = 0; t < 8; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = (warp * MT + mt) * 16 + frag_row(i), cc = c0 + frag_col(t, i);
                    hT[(long long)r * DV + cc] = hs[mt][t][i];
                }
    }
}

// ---------------------------------------------------------------- output

template <typename T, int DK, int DV>
struct OutSmem {
    static constexpr int PK = pitch<T>(DK), PV = pitch<T>(DV), PL = pitch<T>(64);
    static constexpr size_t bytes() {
        size_t o = 0;
        o = carve_bytes(o, sizeof(T) * 64 * PK);   // Q~
        o = carve_bytes(o, sizeof(T) * 64 * PK);   // K
        o = carve_bytes(o, sizeof(T) * 64 * PL);   // P
        o = carve_bytes(o, sizeof(T) * DK * PV);   // H
        o = carve_bytes(o, sizeof(T) * 64 * PV);   // E
        o = carve_bytes(o, sizeof(float) * 64);    // G
        return o;
    }
};

template <typename T, int DK, int DV>
__global__ void __launch_bounds__(128) k_output(ChunkParams p) {
    using S = OutSmem<T, DK, DV>;
    const int slot = blockIdx.x, h = blockIdx.y;
    const SlotInfo si = p.slot_info[slot];
    if (si.len <= 0) return;
    const int L = si.len;
    const long long t0 = si.start;
    const long long idx = (long long)slot * p.H + h;
    const int tid = threadIdx.x, warp = tid >> 5;

    extern __shared__ __align__(128) char smem[];
    SmemCarver sc(smem);
    T* sQ = sc.take<T>(64 * S::PK);
    T* sK = sc.take<T>(64 * S::PK);
    T* sP = sc.take<T>(64 * S::PL);
    T* sH = sc.take<T>(DK * S::PV);
    T* sE = sc.take<T>(64 * S::PV);
    float* sG = sc.take<float>(64);

    load_tile_async<T>(sQ, S::PK, (const T*)p.q + (t0 * p.H + h) * DK, (long long)p.H * DK, 64, DK, L, tid, 128);
    load_tile_async<T>(sK, S::PK, (const T*)p.k + (t0 * p.H + h) * DK, (long long)p.H * DK, 64, DK, L, tid, 128);
    load_tile_async<T>(sH, S::PV, (const T*)p.Hb + idx * DK * DV, DV, DK, DV, DK, tid, 128);
    load_tile_async<T>(sE, S::PV, (const T*)p.Eb + idx * 64 * DV, DV, 64, DV, 64, tid, 128);
    cp_async_commit();
    if (tid < 64) sG[tid] = p.Gb[idx * 64 + tid];
    cp_async_wait<0>();
    __syncthreads();
    const float dh = p.d[h];
    for (int e = tid; e < 64 * DK; e += 128) {
        const int r = e / DK, c = e % DK;
        sQ[r * S::PK + c] = from_f<T>(to_f(sQ[r * S::PK + c]) - dh * to_f(sK[r * S::PK + c]));
    }
    __syncthreads();

    {
        float s[8][4];
        zero(s);
        warp_gemm<true, true, 8>(s, sQ, S::PK, sK, S::PK, 16 * warp, 0, DK);
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = 16 * warp + frag_row(i), c = frag_col(t, i);
                const float v = (c <= r && r < L) ? s[t][i] * expf(sG[r] - sG[c]) : 0.f;
                sP[r * S::PL + c] = from_f<T>(v);
            }
    }
    __syncthreads();

    float o[DV / 8][4];
    zero(o);
    warp_gemm<true, false, DV / 8>(o, sQ, S::PK, sH, S::PV, 16 * warp, 0, DK);
    {
        const float e0 = expf(sG[16 * warp + frag_row(0)]);
        const float e1 = expf(sG[16 * warp + frag_row(2)]);
#pragma unroll
        for (int t = 0; t < DV / 8; ++t) {
            o[t][0] *= e0; o[t][1] *= e0;
            o[t][2] *= e1; o[t][3] *= e1;
        }
    }
    warp_gemm<true, false, DV / 8>(o, sP, S::PL, sE, S::PV, 16 * warp, 0, 64);
    frag_store_global<T, DV / 8>((T*)p.o + (t0 * p.H + h) * DV, (long long)p.H * DV, 16 * warp, 0, o, L);
}

// -------------------------------------------------------------- launchers

template <typename T, int DK, int DV>
static cudaError_t run_fwd(const ChunkParams& p, bool for_backward, cudaStream_t s, int ev0) {
    const size_t sm_prep = PrepSmem<T, DK, DV>::bytes();
    const size_t sm_scan = ScanSmem<T, DK>::bytes();
    const size_t sm_out = OutSmem<T, DK, DV>::bytes();
    cudaError_t e;
    if ((e = cudaFuncSetAttribute(k_prep<T, DK, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_prep)))
        return e;
    if ((e = cudaFuncSetAttribute(k_scan_fwd<T, DK, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_scan)))
        return e;
    if ((e = cudaFuncSetAttribute(k_output<T, DK, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_out)))
        return e;
    mark(p, ev0, s);
    if (p.slots > 0) k_prep<T, DK, DV><<<dim3(p.slots, p.H), 128, sm_prep, s>>>(p);
    if ((e = cudaGetLastError())) return e;
    mark(p, ev0 + 1, s);
    k_scan_fwd<T, DK, DV><<<dim3((DV / 64) * p.N, p.H), 128, sm_scan, s>>>(p);
    if ((e = cudaGetLastError())) return e;
    if (!for_backward) {
        mark(p, ev0 + 2, s);
        if (p.slots > 0) k_output<T, DK, DV><<<dim3(p.slots, p.H), 128, sm_out, s>>>(p);
        if ((e = cudaGetLastError())) return e;
        mark(p, ev0 + 3, s);
    }
    return cudaSuccess;
}

cudaError_t launch_chunk_map(const ChunkParams& p, cudaStream_t s) {
    k_chunk_map<<<1, 1024, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_fwd(const ChunkParams& p, bool is_bf16, bool for_backward, cudaStream_t s, int ev0) {
    if (is_bf16) {
        if (p.dk == 128 && p.dv == 128) return run_fwd<bf16, 128, 128>(p, for_backward, s, ev0);
        if (p.dk == 128 && p.dv == 64) return run_fwd<bf16, 128, 64>(p, for_backward, s, ev0);
        if (p.dk == 64 && p.dv == 128) return run_fwd<bf16, 64, 128>(p, for_backward, s, ev0);
        if (p.dk == 64 && p.dv == 64) return run_fwd<bf16, 64, 64>(p, for_backward, s, ev0);
    } else {
        if (p.dk == 128 && p.dv == 128) return run_fwd<float, 128, 128>(p, for_backward, s, ev0);
        if (p.dk == 128 && p.dv == 64) return run_fwd<float, 128, 64>(p, for_backward, s, ev0);
        if (p.dk == 64 && p.dv == 128) return run_fwd<float, 64, 128>(p, for_backward, s, ev0);
        if (p.dk == 64 && p.dv == 64) return run_fwd<float, 64, 64>(p, for_backward, s, ev0);
    }
    return cudaErrorInvalidValue;
}

size_t fwd_smem_bytes(int kernel, bool is_bf16, int dk, int dv) {
#define COMBA_SM(T, DK, DV)                                                                          \
    if (dk == DK && dv == DV)                                                                        \
        return kernel == 0 ? PrepSmem<T, DK, DV>::bytes()                                            \
                           : (kernel == 1 ? ScanSmem<T, DK>::bytes() : OutSmem<T, DK, DV>::bytes());
    if (is_bf16) {
        COMBA_SM(bf16, 128, 128) COMBA_SM(bf16, 128, 64) COMBA_SM(bf16, 64, 128) COMBA_SM(bf16, 64, 64)
    } else {
        COMBA_SM(float, 128, 128) COMBA_SM(float, 128, 64) COMBA_SM(float, 64, 128) COMBA_SM(float, 64, 64)
    }
#undef COMBA_SM
    return 0;
}

}  // namespace comba
