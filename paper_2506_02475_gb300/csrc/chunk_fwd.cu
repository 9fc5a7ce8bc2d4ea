// Chunk-parallel Comba forward (section 3.2 of the paper):
//   k_chunk_map : chunk slots of (packed) sequences
//   k_prep      : per chunk, the decay-masked btilde-scaled Gram matrix, its
//                 UT inverse M, the WY factors W = M Diag(btilde gamma_{r-1}) K
//                 and U = M Diag(beta) V (Eq. "prepare WY_M"), and the chunk's
//                 affine state map H -> gamma_C H + Atilde H + B with
//                 Atilde = -Kbar^T W, B = Kbar^T U (the inter-chunk state
//                 equation with Kbar = Diag(gamma_C / gamma_r) K)
//   (scan.cu)   : the sequential scan of those maps
//   k_output    : per chunk, E = U - W H_n and the output equation
//                 O = Diag(gamma) Q~ H_n + Tril(Q~ K^T * Gamma) E, Q~ = Q - d K
// These serve the shapes off the tcgen05 kernels (chunk_tc.cu for bf16 d = 128,
// wide_tc.cu for bf16 head dim 256).
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
    if (tid == 0) {
        carry = 0;
        if (p.err) *p.err = 0;
    }
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
    // dk <= 128: the chunk map (Atilde, B^T) is formed from Kbar-scaled copies of W and U that
    // reuse the A and M regions; at dk = 256 there is no map and those regions hold fp32 only.
    static constexpr bool kMap = DK <= 128;
    static constexpr int PK = pitch<T>(DK), PV = pitch<T>(DV), PL = pitch<T>(64);
    static constexpr size_t F64 = sizeof(float) * 64 * 65;
    static constexpr size_t RA = kMap && sizeof(T) * 64 * PK > F64 ? sizeof(T) * 64 * PK : F64;
    static constexpr size_t RM = kMap && sizeof(T) * 64 * PV > F64 ? sizeof(T) * 64 * PV : F64;
    static constexpr size_t OK = 0;
    static constexpr size_t OV = align128(OK + sizeof(T) * 64 * PK);
    static constexpr size_t OA = align128(OV + sizeof(T) * 64 * PV);   // A (fp32), later Diag(s) W
    static constexpr size_t OM = align128(OA + RA);                    // M (fp32), later Diag(s) U
    static constexpr size_t OT = align128(OM + RM);                    // inverse scratch
    static constexpr size_t OMW = align128(OT + sizeof(float) * 3 * 272);
    static constexpr size_t OMU = align128(OMW + sizeof(T) * 64 * PL);
    static constexpr size_t OF = align128(OMU + sizeof(T) * 64 * PL);  // G, Gm1, btilde, beta, s
    static constexpr size_t OP = align128(OF + sizeof(float) * 64 * 5);  // Comba-pk feedback vectors P
    static constexpr size_t bytes(bool pk = false) { return pk ? OP + sizeof(T) * 64 * PK : OF + sizeof(float) * 64 * 5; }
};

// Store a [rows x cols] product computed in 16-row m-tiles and 64-column passes.
template <typename T, bool AK, bool BK, int ROWS, int COLS>
__device__ __forceinline__ void gemm_to_global(T* g, const T* sA, int lda, const T* sB, int ldb, int K, float sign,
                                               int warp) {
    constexpr int MT = ROWS / 64;  // m-tiles per warp (4 warps)
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
        const int m0 = (warp * MT + mt) * 16;
#pragma unroll
        for (int n0 = 0; n0 < COLS; n0 += 64) {
            float acc[8][4];
            zero(acc);
            warp_gemm<AK, BK, 8>(acc, sA, lda, sB, ldb, m0, n0, K);
            frag_store_global<T, 8>(g, COLS, m0, n0, acc, ROWS, sign);
        }
    }
}

// One CTA per (chunk slot, key head).  The Gram, the UT inverse and W depend on the key head
// only: they are formed once, and W, M and the log-decays G are stored once, at the key head's
// first value-head unit slot * H + hk * vg, where every mma.sync kernel and the dk = 256 scan read
// them.  The vg value heads (units slot * H + hk * vg + j) differ in V and so in U = M Diag(beta) V.
template <typename T, int DK, int DV>
__global__ void __launch_bounds__(128) k_prep(ChunkParams p) {
    using S = PrepSmem<T, DK, DV>;
    constexpr bool kMap = S::kMap;
    const int slot = blockIdx.x, hk = blockIdx.y, Hk = p.H / p.vg;
    const SlotInfo si = p.slot_info[slot];
    if (si.len <= 0) return;
    const int L = si.len;
    const long long t0 = si.start;
    auto vidx = [&](int j) { return (long long)slot * p.H + hk * p.vg + j; };   // value-head units
    const int tid = threadIdx.x, warp = tid >> 5;

    extern __shared__ __align__(128) char smem[];
    T* sK = reinterpret_cast<T*>(smem + S::OK);
    T* sV = reinterpret_cast<T*>(smem + S::OV);
    float* sA = reinterpret_cast<float*>(smem + S::OA);
    float* sM = reinterpret_cast<float*>(smem + S::OM);
    T* sWs = reinterpret_cast<T*>(smem + S::OA);
    T* sUs = reinterpret_cast<T*>(smem + S::OM);
    float* sTmp = reinterpret_cast<float*>(smem + S::OT);
    T* sMw = reinterpret_cast<T*>(smem + S::OMW);
    T* sMu = reinterpret_cast<T*>(smem + S::OMU);
    float* sG = reinterpret_cast<float*>(smem + S::OF);
    float* sGm1 = sG + 64;
    float* sBt = sG + 128;
    float* sBe = sG + 192;
    float* sS = sG + 256;
    // feedback vectors: P for Comba-pk (Gram P K^T, W = M Diag P), else K itself
    T* sF = p.p ? reinterpret_cast<T*>(smem + S::OP) : sK;

    const long long kr0 = t0 * Hk + hk, kld = (long long)Hk * DK;   // key-side rows
    auto load_v = [&](int j) {
        load_tile_async<T>(sV, S::PV, (const T*)p.v + (t0 * p.H + hk * p.vg + j) * DV, (long long)p.H * DV, 64, DV,
                           L, tid, 128);
    };
    // The per-position gates go first, so that their loads do not queue behind the tiles' cp.async
    // traffic; the log-cumsum then runs while the tiles arrive.
    const int lane = tid & 31;
    float a0 = 1.f, a1 = 1.f, bev = 0.f, alv = 1.f, bh = 1.f;
    if (warp == 0) {
        a0 = lane < L ? p.alpha[kr0 + (long long)lane * Hk] : 1.f;
        a1 = lane + 32 < L ? p.alpha[kr0 + (long long)(lane + 32) * Hk] : 1.f;
    }
    if (tid < 64) {
        bev = tid < L ? p.beta[kr0 + (long long)tid * Hk] : 0.f;
        alv = tid < L ? p.alpha[kr0 + (long long)tid * Hk] : 1.f;
        bh = p.b ? p.b[hk] : 1.f;
    }
    load_tile_async<T>(sK, S::PK, (const T*)p.k + kr0 * DK, kld, 64, DK, L, tid, 128);
    if (p.p) load_tile_async<T>(sF, S::PK, (const T*)p.p + kr0 * DK, kld, 64, DK, L, tid, 128);
    load_v(0);
    cp_async_commit();
    if (warp == 0) chunk_log_cumsum_vals(a0, a1, L, sG, sGm1);
    if (tid < 64) {
        sBe[tid] = bev;
        sBt[tid] = bh * bev * feedback_scale(p.iplr, alv);
    }
    cp_async_wait<0>();
    __syncthreads();
    if (tid < 64) sS[tid] = tid < L ? expf(sG[L - 1] - sG[tid]) : 0.f;   // Kbar row scale gamma_C / gamma_r

    // Strictly-lower A = Diag(btilde) (gamma_{r-1}/gamma_i * P K^T) (P = K unless Comba-pk);
    // exp taken only below the diagonal.
    {
        float acc[8][4];
        zero(acc);
        warp_gemm<true, true, 8>(acc, sF, S::PK, sK, S::PK, 16 * warp, 0, DK);
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
    for (int e = tid; e < 64 * 64; e += 128) {
        const int r = e >> 6, c = e & 63;
        const float m = sM[r * 65 + c];
        sMw[r * S::PL + c] = from_f<T>(m * sBt[c] * expf(sGm1[c]));
        sMu[r * S::PL + c] = from_f<T>(m * sBe[c]);
        if (p.Mb) ((T*)p.Mb + vidx(0) * 4096)[e] = from_f<T>(m);
    }
    if (tid < 64) p.Gb[vidx(0) * 64 + tid] = sG[tid];
    __syncthreads();

    // W = Mw P, U = Mu V (stored) and, for the chunk's state map, their Kbar-row-scaled copies.
    // At dk = 256 the scan applies E = U - W H itself and no map is formed.
    const float sa = sS[16 * warp + frag_row(0)], sb = sS[16 * warp + frag_row(2)];
    {
        float acc[DK / 8][4];
        zero(acc);
        warp_gemm<true, false, DK / 8>(acc, sMw, S::PL, sF, S::PK, 16 * warp, 0, 64);
        frag_store_global<T, DK / 8>((T*)p.Wb + vidx(0) * 64 * DK, DK, 16 * warp, 0, acc, 64);
        if constexpr (kMap) {
#pragma unroll
            for (int t = 0; t < DK / 8; ++t) { acc[t][0] *= sa; acc[t][1] *= sa; acc[t][2] *= sb; acc[t][3] *= sb; }
            frag_store<T, DK / 8>(sWs, S::PK, 16 * warp, 0, acc);
        }
    }
    for (int j = 0; j < p.vg; ++j) {
        const long long idx = vidx(j);
        if (j > 0) {   // the previous value head's products have read V
            __syncthreads();
            load_v(j);
            cp_async_commit();
            cp_async_wait<0>();
            __syncthreads();
        }
        {
            float acc[DV / 8][4];
            zero(acc);
            warp_gemm<true, false, DV / 8>(acc, sMu, S::PL, sV, S::PV, 16 * warp, 0, 64);
            frag_store_global<T, DV / 8>((T*)p.Ub + idx * 64 * DV, DV, 16 * warp, 0, acc, 64);
            if constexpr (kMap) {
#pragma unroll
                for (int t = 0; t < DV / 8; ++t) { acc[t][0] *= sa; acc[t][1] *= sa; acc[t][2] *= sb; acc[t][3] *= sb; }
                frag_store<T, DV / 8>(sUs, S::PV, 16 * warp, 0, acc);
            }
        }
        if constexpr (kMap) {
            __syncthreads();
            // Atilde = -K^T Diag(s) W [dk][dk];  B^T = (Diag(s) U)^T K [dv][dk];  Atilde^T = -(Diag(s) W)^T K.
            gemm_to_global<T, false, false, DK, DK>((T*)p.Ab + idx * DK * DK, sK, S::PK, sWs, S::PK, 64, -1.f, warp);
            gemm_to_global<T, false, false, DV, DK>((T*)p.Bb + idx * DV * DK, sUs, S::PV, sK, S::PK, 64, 1.f, warp);
            if (p.ATb)
                gemm_to_global<T, false, false, DK, DK>((T*)p.ATb + idx * DK * DK, sWs, S::PK, sK, S::PK, 64, -1.f,
                                                        warp);
            if (j + 1 < p.vg) __syncthreads();   // the next U's scaled copy replaces this one
        }
    }
}

// ---------------------------------------------------------------- output

template <typename T, int DK, int DV>
struct OutSmem {
    static constexpr int PK = pitch<T>(DK), PV = pitch<T>(DV), PL = pitch<T>(64);
    static constexpr size_t OQ = 0;                                          // Q~
    static constexpr size_t OK = align128(OQ + sizeof(T) * 64 * PK);         // K
    static constexpr size_t OW = align128(OK + sizeof(T) * 64 * PK);         // W
    static constexpr size_t OP = align128(OW + sizeof(T) * 64 * PK);         // P
    static constexpr size_t OG = align128(OP + sizeof(T) * 64 * PL);         // log-decays
    static constexpr size_t OB = align128(OG + sizeof(float) * 64);          // value-head buffers: U (later E), H^T
    static constexpr size_t BU = 0;
    static constexpr size_t BH = align128(sizeof(T) * 64 * PV);
    static constexpr size_t BUF = align128(BH + sizeof(T) * DV * PK);
    // a second buffer when a key head has several value heads (the next one's tiles stream in)
    static constexpr size_t bytes(bool two = false) { return OB + (two ? 2 : 1) * BUF; }
};

// One CTA per (chunk slot, key head).  Q~ and P = Tril(Q~ K^T * Gamma) depend on the key head
// only; each of its value heads j then forms E_j = U_j - W H_j and O_j = Diag(gamma) Q~ H_j + P E_j,
// with the next value head's U and H^T loading meanwhile.
template <typename T, int DK, int DV>
__global__ void __launch_bounds__(128) k_output(ChunkParams p) {
    using S = OutSmem<T, DK, DV>;
    const int slot = blockIdx.x, hk = blockIdx.y, Hk = p.H / p.vg, vg = p.vg;
    const SlotInfo si = p.slot_info[slot];
    if (si.len <= 0) return;
    const int L = si.len;
    const long long t0 = si.start;
    const long long idx0 = (long long)slot * p.H + hk * vg;   // the key head's first value head
    const int tid = threadIdx.x, warp = tid >> 5;

    extern __shared__ __align__(128) char smem[];
    T* sQ = reinterpret_cast<T*>(smem + S::OQ);
    T* sK = reinterpret_cast<T*>(smem + S::OK);
    T* sW = reinterpret_cast<T*>(smem + S::OW);
    T* sP = reinterpret_cast<T*>(smem + S::OP);
    float* sG = reinterpret_cast<float*>(smem + S::OG);
    auto sU = [&](int j) { return reinterpret_cast<T*>(smem + S::OB + (j & 1) * S::BUF + S::BU); };
    auto sH = [&](int j) { return reinterpret_cast<T*>(smem + S::OB + (j & 1) * S::BUF + S::BH); };
    auto load_vh = [&](int j) {   // value head j's U and H^T
        const long long idx = idx0 + j;
        load_tile_async<T>(sU(j), S::PV, (const T*)p.Ub + idx * 64 * DV, DV, 64, DV, 64, tid, 128);
        load_tile_async<T>(sH(j), S::PK, (const T*)p.Hb + idx * DV * DK, DK, DV, DK, DV, tid, 128);
    };

    const long long kr0 = t0 * Hk + hk, kld = (long long)Hk * DK;   // key-side rows
    const float dh = p.d[hk];   // loaded ahead of the tiles' cp.async traffic, as are the log-decays
    const float gv = tid < 64 ? p.Gb[idx0 * 64 + tid] : 0.f;
    load_tile_async<T>(sQ, S::PK, (const T*)p.q + kr0 * DK, kld, 64, DK, L, tid, 128);
    load_tile_async<T>(sK, S::PK, (const T*)p.k + kr0 * DK, kld, 64, DK, L, tid, 128);
    load_tile_async<T>(sW, S::PK, (const T*)p.Wb + idx0 * 64 * DK, DK, 64, DK, 64, tid, 128);
    load_vh(0);
    cp_async_commit();
    if (vg > 1) load_vh(1);
    cp_async_commit();
    if (tid < 64) sG[tid] = gv;
    cp_async_wait<1>();
    __syncthreads();

    for (int e = tid; e < 64 * DK; e += 128) {
        const int r = e / DK, c = e % DK;
        sQ[r * S::PK + c] = from_f<T>(to_f(sQ[r * S::PK + c]) - dh * to_f(sK[r * S::PK + c]));
    }
    __syncthreads();
    // head dim 256 with the backward's workspace: Z = Diag(gamma) Q~ - P W is saved for the reverse
    // scan, which forms the additive term C^T = dO^T Z itself
    const bool zout = DK == 256 && p.Zb != nullptr;
    if (p.o || zout) {
        float sc[8][4];
        zero(sc);
        warp_gemm<true, true, 8>(sc, sQ, S::PK, sK, S::PK, 16 * warp, 0, DK);
#pragma unroll
        for (int t = 0; t < 8; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = 16 * warp + frag_row(i), c = frag_col(t, i);
                const float v = (c <= r && r < L) ? sc[t][i] * expf(sG[r] - sG[c]) : 0.f;
                sP[r * S::PL + c] = from_f<T>(v);
            }
    }
    const float e0 = expf(sG[16 * warp + frag_row(0)]);
    const float e1 = expf(sG[16 * warp + frag_row(2)]);
    if constexpr (DK == 256) {
        if (zout) {
            // Z [64][dk] at the key head's first value head (like W); each warp its own 16 rows, whose
            // P rows it wrote itself.  Rows past a short chunk are zero (Q~ and P rows are).
            __syncwarp();
            T* zg = (T*)p.Zb + idx0 * 64 * DK;
#pragma unroll 1
            for (int n0 = 0; n0 < DK; n0 += 128) {
                float z[16][4];
                zero(z);
                warp_gemm<true, false, 16>(z, sP, S::PL, sW, S::PK, 16 * warp, n0, 64);
#pragma unroll
                for (int t = 0; t < 16; ++t)
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int r = 16 * warp + frag_row(i), c = n0 + frag_col(t, i);
                        z[t][i] = (i < 2 ? e0 : e1) * to_f(sQ[r * S::PK + c]) - z[t][i];
                    }
                frag_store_global<T, 16>(zg, DK, 16 * warp, n0, z, 64);
            }
        }
    }

    for (int j = 0; j < vg; ++j) {
        const long long idx = idx0 + j;
        if (j > 0) {
            cp_async_wait<1>();   // this value head's tiles (only the newest group may be pending)
            __syncthreads();
        }
        T* sE = sU(j);
        T* sHj = sH(j);
        // E = U - W H  (B operand H[c][jj] read from H^T[jj][c]); E replaces U.  Each warp reads
        // and writes only its own 16 rows of U / E.
        {
            float e[DV / 8][4];
            zero(e);
            warp_gemm<true, true, DV / 8>(e, sW, S::PK, sHj, S::PK, 16 * warp, 0, DK);
#pragma unroll
            for (int t = 0; t < DV / 8; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = 16 * warp + frag_row(i), c = frag_col(t, i);
                    e[t][i] = to_f(sE[r * S::PV + c]) - e[t][i];
                }
            if (p.Eb) frag_store_global<T, DV / 8>((T*)p.Eb + idx * 64 * DV, DV, 16 * warp, 0, e, 64);
            frag_store<T, DV / 8>(sE, S::PV, 16 * warp, 0, e);
        }
        __syncthreads();   // E (and, for j = 0, P) complete
        if (p.o) {
            float o[DV / 8][4];
            zero(o);
            warp_gemm<true, true, DV / 8>(o, sQ, S::PK, sHj, S::PK, 16 * warp, 0, DK);
#pragma unroll
            for (int t = 0; t < DV / 8; ++t) {
                o[t][0] *= e0; o[t][1] *= e0;
                o[t][2] *= e1; o[t][3] *= e1;
            }
            warp_gemm<true, false, DV / 8>(o, sP, S::PL, sE, S::PV, 16 * warp, 0, 64);
            frag_store_global<T, DV / 8>((T*)p.o + (t0 * p.H + hk * vg + j) * DV, (long long)p.H * DV, 16 * warp, 0,
                                         o, L);
        }
        if (j + 2 < vg) {
            __syncthreads();   // this buffer is fully read
            load_vh(j + 2);
        }
        cp_async_commit();
    }
}

// -------------------------------------------------------------- launchers

template <typename T, int DK, int DV>
static cudaError_t run_fwd(const ChunkParams& p, bool save, cudaStream_t s, int ev0) {
    const size_t sm_prep = PrepSmem<T, DK, DV>::bytes(p.p != nullptr);
    const size_t sm_out = OutSmem<T, DK, DV>::bytes(p.vg > 1);
    cudaError_t e;
    if (!(DK == 256 && sizeof(T) == 2) &&   // head dim 256 (bf16) runs the tcgen05 prep kernel
        (e = cudaFuncSetAttribute(k_prep<T, DK, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_prep)))
        return e;
    if (!(DK == 256 && sizeof(T) == 2) &&   // head dim 256 (bf16) runs the tcgen05 output kernel
        (e = cudaFuncSetAttribute(k_output<T, DK, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_out)))
        return e;
    const bool tcp = use_tc_path(sizeof(T) == 2, DK, DV);
    ChunkParams q = p;
    if (!save) { q.Mb = nullptr; q.ATb = nullptr; q.Eb = nullptr; q.Zb = nullptr; }
    if (tcp) q.ATb = nullptr;   // the tcgen05 reverse scan reads Atilde directly
    mark(q, ev0, s);
    if (tcp) {
        if ((e = launch_prep_tc(q, s))) return e;
    } else if (DK == 256 && sizeof(T) == 2) {
        if ((e = launch_prep_wide_tc(q, s))) return e;
    } else if (q.slots > 0) {
        k_prep<T, DK, DV><<<dim3(q.slots, q.H / q.vg), 128, sm_prep, s>>>(q);   // one CTA per key head
    }
    if ((e = cudaGetLastError())) return e;
    mark(q, ev0 + 1, s);
    ScanArgs a;
    a.H = q.H; a.vg = q.vg; a.N = q.N; a.T = q.T; a.slots = q.slots; a.Ttot = q.Ttot; a.cu = q.cu;
    a.seq_first = q.seq_first;
    a.Gb = q.Gb; a.init = q.h0; a.fin = q.hT; a.Sout = q.Hb; a.X = q.Ab; a.Y = q.Bb; a.reverse = 0; a.x_mn = 0;
    a.W = q.Wb; a.K = q.k;
    if (DK == 256) a.Y = q.Ub;   // the wide scan forms E = U - W H itself
    if (tcp) {                   // B^T = U_s^T K formed in the scan
        a.ym = 2;
        a.F = q.Usb;
        a.tok = q.k;
        a.Y = nullptr;
    }
    a.err = q.err;
    a.wait_ns = q.wait_ns;
    if ((e = launch_scan(a, sizeof(T) == 2, DK, DV, (long long)q.slots * q.H, s))) return e;
    mark(q, ev0 + 2, s);
    if (q.o || q.Eb) {
        if (tcp) {
            if ((e = launch_output_tc(q, s))) return e;
        } else if (DK == 256 && sizeof(T) == 2) {
            if ((e = launch_output_wide_tc(q, s))) return e;
        } else if (q.slots > 0) {
            k_output<T, DK, DV><<<dim3(q.slots, q.H / q.vg), 128, sm_out, s>>>(q);   // one CTA per key head
        }
    }
    if ((e = cudaGetLastError())) return e;
    mark(q, ev0 + 3, s);
    return cudaSuccess;
}

cudaError_t launch_chunk_map(const ChunkParams& p, cudaStream_t s) {
    k_chunk_map<<<1, 1024, 0, s>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_fwd(const ChunkParams& p, bool is_bf16, bool save, cudaStream_t s, int ev0) {
#define COMBA_FWD(T, DK, DV) \
    if (p.dk == DK && p.dv == DV) return run_fwd<T, DK, DV>(p, save, s, ev0);
    if (is_bf16) {
        COMBA_FWD(bf16, 128, 128) COMBA_FWD(bf16, 128, 64) COMBA_FWD(bf16, 64, 128) COMBA_FWD(bf16, 64, 64)
        COMBA_FWD(bf16, 256, 64)
    } else {
        COMBA_FWD(float, 128, 128) COMBA_FWD(float, 128, 64) COMBA_FWD(float, 64, 128) COMBA_FWD(float, 64, 64)
    }
#undef COMBA_FWD
    return cudaErrorInvalidValue;
}

size_t fwd_smem_bytes(int kernel, bool is_bf16, int dk, int dv, bool pk, bool groups) {
    if (kernel == 1) return scan_smem_bytes(is_bf16, dk, dv);
    if (use_tc_path(is_bf16, dk, dv)) return tc_smem_bytes(kernel == 0 ? 0 : 1);
    if (is_bf16 && dk == 256) return kernel == 0 ? prep_wide_tc_smem_bytes() : output_wide_tc_smem_bytes();
#define COMBA_SM(T, DK, DV) \
    if (dk == DK && dv == DV) return kernel == 0 ? PrepSmem<T, DK, DV>::bytes(pk) : OutSmem<T, DK, DV>::bytes(groups);
    if (is_bf16) {
        COMBA_SM(bf16, 128, 128) COMBA_SM(bf16, 128, 64) COMBA_SM(bf16, 64, 128) COMBA_SM(bf16, 64, 64)
        COMBA_SM(bf16, 256, 64)
    } else {
        COMBA_SM(float, 128, 128) COMBA_SM(float, 128, 64) COMBA_SM(float, 64, 128) COMBA_SM(float, 64, 64)
    }
#undef COMBA_SM
    return 0;
}

}  // namespace comba
