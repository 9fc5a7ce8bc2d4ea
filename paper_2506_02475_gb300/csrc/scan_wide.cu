// Sequential inter-chunk scan for head dim dk = 256.
//
// At dk = 256 a chunk's folded map Atilde = -Kbar^T W is 256 x 256 (128 KB in
// bf16): writing and reading it per (chunk, head) would cost twice W and K
// together.  So this scan applies section 3.3's chunk equations directly, two
// products per chunk:
//     forward:   E = U - W H,            H' = gamma_C H + Kbar^T E
//     backward:  R = Kbar dH',           dH = gamma_C dH' + C - W^T R
// with Kbar = Diag(s) K, s_r = gamma_C / gamma_r for positions r < L (zero past
// the chunk).  Both run transposed over one value head's 64 state rows (dv):
//     Pt = (Z - S^T F1^T) Diag(s),       S^T <- gamma_C S^T + Pt F2 + Y
// forward:  F1 = W, F2 = K, Z = U^T, Y = 0 (Pt = E^T Diag(s));
// backward: F1 = K, F2 = W, Z = 0,   Y = C^T (Pt = -R^T).
// W rows past the chunk are zero (prep zero-fills its key rows), so partial
// chunks need no other masking.
//
// One CTA per (sequence, value head), 256 threads: warp (wr, wc) owns state rows
// 16 wr .. 16 wr + 15 and columns 128 wc .. 128 wc + 127 as m16n8 fragments (64
// fp32 values per thread, resident across the whole sequence).  Tile products
// are mma.sync m16n8k16 (bf16 operands, fp32 accumulation).  F1 is single-buffered
// and refilled for the next chunk as soon as the first product has read it; F2,
// Z / Y and the chunk's log-decays are double-buffered one chunk ahead.  Each chunk
// stores the state it starts from (H_n^T, or dH_{n+1}^T in the backward) in bf16.
#include "params.cuh"

namespace comba {

namespace {

constexpr int kWideDK = 256, kWideDV = 64;

struct WideSmem {
    static constexpr int PK = pitch<bf16>(kWideDK), PL = pitch<bf16>(64);
    static constexpr size_t S_BYTES = sizeof(bf16) * 64 * PK;    // a 64 x dk tile
    static constexpr size_t E_BYTES = sizeof(bf16) * 64 * PL;    // a 64 x 64 tile
    static constexpr size_t OS = 0;                               // S^T (bf16): A operand and stored chunk state
    static constexpr size_t OE = OS + S_BYTES;                    // Pt
    static constexpr size_t OF1 = OE + E_BYTES;                   // F1 (one buffer)
    static constexpr size_t OST = OF1 + S_BYTES;                  // two stages: F2, Z or Y, log-decays
    __host__ __device__ static constexpr size_t z_bytes(bool reverse) { return reverse ? S_BYTES : E_BYTES; }
    __host__ __device__ static constexpr size_t stage_bytes(bool reverse) {
        return S_BYTES + z_bytes(reverse) + sizeof(float) * 64;
    }
    __host__ __device__ static constexpr size_t bytes(bool reverse) { return OST + 2 * stage_bytes(reverse); }
};

__device__ __forceinline__ void wide_seq_range(const ScanArgs& a, int n, long long& start, long long& len) {
    long long s = a.cu ? a.cu[n] : (long long)n * a.T;
    long long e = a.cu ? a.cu[n + 1] : (long long)(n + 1) * a.T;
    s = s < 0 ? 0 : (s > a.Ttot ? a.Ttot : s);
    e = e < s ? s : (e > a.Ttot ? a.Ttot : e);
    start = s;
    len = e - s;
}

__global__ void __launch_bounds__(256, 1) k_scan_wide(ScanArgs a) {
    using S = WideSmem;
    constexpr int DK = kWideDK, DV = kWideDV, PK = S::PK, PL = S::PL;
    constexpr int NT = DK / 16;   // state n-tiles per warp (128 columns)
    extern __shared__ __align__(128) char smem[];
    const int tid = threadIdx.x, warp = tid >> 5;
    const int wr = warp & 3, wc = warp >> 2;
    const int m0 = 16 * wr, n0 = 128 * wc;
    const int n = blockIdx.x, h = blockIdx.y;
    const bool rev = a.reverse != 0;
    const int Hk = a.H / a.vg, hk = h / a.vg;

    bf16* sS = reinterpret_cast<bf16*>(smem + S::OS);
    bf16* sE = reinterpret_cast<bf16*>(smem + S::OE);
    bf16* sF1 = reinterpret_cast<bf16*>(smem + S::OF1);
    const size_t stb = S::stage_bytes(rev);
    auto sF2 = [&](int it) { return reinterpret_cast<bf16*>(smem + S::OST + (it & 1) * stb); };
    auto sZ = [&](int it) { return reinterpret_cast<bf16*>(smem + S::OST + (it & 1) * stb + S::S_BYTES); };
    auto sG = [&](int it) {
        return reinterpret_cast<float*>(smem + S::OST + (it & 1) * stb + S::S_BYTES + S::z_bytes(rev));
    };

    long long start, len;
    wide_seq_range(a, n, start, len);
    const int s0 = a.seq_first[n];
    int nch = (int)((len + kChunk - 1) / kChunk);
    if (s0 + nch > a.slots) nch = a.slots - s0 > 0 ? a.slots - s0 : 0;
    auto chunk_of = [&](int it) { return rev ? nch - 1 - it : it; };
    auto unit_of = [&](int it) { return (long long)(s0 + chunk_of(it)) * a.H + h; };
    auto len_of = [&](int it) {
        const long long rest = len - (long long)chunk_of(it) * kChunk;
        return (int)(rest < kChunk ? rest : kChunk);
    };

    const bf16* Wg = static_cast<const bf16*>(a.W);
    const bf16* Kg = static_cast<const bf16*>(a.K);
    const bf16* Yg = static_cast<const bf16*>(a.Y);
    // the chunk's W (all 64 rows stored) or its raw key rows (zero-filled past the chunk)
    auto load_w = [&](bf16* dst, int it) {
        load_tile_async<bf16>(dst, PK, Wg + unit_of(it) * 64 * DK, DK, 64, DK, 64, tid, 256);
    };
    auto load_k = [&](bf16* dst, int it) {
        const long long t0 = start + (long long)chunk_of(it) * kChunk;
        load_tile_async<bf16>(dst, PK, Kg + (t0 * Hk + hk) * DK, (long long)Hk * DK, 64, DK, len_of(it), tid, 256);
    };
    auto load_f1 = [&](int it) { if (rev) load_k(sF1, it); else load_w(sF1, it); };
    auto load_stage = [&](int it) {
        if (rev) {
            load_w(sF2(it), it);
            load_tile_async<bf16>(sZ(it), PK, Yg + unit_of(it) * DV * DK, DK, DV, DK, DV, tid, 256);   // C^T
        } else {
            load_k(sF2(it), it);
            load_tile_async<bf16>(sZ(it), PL, Yg + unit_of(it) * 64 * DV, DV, 64, DV, 64, tid, 256);   // U
        }
        if (tid < 16) cp_async16(sG(it) + 4 * tid, a.Gb + unit_of(it) * 64 + 4 * tid, true);
    };

    // state fragments: rows m0 + g (+ 8), columns n0 + 8 t + 2 q (+ 1)
    float st[NT][4];
    const long long soff = [&] {
        const int j = h - hk * a.vg;
        return ((long long)n * Hk + hk) * DK * ((long long)a.vg * DV) + (long long)j * DV;
    }();
    const long long sld = (long long)a.vg * DV;   // stride between state rows (dk index) of init / fin
#pragma unroll
    for (int t = 0; t < NT; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int j = m0 + frag_row(i), c = n0 + frag_col(t, i);
            st[t][i] = a.init ? a.init[soff + (long long)c * sld + j] : 0.f;
        }

    if (nch > 0) {
        load_f1(0);
        load_stage(0);
    }
    cp_async_commit();
    if (nch > 1) load_stage(1);
    cp_async_commit();

    for (int it = 0; it < nch; ++it) {
        const int L = len_of(it);
        // the state this chunk starts from, as the first product's A operand
        frag_store<bf16, NT>(sS, PK, m0, n0, st);
        cp_async_wait<1>();   // F1 of this chunk and its stage have landed (only the newest group may be pending)
        __syncthreads();

        // S^T F1^T  [64 x 64]: rows m0.., columns 32 wc..
        float pr[4][4];
        zero(pr);
        warp_gemm<true, true, 4>(pr, sS, PK, sF1, PK, m0, 32 * wc, DK);
        // the chunk's starting state, bf16 [dv][dk]
        store_tile<bf16>(static_cast<bf16*>(a.Sout) + unit_of(it) * DV * DK, DK, sS, PK, DV, DK, DV, tid, 256);
        __syncthreads();   // F1 and S^T fully read
        if (it + 1 < nch) load_f1(it + 1);
        cp_async_commit();

        const float* g = sG(it);
        const float gL = g[L - 1];
        {
            const bf16* z = sZ(it);
#pragma unroll
            for (int t = 0; t < 4; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int j = m0 + frag_row(i), r = 32 * wc + frag_col(t, i);
                    const float sr = r < L ? __expf(gL - g[r]) : 0.f;
                    const float zv = rev ? 0.f : to_f(z[r * PL + j]);   // U^T
                    pr[t][i] = sr * (zv - pr[t][i]);
                }
            frag_store<bf16, 4>(sE, PL, m0, 32 * wc, pr);
        }
        __syncthreads();

        // S^T <- gamma_C S^T + Y + Pt F2
        const float gam = __expf(gL);
        if (rev) {
            const bf16* y = sZ(it);
#pragma unroll
            for (int t = 0; t < NT; ++t)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const int j = m0 + frag_row(2 * hh), c = n0 + frag_col(t, 0);
                    const float2 yv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(y + j * PK + c));
                    st[t][2 * hh] = fmaf(gam, st[t][2 * hh], yv.x);
                    st[t][2 * hh + 1] = fmaf(gam, st[t][2 * hh + 1], yv.y);
                }
        } else {
#pragma unroll
            for (int t = 0; t < NT; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) st[t][i] *= gam;
        }
        warp_gemm<true, false, NT>(st, sE, PL, sF2(it), PK, m0, n0, 64);
        __syncthreads();   // this stage and Pt fully read
        if (it + 2 < nch) load_stage(it + 2);
        cp_async_commit();
    }
    cp_async_wait<0>();   // nothing still writes shared memory at exit

    if (a.fin) {
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int j = m0 + frag_row(i), c = n0 + frag_col(t, i);
                a.fin[soff + (long long)c * sld + j] = st[t][i];
            }
    }
}

}  // namespace

cudaError_t launch_scan_wide(const ScanArgs& a, cudaStream_t s) {
    const size_t sm = WideSmem::bytes(a.reverse != 0);
    cudaError_t e = cudaFuncSetAttribute(k_scan_wide, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    if (a.N > 0 && a.H > 0) k_scan_wide<<<dim3(a.N, a.H), 256, sm, s>>>(a);
    return cudaGetLastError();
}

size_t scan_wide_smem_bytes() { return WideSmem::bytes(true); }

}  // namespace comba
