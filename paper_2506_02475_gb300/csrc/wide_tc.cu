// Prep and output kernels of the bf16 head-dim-256 path on the 5th-generation tensor cores.
//
// k_prep_wide_tc, per (chunk slot, key head) unit (section 3.2, Eq. "prepare WY_M"; the key
// head's vg value heads are 64 wide):
//
//   A = strict_lower(Diag(btilde) (Gamma- * F K^T)),  M = (I + A)^{-1},
//   W = M Diag(btilde gamma_{r-1}) F,   per value head j:  U_j = M Diag(beta) V_j
//
// (F = K, or the feedback vectors P of Comba-pk), storing W, M and the log-decays once per key
// head and U_j per value head.  At head dim 256 no chunk map is formed: the scan applies
// E = U - W H per chunk itself.
//
// k_output_wide_tc, per (chunk slot, key head) unit (section 3.2's output equation, and the
// chunk factors the backward reuses):
//
//   Q~ = Q - d K,   S = Q~ K^T,   P = Tril(S * Gamma),   Qhat = Diag(gamma) Q~
//   Z = Qhat - P W                      (saved once per key head for the reverse scan)
//   per value head j:  E_j = U_j - W H_j,   O_j = Qhat H_j + P E_j
//
// with H_j the chunk state of value head j (H_j^T [64][256] in the workspace), W [64][256],
// U_j [64][64].  In both kernels every product is a tcgen05.mma with M = 64 (the chunk rows) issued by one
// thread; K = 256 contractions take sixteen 16-deep steps over the four 64-column blocks of the
// 128-byte-swizzled tiles.  The accumulators are read with tcgen05.ld.16x256b into the m16n8
// fragment layout (warp w: rows 16 (w % 4) .. + 15, column half w / 4), and the epilogues move
// fragment tiles through stmatrix / ldmatrix.  In the output kernel tiles arrive by TMA (Q, K
// and W in one group, each value head's H_j^T and U_j double-buffered); Z, E_j and full chunks'
// O_j leave by bulk tensor stores.  The value heads run one after another: value head j + 1's two
// products are issued as soon as P E_j is, into the other of two TMEM column sets.  Prep takes
// the UT inverse of the tcgen05 d = 128 prep (fp32 diagonal blocks, tf32 tile products for the
// rest).  Both zero the rows of their token tiles past a short chunk (the next sequence's tokens,
// which need not be finite) before any product reads them.
#include <cuda.h>

#include "tc_frag.cuh"

namespace comba {

bool make_bf16_token_map(CUtensorMap* m, const void* base, long long tokens, int heads, int cols);
bool make_bf16_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows);

namespace tc {
namespace {

constexpr int kWK = 256;   // key width of a unit
constexpr int kWV = 64;    // value width of one value head

// ------------------------------------------------------------------ prep

struct PrepWideSmem {
    static constexpr uint32_t OF = 0;                   // F = K or P [64][256]                       32 KB
    static constexpr uint32_t OK = OF + 32768;          // K [64][256] (Comba-pk; else F is K)        32 KB
    static constexpr uint32_t OV = OK + 32768;          // V_j [64][64], two buffers                  16 KB
    static constexpr uint32_t OMW = OV + 16384;         // Mw [64][64]                                 8 KB
    static constexpr uint32_t OMU = OMW + 8192;         // Mu [64][64]                                 8 KB
    static constexpr uint32_t OU = OMU + 8192;          // U_j staging [64][64], two buffers          16 KB
    static constexpr uint32_t OR = OU + 16384;          // A^T, M (fp32), inverse scratch; then the W staging
    static constexpr uint32_t R_BYTES = (64 * kAtPitch + 64 * kMPitch + 1024) * 4;
    static constexpr uint32_t OG = OR + ((R_BYTES + 1023) & ~1023u);   // fp32 per-row vectors
    static constexpr size_t bytes() { return 1024 + OG + 64 * 5 * 4; }
};
static_assert(PrepWideSmem::R_BYTES >= 32768, "the W staging fits over the inverse's fp32 region");

// Tensor maps, 128-byte swizzled: k and p (key heads, {64 columns, 1 head, 64 tokens} boxes), v
// (value heads 64 wide, the same boxes); W ([pairs * 64][256]) and U ([pairs * 64][64]) stores.
struct PrepWideMaps {
    CUtensorMap k, p, v, w, u;
};

__global__ void __launch_bounds__(256, 1) k_prep_wide_tc(ChunkParams p, const __grid_constant__ PrepWideMaps mp) {
    using S = PrepWideSmem;
    constexpr int kTma = 32;
    const int slot = blockIdx.x, hk = blockIdx.y, vg = p.vg, Hk = p.H / p.vg;
    const SlotInfo si = p.slot_info[slot];
    if (si.len <= 0) return;
    const int L = si.len;
    const int t0 = si.start;
    const long long idx0 = (long long)slot * p.H + (long long)hk * vg;   // the key head's first value head
    const bool pk = p.p != nullptr;

    extern __shared__ uint8_t smem_raw[];
    // ldF: F (and K); ldV[b]: value-head buffer b; bar: the Gram, then W = Mw F; barU: U_j
    __shared__ uint64_t ldF, ldV[2], bar, barU;
    __shared__ uint32_t tbase;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wr = warp & 3, wc = warp >> 2, m0 = 16 * wr;
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sF = sm + S::OF;
    uint8_t* sKk = pk ? sm + S::OK : sF;
    uint8_t* sMw = sm + S::OMW;
    uint8_t* sMu = sm + S::OMU;
    uint8_t* stW = sm + S::OR;                          // W staging [64][256], once A^T and M are dead
    auto sV = [&](int j) { return sm + S::OV + (j & 1) * 8192; };
    auto stU = [&](int j) { return sm + S::OU + (j & 1) * 8192; };
    float* sAt = reinterpret_cast<float*>(sm + S::OR);   // A transposed
    float* sM = sAt + 64 * kAtPitch;
    float* sT = sM + 64 * kMPitch;
    float* sG = reinterpret_cast<float*>(sm + S::OG);
    float* sGm1 = sG + 64;
    float* sBt = sG + 128;
    float* sBe = sG + 192;
    float* sWs = sG + 256;   // btilde_c gamma_{c-1}: the column scale of Mw
    const uint32_t uF = smem_u32(sF), uK = smem_u32(sKk), uMw = smem_u32(sMw), uMu = smem_u32(sMu);

    if (tid == 0) {
        mbar_init(smem_u32(&ldF), 1);
        mbar_init(smem_u32(&ldV[0]), 1);
        mbar_init(smem_u32(&ldV[1]), 1);
        mbar_init(smem_u32(&bar), 1);
        mbar_init(smem_u32(&barU), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tbase), 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tbase;
    const uint32_t tq = tmem + ((uint32_t)(32 * wr) << 16);

    int nv = 0;   // thread kTma: value-head loads issued
    auto issue_v = [&](int j) {
        const uint32_t mb = smem_u32(&ldV[j & 1]);
        mbar_expect_tx(mb, 8192u);
        tma_load_3d(smem_u32(sV(j)), &mp.v, 0, hk * vg + j, t0, mb);
        ++nv;
    };
    if (tid == kTma) {
        const uint32_t mb = smem_u32(&ldF);
        mbar_expect_tx(mb, pk ? 65536u : 32768u);
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            tma_load_3d(uF + b * 8192, pk ? &mp.p : &mp.k, 64 * b, hk, t0, mb);
            if (pk) tma_load_3d(uK + b * 8192, &mp.k, 64 * b, hk, t0, mb);
        }
        issue_v(0);
        if (vg > 1) issue_v(1);
    }

    // the chunk's gates: log-decays (warp 0), beta and btilde (threads < 64)
    {
        const float* ag = p.alpha + (long long)t0 * Hk + hk;
        if (warp == 0) {
            const float a0 = lane < L ? ag[(long long)lane * Hk] : 1.f;
            const float a1 = lane + 32 < L ? ag[(long long)(lane + 32) * Hk] : 1.f;
            chunk_log_cumsum_vals(a0, a1, L, sG, sGm1);
        }
        if (tid < 64) {
            const float be = tid < L ? p.beta[((long long)t0 + tid) * Hk + hk] : 0.f;
            const float al = tid < L ? ag[(long long)tid * Hk] : 1.f;
            const float bh = p.b ? p.b[hk] : 1.f;
            sBe[tid] = be;
            sBt[tid] = bh * be * feedback_scale(p.iplr, al);
        }
    }
    __syncthreads();   // sG, sGm1, sBt
    if (tid < 64) {
        sWs[tid] = sBt[tid] * expf(sGm1[tid]);
        p.Gb[idx0 * 64 + tid] = sG[tid];
    }

    uint32_t phB = 0, phU = 0;
    auto wait_warp = [&](uint64_t& b, uint32_t& ph) {
        const bool okw = mbar_wait_polls(smem_u32(&b), ph, p.wait_ns);
        ph ^= 1;
        const bool all = __all_sync(0xffffffffu, okw);
        tc_fence_after();
        return all;
    };

    // the Gram F K^T.  Rows past a short chunk hold the next sequence's tokens (possibly not
    // finite, and 0 * inf is not 0): zeroed first.
    bool ok = true;
    if (L < kChunk) {
        ok = mbar_wait_polls(smem_u32(&ldF), 0, p.wait_ns);
        for (int e = tid; ok && e < (64 - L) * 32; e += 256) {
            const int r = L + (e >> 5), c = 8 * (e & 31);
            *reinterpret_cast<uint4*>(sF + sw128_offset(r, c, 64)) = make_uint4(0, 0, 0, 0);
            if (pk) *reinterpret_cast<uint4*>(sKk + sw128_offset(r, c, 64)) = make_uint4(0, 0, 0, 0);
        }
        ok = publish_ok(ok);
    }
    if (tid == 0) {
        if (ok && L == kChunk) ok = mbar_wait_polls(smem_u32(&ldF), 0, p.wait_ns);
        if (ok) tc_gemm_m64<false, false>(tmem, uF, 64, uK, 64, 64, kWK, false);
        tc_commit(smem_u32(&bar));
    }
    if (warp == 0) ok = __all_sync(0xffffffffu, ok);
    ok = wait_warp(bar, phB) && ok;
    if (ok) {
        // strictly lower A = Diag(btilde) (gamma_{r-1} / gamma_c * F K^T), transposed into fp32; the exp
        // is selected away above the diagonal and past the chunk's end
        float g[4][4];
        tmem_frag<4>(tq + 32 * wc, g);
#pragma unroll
        for (int t = 0; t < 4; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = m0 + frag_row(i), c = 32 * wc + frag_col(t, i);
                sAt[c * kAtPitch + r] = (c < r && r < L) ? sBt[r] * __expf(sGm1[r] - sG[c]) * g[t][i] : 0.f;
            }
    }
    ok = !__syncthreads_or(!ok);   // the inverse's barriers below need a block-uniform flag
    if (ok) {
        unit_lower_inverse64_h16(sAt, sM, sT, tid);
        __syncthreads();
        // Mw = M Diag(btilde gamma_{c-1}), Mu = M Diag(beta) as K-major tiles; M saved for the backward
        bf16* Mg = p.Mb ? (bf16*)p.Mb + idx0 * 4096 : nullptr;
        for (int e = tid; e < 64 * 8; e += 256) {
            const int r = e >> 3, ch = e & 7;
            float mw[8], mu[8], mm[8];
            *reinterpret_cast<float4*>(mm) = *reinterpret_cast<const float4*>(sM + r * kMPitch + 8 * ch);
            *reinterpret_cast<float4*>(mm + 4) = *reinterpret_cast<const float4*>(sM + r * kMPitch + 8 * ch + 4);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const int c = 8 * ch + q;
                mw[q] = mm[q] * sWs[c];
                mu[q] = mm[q] * sBe[c];
            }
            *reinterpret_cast<uint4*>(sMw + sw128_offset(r, 8 * ch, 64)) = pack8(mw);
            *reinterpret_cast<uint4*>(sMu + sw128_offset(r, 8 * ch, 64)) = pack8(mu);
            if (Mg) *reinterpret_cast<uint4*>(Mg + r * 64 + 8 * ch) = pack8(mm);
        }
    }
    ok = publish_ok(ok);

    // W = Mw F on bar, U_0 = Mu V_0 on barU
    auto issue_u = [&](int j) {   // thread 0
        const bool okv = mbar_wait_polls(smem_u32(&ldV[j & 1]), (j >> 1) & 1, p.wait_ns);
        if (okv && L < kChunk) zero_tile_rows(sV(j), L, 1);   // (the next sequence's tokens)
        if (okv) tc_gemm_m64<false, true>(tmem + 64 + 64 * (j & 1), uMu, 64, smem_u32(sV(j)), 64, kWV, 64, false);
        tc_commit(smem_u32(&barU));
        return okv;
    };
    bool okv0 = true;
    if (tid == 0) {
        if (ok) tc_gemm_m64<false, true>(tmem + 256, uMw, 64, uF, 64, kWK, 64, false);   // W = Mw F
        tc_commit(smem_u32(&bar));
        if (ok) okv0 = issue_u(0);
        else tc_commit(smem_u32(&barU));
    }
    ok = wait_warp(bar, phB) && ok;
    if (ok) {
        // W into its staging (over the dead A^T / M region): this warp's rows, columns 128 wc .. + 127
#pragma unroll 1
        for (int pass = 0; pass < 4; ++pass) {
            const int n0 = 128 * wc + 32 * pass;
            float w[4][4];
            tmem_frag<4>(tq + 256 + n0, w);
            frag_store_sw<4>(stW, 64, m0, n0, w);
        }
    }
    if (warp == 0) ok = __all_sync(0xffffffffu, ok && okv0);
    for (int j = 0; j < vg; ++j) {
        ok = wait_warp(barU, phU) && ok;   // U_j
        if (ok && tid == kTma && j + 2 < vg) issue_v(j + 2);   // V_j's readers are done
        if (ok) {
            float u[4][4];
            tmem_frag<4>(tq + 64 + 64 * (j & 1) + 32 * wc, u);
            frag_store_sw<4>(stU(j), 64, m0, 32 * wc, u);
        }
        if (tid == kTma) bulk_wait_all_reads();   // the store of U_{j-2} has read its staging
        bool okv = true;
        if (tid == 0 && j + 1 < vg) {
            if (ok) okv = issue_u(j + 1);
            else tc_commit(smem_u32(&barU));
        }
        if (tid == 0) ok = ok && okv;
        ok = publish_ok(ok);
        if (ok && tid == kTma) {
            if (j == 0)
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_store_2d(&mp.w, 64 * b, (int)(idx0 * 64), smem_u32(stW) + b * 8192);
            tma_store_2d(&mp.u, 0, (int)((idx0 + j) * 64), smem_u32(stU(j)));
        }
        if (tid == kTma) bulk_commit();
        if (!ok) break;
    }

    if (!ok) {
        if (tid == kTma) {
            mbar_drain(smem_u32(&ldF), 0);
            for (int j = nv > 2 ? nv - 2 : 0; j < nv; ++j) mbar_drain(smem_u32(&ldV[j & 1]), (j >> 1) & 1);
        }
        if (tid == 0) {
            flag_error(p);
            tc_commit(smem_u32(&bar));
            mbar_drain(smem_u32(&bar), phB);
        }
    }
    if (tid == kTma) bulk_wait_all_done();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

// ---------------------------------------------------------------- output

struct OutWideSmem {
    static constexpr uint32_t OQK = 0;                  // [128][256]: rows 0-63 Q -> Q~ -> Qhat, rows 64-127 K,
                                                        // then the Z staging                          64 KB
    static constexpr uint32_t OW = OQK + 65536;         // W [64][256]                                32 KB
    static constexpr uint32_t OP = OW + 32768;          // P [64][64]                                  8 KB
    static constexpr uint32_t OE = OP + 8192;           // E_j [64][64], two buffers                  16 KB
    static constexpr uint32_t OO = OE + 16384;          // O_j staging [64][64], two buffers          16 KB
    static constexpr uint32_t OV = OO + 16384;          // value-head buffers: H_j^T [64][256], U_j [64][64]
    static constexpr uint32_t VBUF = 32768 + 8192;      //                                        2 x 40 KB
    static constexpr uint32_t OG = OV + 2 * VBUF;       // fp32 log-decays [64]
    static constexpr size_t bytes() { return 1024 + OG + 64 * 4; }
};

// Tensor maps, 128-byte swizzled: q, k (key heads) and o (value heads) as token tensors with
// {64 columns, 1 head, 64 tokens} boxes; W, H^T, Z ([pairs * 64][256]) and U, E ([pairs * 64][64])
// as 2D views with {64 columns, 64 rows} boxes.
struct OutWideMaps {
    CUtensorMap q, k, o, w, h, u, e, z;
};

// TMEM columns: S, then per value-head parity b the E_j and O_j accumulators, and P W.
constexpr uint32_t kColS = 0, kColPW = 256;
__device__ __forceinline__ uint32_t col_e(int j) { return (j & 1) ? 320u : 64u; }
__device__ __forceinline__ uint32_t col_o(int j) { return (j & 1) ? 384u : 128u; }

__global__ void __launch_bounds__(256, 1) k_output_wide_tc(ChunkParams p, const __grid_constant__ OutWideMaps mp) {
    using S = OutWideSmem;
    constexpr int kTma = 32;   // issues the TMA loads and the bulk stores
    const int slot = blockIdx.x, hk = blockIdx.y, vg = p.vg;
    const SlotInfo si = p.slot_info[slot];
    if (si.len <= 0) return;
    const int L = si.len;
    const int t0 = si.start;
    const long long idx0 = (long long)slot * p.H + (long long)hk * vg;   // the key head's first value head
    const bool zout = p.Zb != nullptr, want_o = p.o != nullptr, eout = p.Eb != nullptr;

    extern __shared__ uint8_t smem_raw[];
    // ldA: Q, K, W; ldV[b]: value-head buffer b; barV: a value head's W H_j, Qhat H_j (and, for the
    // first, S and then P W on their own phases of bar); barO: O_j += P E_j
    __shared__ uint64_t ldA, ldV[2], bar, barV, barO;
    __shared__ uint32_t tbase;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int wr = warp & 3, wc = warp >> 2, m0 = 16 * wr;
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sQK = sm + S::OQK;
    uint8_t* sW = sm + S::OW;
    uint8_t* sP = sm + S::OP;
    float* sG = reinterpret_cast<float*>(sm + S::OG);
    auto sE = [&](int j) { return sm + S::OE + (j & 1) * 8192; };
    auto sO = [&](int j) { return sm + S::OO + (j & 1) * 8192; };
    auto sHt = [&](int j) { return sm + S::OV + (j & 1) * S::VBUF; };
    auto sU = [&](int j) { return sm + S::OV + (j & 1) * S::VBUF + 32768; };
    const uint32_t uQK = smem_u32(sQK), uK = uQK + 64 * 128, uW = smem_u32(sW), uP = smem_u32(sP);

    if (tid == 0) {
        mbar_init(smem_u32(&ldA), 1);
        mbar_init(smem_u32(&ldV[0]), 1);
        mbar_init(smem_u32(&ldV[1]), 1);
        mbar_init(smem_u32(&bar), 1);
        mbar_init(smem_u32(&barV), 1);
        mbar_init(smem_u32(&barO), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tbase), 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tbase;
    const uint32_t tq = tmem + ((uint32_t)(32 * wr) << 16);   // this warp's TMEM lane quadrant

    int nv = 0;   // thread kTma: value-head loads issued
    auto issue_v = [&](int j) {
        const uint32_t mb = smem_u32(&ldV[j & 1]);
        const int y = (int)((idx0 + j) * 64);
        mbar_expect_tx(mb, 32768u + 8192u);
#pragma unroll
        for (int b = 0; b < 4; ++b) tma_load_2d(smem_u32(sHt(j)) + b * 8192, &mp.h, 64 * b, y, mb);
        tma_load_2d(smem_u32(sU(j)), &mp.u, 0, y, mb);
        ++nv;
    };
    if (tid == kTma) {
        const uint32_t mb = smem_u32(&ldA);
        mbar_expect_tx(mb, 3u * 32768u);
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            tma_load_3d(uQK + b * 16384, &mp.q, 64 * b, hk, t0, mb);
            tma_load_3d(uK + b * 16384, &mp.k, 64 * b, hk, t0, mb);
            tma_load_2d(uW + b * 8192, &mp.w, 64 * b, (int)(idx0 * 64), mb);
        }
        issue_v(0);
        if (vg > 1) issue_v(1);
    }
    if (tid < 64) sG[tid] = p.Gb[idx0 * 64 + tid];
    const float dh = p.d[hk];

    uint32_t phB = 0, phV = 0, phO = 0;   // phases of bar, barV, barO
    auto wait_warp = [&](uint64_t& b, uint32_t& ph) {
        const bool okw = mbar_wait_polls(smem_u32(&b), ph, p.wait_ns);
        ph ^= 1;
        const bool all = __all_sync(0xffffffffu, okw);
        tc_fence_after();
        return all;
    };

    // Q, K, W in; rows past a short chunk hold the next sequence's tokens: zeroed; Q~ = Q - d K
    bool ok = mbar_wait_polls(smem_u32(&ldA), 0, p.wait_ns);
    if (ok) {
        for (int e = tid; e < (64 - L) * 32; e += 256) {
            const int r = L + (e >> 5), c = 8 * (e & 31);
            *reinterpret_cast<uint4*>(sQK + sw128_offset(r, c, 128)) = make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4*>(sQK + sw128_offset(64 + r, c, 128)) = make_uint4(0, 0, 0, 0);
        }
        for (int e = tid; e < L * 32; e += 256) {
            const int r = e >> 5, c = 8 * (e & 31);
            uint4* qa = reinterpret_cast<uint4*>(sQK + sw128_offset(r, c, 128));
            const uint4 ka = *reinterpret_cast<const uint4*>(sQK + sw128_offset(64 + r, c, 128));
            float qv[8], kv[8];
            unpack8(*qa, qv);
            unpack8(ka, kv);
#pragma unroll
            for (int i = 0; i < 8; ++i) qv[i] -= dh * kv[i];
            *qa = pack8(qv);
        }
    }
    ok = publish_ok(ok);   // (also publishes sG)

    // S = Q~ K^T
    if (tid == 0) {
        if (ok) tc_gemm_m64<false, false>(tmem + kColS, uQK, 128, uK, 128, 64, kWK, false);
        tc_commit(smem_u32(&bar));
    }
    ok = wait_warp(bar, phB) && ok;
    if (ok) {
        // P = Tril(S * Gamma): this warp's rows, columns 32 wc .. + 31
        float sc[4][4];
        tmem_frag<4>(tq + kColS + 32 * wc, sc);
#pragma unroll
        for (int t = 0; t < 4; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = m0 + frag_row(i), c = 32 * wc + frag_col(t, i);
                sc[t][i] = (c <= r && r < L) ? sc[t][i] * __expf(sG[r] - sG[c]) : 0.f;
            }
        frag_store_sw<4>(sP, 64, m0, 32 * wc, sc);
    }
    // every warp's S product has been read: Qhat = Diag(gamma) Q~ in place (rows < L; the others are 0)
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (ok) {
        for (int e = tid; e < L * 32; e += 256) {
            const int r = e >> 5, c = 8 * (e & 31);
            uint4* qa = reinterpret_cast<uint4*>(sQK + sw128_offset(r, c, 128));
            float qv[8];
            unpack8(*qa, qv);
            const float gr = __expf(sG[r]);
#pragma unroll
            for (int i = 0; i < 8; ++i) qv[i] *= gr;
            *qa = pack8(qv);
        }
    }
    ok = publish_ok(ok);

    // P W (for Z) on bar; value head 0's W H_0 and Qhat H_0 on barV
    auto issue_vproducts = [&](int j) {   // thread 0
        bool okv = mbar_wait_polls(smem_u32(&ldV[j & 1]), (j >> 1) & 1, p.wait_ns);
        if (okv) {
            const uint32_t uH = smem_u32(sHt(j));
            tc_gemm_m64<false, false>(tmem + col_e(j), uW, 64, uH, 64, kWV, kWK, false);       // W H_j
            if (want_o) tc_gemm_m64<false, false>(tmem + col_o(j), uQK, 128, uH, 64, kWV, kWK, false);   // Qhat H_j
        }
        tc_commit(smem_u32(&barV));
        return okv;
    };
    bool okv0 = true;   // thread 0: value head 0's tiles arrived
    if (tid == 0) {
        if (ok && zout) tc_gemm_m64<false, true>(tmem + kColPW, uP, 64, uW, 64, kWK, 64, false);   // P W
        tc_commit(smem_u32(&bar));
        if (ok) okv0 = issue_vproducts(0);
        else tc_commit(smem_u32(&barV));
    }
    ok = wait_warp(bar, phB) && ok;
    if (ok && zout) {
        // Z = Qhat - P W: this warp's rows, columns 128 wc .. + 127 in four 32-column passes, staged
        // over K's rows of the Q/K tile (dead since S)
#pragma unroll 1
        for (int pass = 0; pass < 4; ++pass) {
            const int n0 = 128 * wc + 32 * pass;
            float z[4][4];
            tmem_frag<4>(tq + kColPW + n0, z);
            uint32_t w[8];
            frag_load_sw<4>(sQK, 128, m0, n0, w);
#pragma unroll
            for (int t = 0; t < 4; ++t)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const float2 q2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[2 * t + hh]));
                    z[t][2 * hh] = q2.x - z[t][2 * hh];
                    z[t][2 * hh + 1] = q2.y - z[t][2 * hh + 1];
                }
            frag_store_sw<4>(sQK, 128, 64 + m0, n0, z);
        }
    }
    if (warp == 0) ok = __all_sync(0xffffffffu, ok && okv0);   // (warp-uniform ahead of the TMEM loads)

    for (int j = 0; j < vg; ++j) {
        ok = wait_warp(barV, phV) && ok;   // W H_j and Qhat H_j (thread 0's tile wait folds in at the barrier)
        if (ok) {
            // E_j = U_j - W H_j: this warp's rows, columns 32 wc .. + 31 (rows past a short chunk are
            // zero: W and U rows there are)
            float ev[4][4];
            tmem_frag<4>(tq + col_e(j) + 32 * wc, ev);
            uint32_t w[8];
            frag_load_sw<4>(sU(j), 64, m0, 32 * wc, w);
#pragma unroll
            for (int t = 0; t < 4; ++t)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const float2 u2 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[2 * t + hh]));
                    ev[t][2 * hh] = u2.x - ev[t][2 * hh];
                    ev[t][2 * hh + 1] = u2.y - ev[t][2 * hh + 1];
                }
            frag_store_sw<4>(sE(j), 64, m0, 32 * wc, ev);
        }
        ok = publish_ok(ok);
        if (ok && tid == kTma) {
            if (j == 0 && zout)
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_store_2d(&mp.z, 64 * b, (int)(idx0 * 64), uK + b * 16384);
            if (eout) tma_store_2d(&mp.e, 0, (int)((idx0 + j) * 64), smem_u32(sE(j)));
        }
        // O_j += P E_j, then value head j + 1's products into the other column set
        bool okv = true;
        if (tid == 0) {
            if (ok && want_o) tc_gemm_m64<false, true>(tmem + col_o(j), uP, 64, smem_u32(sE(j)), 64, kWV, 64, true);
            tc_commit(smem_u32(&barO));
            if (j + 1 < vg) {
                if (ok) okv = issue_vproducts(j + 1);
                else tc_commit(smem_u32(&barV));
            }
        }
        ok = wait_warp(barO, phO) && ok;
        // value head j's buffer is free (its products are complete): value head j + 2's tiles
        if (ok && tid == kTma && j + 2 < vg) issue_v(j + 2);
        if (ok && want_o) {
            float o[4][4];
            tmem_frag<4>(tq + col_o(j) + 32 * wc, o);
            frag_store_sw<4>(sO(j), 64, m0, 32 * wc, o);
        }
        // the stores of value head j - 1 have read their staging (the next value head reuses it)
        if (tid == kTma) bulk_wait_all_reads();
        if (tid == 0) ok = ok && okv;
        ok = publish_ok(ok);
        if (ok && want_o) {
            const int hv = hk * vg + j;
            if (L == kChunk) {
                if (tid == kTma) tma_store_3d(&mp.o, 0, hv, t0, smem_u32(sO(j)));
            } else {
                // a short chunk by rows (a 64-row box would run into the next sequence)
                bf16* og = (bf16*)p.o + ((long long)t0 * p.H + hv) * kWV;
                for (int e = tid; e < L * 8; e += 256) {
                    const int r = e >> 3, ch = e & 7;
                    *reinterpret_cast<uint4*>(og + (long long)r * p.H * kWV + 8 * ch) =
                        *reinterpret_cast<const uint4*>(sO(j) + sw128_offset(r, 8 * ch, 64));
                }
            }
        }
        if (tid == kTma) bulk_commit();
        if (!ok) break;
    }

    if (!ok) {
        // a wait gave up: let every load and product in flight land before the block's shared memory
        // and TMEM go (the waits still pending are the last issued of each barrier)
        if (tid == kTma) {
            mbar_drain(smem_u32(&ldA), 0);
            for (int j = nv > 2 ? nv - 2 : 0; j < nv; ++j) mbar_drain(smem_u32(&ldV[j & 1]), (j >> 1) & 1);
        }
        if (tid == 0) {
            flag_error(p);
            tc_commit(smem_u32(&bar));
            mbar_drain(smem_u32(&bar), phB);
        }
    }
    if (tid == kTma) bulk_wait_all_done();   // every bulk store has completed before the block exits
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

}  // namespace
}  // namespace tc

cudaError_t launch_output_wide_tc(const ChunkParams& p, cudaStream_t s) {
    using namespace tc;
    const size_t sm = OutWideSmem::bytes();
    cudaError_t e = cudaFuncSetAttribute(k_output_wide_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    if (p.slots <= 0) return cudaSuccess;
    const long long pairs = (long long)p.slots * p.H;
    if (pairs * 64 >= (1ll << 31)) return cudaErrorInvalidValue;   // TMA row coordinates are 32-bit
    const int Hk = p.H / p.vg;
    OutWideMaps mp;
    bool good = make_bf16_token_map(&mp.q, p.q, p.Ttot, Hk, kWK) && make_bf16_token_map(&mp.k, p.k, p.Ttot, Hk, kWK) &&
                make_bf16_map(&mp.w, p.Wb, pairs * 64, kWK, 64) && make_bf16_map(&mp.h, p.Hb, pairs * 64, kWK, 64) &&
                make_bf16_map(&mp.u, p.Ub, pairs * 64, kWV, 64);
    if (good && p.o) good = make_bf16_token_map(&mp.o, p.o, p.Ttot, p.H, kWV);
    else mp.o = mp.q;   // not used
    if (good && p.Eb) good = make_bf16_map(&mp.e, p.Eb, pairs * 64, kWV, 64);
    else mp.e = mp.u;   // not used
    if (good && p.Zb) good = make_bf16_map(&mp.z, p.Zb, pairs * 64, kWK, 64);
    else mp.z = mp.w;   // not used
    if (!good) return cudaErrorInvalidValue;
    k_output_wide_tc<<<dim3(p.slots, Hk), 256, sm, s>>>(p, mp);
    return cudaGetLastError();
}

size_t output_wide_tc_smem_bytes() { return tc::OutWideSmem::bytes(); }

cudaError_t launch_prep_wide_tc(const ChunkParams& p, cudaStream_t s) {
    using namespace tc;
    const size_t sm = PrepWideSmem::bytes();
    cudaError_t e = cudaFuncSetAttribute(k_prep_wide_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    if (p.slots <= 0) return cudaSuccess;
    const long long pairs = (long long)p.slots * p.H;
    if (pairs * 64 >= (1ll << 31)) return cudaErrorInvalidValue;   // TMA row coordinates are 32-bit
    const int Hk = p.H / p.vg;
    PrepWideMaps mp;
    bool good = make_bf16_token_map(&mp.k, p.k, p.Ttot, Hk, kWK) && make_bf16_token_map(&mp.v, p.v, p.Ttot, p.H, kWV) &&
                make_bf16_map(&mp.w, p.Wb, pairs * 64, kWK, 64) && make_bf16_map(&mp.u, p.Ub, pairs * 64, kWV, 64);
    if (good && p.p) good = make_bf16_token_map(&mp.p, p.p, p.Ttot, Hk, kWK);
    else mp.p = mp.k;   // not used
    if (!good) return cudaErrorInvalidValue;
    k_prep_wide_tc<<<dim3(p.slots, Hk), 256, sm, s>>>(p, mp);
    return cudaGetLastError();
}

size_t prep_wide_tc_smem_bytes() { return tc::PrepWideSmem::bytes(); }

}  // namespace comba
