// tcgen05 (5th-generation tensor core) kernels for the bf16, dk = dv = 128 path.
//
// Every tile product is issued by one thread as tcgen05.mma (M = 128, fp32
// accumulator in TMEM) on 128-byte-swizzled shared-memory tiles that TMA
// loads; the other threads run the epilogues on the
// rows they read back from TMEM (one row per thread).  Products are formed
// transposed where that puts a 128-wide head dimension on M (W^T, U^T, E^T,
// O^T, (P W)^T); 64 x 64 chunk products pad M to 128 with zero rows.
//
//   k_prep_tc      Gram K K^T -> decay/btilde mask -> UT inverse M (fp32 forward
//                  substitution on the 16 x 16 diagonal blocks, tf32 tile products for
//                  the off-diagonal levels) -> W^T = K^T Mw^T, U^T = V^T Mu^T ->
//                  Atilde = -K^T Diag(s) W  (s = gamma_C/gamma_r), and U_s^T = (Diag(s) U)^T
//                  for the forward scan, which forms B^T = U_s^T K itself;
//                  with Comba-pk feedback vectors P: Gram P K^T and W^T = P^T Mw^T
//   k_output_tc    P = Tril(Q~ K^T * Gamma), E^T = U^T - H^T W^T,
//                  O^T = H^T Qhat^T + E^T P^T  (Qhat = Diag(gamma) Q~); for the
//                  backward also Z^T = Qhat^T - W^T P^T, the factor of the reverse
//                  scan's additive term C = Z^T dO (formed by the scan itself)
//
// Workspace tensors of this path: W^T, U^T, U_s^T, Z^T [pairs][128][64]; Atilde,
// H^T, dH^T [pairs][128][128]; E [pairs][64][128] row-major; M [pairs][64][64].
#include <cuda.h>

#include "tc_tiles.cuh"

namespace comba {

bool make_bf16_token_map(CUtensorMap* m, const void* base, long long tokens, int heads, int cols);
bool make_bf16_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows);

namespace tc {

// ------------------------------------------------------------------ prep

struct PrepTcSmem {
    static constexpr uint32_t OK = 0;                    // K  [128 alloc rows][128]   32 KB
    static constexpr uint32_t OV = OK + 32768;           // V  [64][128]               16 KB
    static constexpr uint32_t OMW = OV + 16384;          // Mw [64][64] K-major         8 KB
    static constexpr uint32_t OMU = OMW + 8192;          // Mu [64][64]                 8 KB
    static constexpr uint32_t OR = OMU + 8192;           // A^T, M (pitches kAtPitch, kMPitch), T fp32, then sW^T, sU_s^T [128][64],
                                                         // then the Atilde staging [128][128]
    static constexpr uint32_t R_BYTES = (64 * kAtPitch + 64 * kMPitch + 1024) * 4;
    static constexpr uint32_t OF = OR + ((R_BYTES + 1023) & ~1023u);
    static constexpr size_t bytes() { return 1024 + OF + 64 * 6 * 4; }
};

// Tensor maps of the prep kernel's traffic, 128-byte swizzled: token tiles {64 columns, 1 head,
// 64 tokens} of k and p (key heads) and v (value heads) in; the workspace tiles W^T, U^T, U_s^T
// ([pairs * 128][64], one 128-row box) and Atilde ([pairs * 128][128], two 128-row boxes of 64
// columns) out by bulk tensor stores.
struct PrepMaps {
    CUtensorMap k, p, v;
    CUtensorMap w, u, us, a;
};

// 256 threads: warps w and w + 4 read the same TMEM lane quadrant and split its columns.
// Persistent: two CTAs per SM, CTA b taking units b, b + G, ... (G = gridDim.x).  A unit's gates
// are requested at the previous unit's start and its K (or [P; K]) and V tiles by TMA as soon as
// the previous unit's Atilde product has read K (Atilde is staged in the dead W^T / U_s^T region),
// so that loads overlap the previous unit's last epilogue and copies.  W^T, U^T, U_s^T and Atilde
// leave by bulk tensor stores (thread 32) from swizzled staging tiles; each staging tile is
// reused only once those stores have read it.
__global__ void __launch_bounds__(256, 2) k_prep_tc(ChunkParams p, long long pairs, const __grid_constant__ PrepMaps mp) {
    constexpr int NTH = 256;
    constexpr int kStore = 32;   // issues the bulk tensor stores and waits for them
    using S = PrepTcSmem;
    extern __shared__ uint8_t smem_raw[];
    // stall_bar: nothing arrives (COMBA_DIAG_STALL); ld: a unit's tiles (one phase per unit)
    __shared__ uint64_t bar, stall_bar, ld;
    __shared__ uint32_t tbase;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sK = sm + S::OK;
    uint8_t* sV = sm + S::OV;
    uint8_t* sMw = sm + S::OMW;
    uint8_t* sMu = sm + S::OMU;
    float* sAt = reinterpret_cast<float*>(sm + S::OR);   // A transposed
    float* sM = sAt + 64 * kAtPitch;
    float* sTi = sM + 64 * kMPitch;                    // inverse scratch, 1024 floats
    uint8_t* sWt = sm + S::OR;            // aliases A after the inverse
    uint8_t* sUt = sm + S::OR + 16384;    // aliases M after Mw/Mu are built
    uint8_t* stA = sm + S::OR;            // Atilde staging [128][128], once W^T / U_s^T are dead
    float* sG = reinterpret_cast<float*>(sm + S::OF);
    float* sGm1 = sG + 64;
    float* sBt = sG + 128;
    float* sBe = sG + 192;
    float* sS = sG + 256;
    float* sWs = sG + 320;   // btilde_c gamma_{c-1}: the column scale of Mw

    // K into both halves of the 128-row tile: rows 64..127 repeat rows 0..63, so the
    // padded Gram product puts a copy of each Gram row in TMEM lanes r and r + 64.  With
    // Comba-pk feedback vectors the tile is [P; K] instead: the Gram's lanes 0..63 hold
    // P K^T, and K (rows 64..127) is the operand of every later product that takes K.
    const bool pk = p.p != nullptr;
    const int Hk = p.H / p.vg;
    const uint32_t Hh = (uint32_t)p.H;   // (unit indices fit 32 bits: the launcher checks)
    if (tid == 0) {
        mbar_init(smem_u32(&bar), 1);
        mbar_init(smem_u32(&stall_bar), 1);
        mbar_init(smem_u32(&ld), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tbase), 256);
    tc_fence_before();
    __syncthreads();   // barriers initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem = tbase;
    MmaSync ms{smem_u32(&bar), smem_u32(p.stall ? &stall_bar : &bar), 0, p.wait_ns};
    const int row = tid & 127, half = tid >> 7;   // TMEM lane / accumulator row, and which column half
    const uint32_t trow = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const uint8_t* sKk = pk ? sK + 64 * 128 : sK;   // the 64 key rows (rows 64.. of each K-half for pk)

    // a unit's gates into registers: warp 0 the log-decay inputs, threads < 64 beta, alpha and b
    struct Gates { float a0, a1, bev, alv, bh; };
    auto fetch_gates = [&](long long x, const SlotInfo& si) {
        Gates g{1.f, 1.f, 0.f, 1.f, 1.f};
        const int hkx = (int)((uint32_t)x % Hh) / p.vg;
        const float* ag = p.alpha + (long long)si.start * Hk + hkx;
        if (warp == 0) {
            g.a0 = lane < si.len ? ag[(long long)lane * Hk] : 1.f;
            g.a1 = lane + 32 < si.len ? ag[(long long)(lane + 32) * Hk] : 1.f;
        }
        if (tid < 64) {
            g.bev = tid < si.len ? p.beta[((long long)si.start + tid) * Hk + hkx] : 0.f;
            g.alv = tid < si.len ? ag[(long long)tid * Hk] : 1.f;
            g.bh = p.b ? p.b[hkx] : 1.f;
        }
        return g;
    };
    auto slot_of = [&](long long x) { return x < pairs ? p.slot_info[(uint32_t)x / Hh] : SlotInfo{0, 0, 0, 0}; };
    auto issue_tiles = [&](long long x, const SlotInfo& si) {   // thread 0
        const int hx = (int)((uint32_t)x % Hh), hkx = hx / p.vg;
        const uint32_t mb = smem_u32(&ld);
        mbar_expect_tx(mb, 32768u + 16384u);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            tma_load_3d(smem_u32(sK) + hh * 16384, pk ? &mp.p : &mp.k, 64 * hh, hkx, si.start, mb);
            tma_load_3d(smem_u32(sK) + 8192 + hh * 16384, &mp.k, 64 * hh, hkx, si.start, mb);
            tma_load_3d(smem_u32(sV) + hh * 8192, &mp.v, 64 * hh, hx, si.start, mb);
        }
    };

    bool ok = true;
    uint32_t ph = 0;      // phase parity of `ld` for the current unit
    bool pend = false;    // thread 0: the coming unit's tiles are requested already
    long long u = blockIdx.x;
    const long long G = gridDim.x;
    SlotInfo s0 = slot_of(u), s1 = slot_of(u + G);   // this unit's slot and the next one's
    Gates g0 = s0.len > 0 ? fetch_gates(u, s0) : Gates{1.f, 1.f, 0.f, 1.f, 1.f};
    for (; u < pairs && ok; u += G) {
        const SlotInfo sc = s0;
        const Gates gc = g0;
        s0 = s1;                                        // the next unit: its gates now, its slot's
        g0 = s0.len > 0 ? fetch_gates(u + G, s0) : Gates{1.f, 1.f, 0.f, 1.f, 1.f};
        s1 = slot_of(u + 2 * G);                        // successor a unit later
        if (sc.len <= 0) continue;
        const int L = sc.len;
        const long long idx = u;

        if (tid == 0) {
            if (!pend) issue_tiles(u, sc);
            pend = false;
        }
        if (warp == 0) chunk_log_cumsum_vals(gc.a0, gc.a1, L, sG, sGm1);
        if (tid < 64) {
            sBe[tid] = gc.bev;
            sBt[tid] = gc.bh * gc.bev * feedback_scale(p.iplr, gc.alv);
        }
        __syncthreads();   // sG, sGm1, sBt complete
        if (tid < 64) sWs[tid] = sBt[tid] * expf(sGm1[tid]);
        // the tiles: rows past a short chunk hold the next sequence's tokens, zeroed here
        const bool okl = mbar_wait_polls(smem_u32(&ld), ph, p.wait_ns);
        if (okl && L < kChunk) {
            for (int e = tid; e < (64 - L) * 16; e += NTH) {
                const int r = L + (e >> 4), ch = e & 15;
                const uint4 z = make_uint4(0, 0, 0, 0);
                *reinterpret_cast<uint4*>(sK + sw128_offset(r, 8 * ch, 128)) = z;
                *reinterpret_cast<uint4*>(sK + sw128_offset(64 + r, 8 * ch, 128)) = z;
                *reinterpret_cast<uint4*>(sV + sw128_offset(r, 8 * ch, 64)) = z;
            }
        }
        if (tid == kStore) bulk_wait_all_reads();   // the previous unit's Atilde store has read A^T's region
        fence_async_smem();
        tc_fence_before();
        ok = !__syncthreads_or(!okl);
        tc_fence_after();

        // Gram K K^T over the 128-row tile (P K^T in lanes 0..63 for Comba-pk).
        if (tid == 0 && ok) tc_gemm<false, false>(tmem, smem_u32(sK), 128, smem_u32(sKk), 128, 64, D, false);
        if (tid < 64) sS[tid] = tid < L ? expf(sG[L - 1] - sG[tid]) : 0.f;
        ok = ms.finish_warp(tid) && ok;
        if (ok && !pk) {
            // Strictly-lower A = Diag(btilde)(gamma_{r-1}/gamma_i * K K^T), stored transposed; exp only
            // below the diagonal.  Lane l holds Gram row l & 63; its two threads fill columns
            // [32 (l >> 6) + 16 half, +16).
            const int r = row & 63, i0 = 32 * (row >> 6) + 16 * half;
            float d[16];
            tmem_ld16(trow + i0, d);
            const float br = r < L ? sBt[r] : 0.f, gr = sGm1[r];
#pragma unroll
            for (int c = 0; c < 16; ++c) {
                const int i = i0 + c;
                sAt[i * kAtPitch + r] = i < r ? br * __expf(gr - sG[i]) * d[c] : 0.f;
            }
        } else if (ok && row < 64) {
            // Comba-pk: P K^T rows are in lanes 0..63 only; the two threads of each take one column half.
            const int r = row, i0 = 32 * half;
            const float br = r < L ? sBt[r] : 0.f, gr = sGm1[r];
            float d[32];
            tmem_ld32(trow + i0, d);
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                const int i = i0 + c;
                sAt[i * kAtPitch + r] = i < r ? br * __expf(gr - sG[i]) * d[c] : 0.f;
            }
        }
        ok = !__syncthreads_or(!ok);   // the inverse's barriers below need a block-uniform flag
        if (ok) {
            unit_lower_inverse64_h16(sAt, sM, sTi, tid);
            __syncthreads();
            // Mw = M Diag(btilde gamma_{r-1}), Mu = M Diag(beta) as K-major [p][p'] tiles; M saved for the backward.
            bf16* Mg = p.Mb ? (bf16*)p.Mb + idx * 4096 : nullptr;
            for (int e = tid; e < 64 * 8; e += NTH) {
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
            if (tid < 64) p.Gb[idx * 64 + tid] = sG[tid];
        }
        publish_smem();

        // W^T = K^T Mw^T (A = K as MN-major; P^T Mw^T for Comba-pk, tile rows 0..63), U^T = V^T Mu^T.
        if (ok && tid == 0) {
            tc_gemm<true, false>(tmem + 64, smem_u32(sK), 128, smem_u32(sMw), 64, 64, 64, false);
            tc_gemm<true, false>(tmem + 128, smem_u32(sV), 64, smem_u32(sMu), 64, 64, 64, false);
        }
        ok = ok && ms.finish_warp(tid);   // (ok is block-uniform here: every thread takes the same branch)
        // W^T and U^T for the workspace are staged (swizzled) over the dead V and Mw/Mu tiles.
        uint8_t* stW = sV;
        uint8_t* stU = sMw;
        if (ok) {
            float d[32], v[8], w[8];
            {
                const int g = half;
                tmem_ld32(trow + 64 + g * 32, d);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        v[e] = d[8 * q + e];
                        w[e] = v[e] * sS[32 * g + 8 * q + e];
                    }
                    *reinterpret_cast<uint4*>(stW + sw128_offset(row, 32 * g + 8 * q, 128)) = pack8(v);
                    *reinterpret_cast<uint4*>(sWt + sw128_offset(row, 32 * g + 8 * q, 128)) = pack8(w);
                }
            }
            {
                const int g = half;
                tmem_ld32(trow + 128 + g * 32, d);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        v[e] = d[8 * q + e];
                        w[e] = v[e] * sS[32 * g + 8 * q + e];
                    }
                    *reinterpret_cast<uint4*>(stU + sw128_offset(row, 32 * g + 8 * q, 128)) = pack8(v);
                    *reinterpret_cast<uint4*>(sUt + sw128_offset(row, 32 * g + 8 * q, 128)) = pack8(w);
                }
            }
        }
        ok = publish_ok(ok);

        // Atilde = -K^T (Diag(s) W) -> cols [0,128)
        if (ok && tid == 0) tc_gemm<true, false>(tmem, smem_u32(sKk), 128, smem_u32(sWt), 128, 128, 64, false);
        if (ok && tid == kStore) {
            // W^T, U^T and U_s^T out while the tensor core works; their staging is reused only once
            // the stores have read it
            const int y = (int)((uint32_t)u * (uint32_t)D);
            tma_store_2d(&mp.w, 0, y, smem_u32(stW));
            tma_store_2d(&mp.u, 0, y, smem_u32(stU));
            tma_store_2d(&mp.us, 0, y, smem_u32(sUt));
            bulk_commit();
            bulk_wait_all_reads();
        }
        ok = ok && ms.finish_warp(tid);
        // K, V and the W^T / U^T / U_s^T staging are dead now, for every thread: the next unit's
        // tiles may load, and Atilde is staged over W^T / U_s^T's region
        ok = !__syncthreads_or(!ok);
        if (!ok) break;
        if (tid == 0 && u + G < pairs && s0.len > 0) {
            issue_tiles(u + G, s0);
            pend = true;
        }
        {
            float d[32], v[8];
#pragma unroll
            for (int g = 2 * half; g < 2 * half + 2; ++g) {
                tmem_ld32(trow + g * 32, d);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) v[e] = -d[8 * q + e];
                    *reinterpret_cast<uint4*>(stA + sw128_offset(row, 32 * g + 8 * q, 128)) = pack8(v);
                }
            }
        }
        fence_async_smem();
        tc_fence_before();   // the unit's last TMEM reads: the next unit's Gram may follow
        __syncthreads();
        tc_fence_after();
        if (tid == kStore) {   // Atilde out; the next unit's A^T (over the staging) waits for the read
            const int y = (int)((uint32_t)u * (uint32_t)D);
            tma_store_2d(&mp.a, 0, y, smem_u32(stA));
            tma_store_2d(&mp.a, 64, y, smem_u32(stA) + 16384);
            bulk_commit();
        }
        ph ^= 1;
    }
    if (!ok) {
        if (tid == 0) {
            flag_error(p);
            mbar_drain(smem_u32(&ld), ph);   // the tile loads have ended before the block's memory goes
        }
        ms.drain(tid);
    }
    if (tid == kStore) bulk_wait_all_done();   // and every bulk store has completed
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 256);
}

// ---------------------------------------------------------------- output

struct OutTcSmem {
    static constexpr uint32_t OQK = 0;             // [128 rows][128]: rows 0-63 Q -> Q~ -> Qhat, rows 64-127 K;
                                                   // P [64][64] later over K's first half     32 KB
    static constexpr uint32_t OW = 32768;          // W^T [128][64] (MN-major B, then K-major A), later E [64][128]  16 KB
    static constexpr uint32_t OU = OW + 16384;     // U^T [128][64], then E^T in place, later Z^T staging             16 KB
    static constexpr uint32_t OH = OU + 16384;     // H^T [128][128] K-major, later O staging [64][128]              32 KB
    static constexpr uint32_t OG = OH + 32768;
    static constexpr size_t bytes() { return 1024 + OG + 64 * 4; }
};

// Tensor maps of the output kernel: token tiles {64 columns, 1 head, 64 tokens} of q, k (key heads)
// and o (value heads); workspace tiles of W^T, U^T, Z^T ([pairs * 128][64], 128-row boxes) and
// H^T ([pairs * 128][128], 128-row boxes of 64 columns).  All 128-byte swizzled.
struct OutMaps {
    CUtensorMap q, k, o, w, u, h, z;
};

// 256 threads: warps w and w + 4 read the same TMEM lane quadrant and split its columns.
// Persistent: two CTAs per SM, CTA b taking units b, b + G, b + 2G, ... (G = gridDim.x).  Tiles
// arrive by TMA in two groups: Q and K (all that Q~, S = Q~ K^T and P need), requested as soon as
// the previous unit's Qhat is dead, and H^T, W^T and U^T, requested once the previous unit's
// bulk stores have read their staging tiles, so that a unit's Q/K load overlaps the previous
// unit's stores and Q~, S and P overlap the larger load.  O and Z^T leave by bulk tensor stores
// and E by a bulk copy, from staging tiles over the dead inputs.
__global__ void __launch_bounds__(256, 2) k_output_tc(ChunkParams p, long long pairs, const __grid_constant__ OutMaps mp) {
    constexpr int NTH = 256;
    using S = OutTcSmem;
    extern __shared__ uint8_t smem_raw[];
    // ldA: Q/K landed; ldB: H^T, W^T, U^T landed; barS: S; barE: H^T W^T; bar: the second products;
    // stall_bar: nothing arrives (COMBA_DIAG_STALL).  ldA .. barE complete one phase per unit.
    __shared__ uint64_t ldA, ldB, barS, barE, bar, stall_bar;
    __shared__ uint32_t tbase;
    const int tid = threadIdx.x, warp = tid >> 5;
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sQK = sm + S::OQK;
    uint8_t* sP = sQK + 64 * 128;   // K's rows of the first 64-column half, dead after S = Q~ K^T
    uint8_t* sWt = sm + S::OW;
    uint8_t* sUt = sm + S::OU;
    uint8_t* sEt = sUt;                        // E^T replaces U^T row by row
    bf16* sE = reinterpret_cast<bf16*>(sWt);   // [64][128] row-major staging of E, once W^T is dead
    uint8_t* stZ = sUt;                        // Z^T staging (128-byte swizzled), once E^T is dead
    uint8_t* sHt = sm + S::OH;
    uint8_t* stO = sHt;                        // O staging: two [64][64] swizzled halves, once H^T is dead
    float* sG = reinterpret_cast<float*>(sm + S::OG);
    const uint32_t uA = smem_u32(&ldA), uB = smem_u32(&ldB);

    if (tid == 0) {
        mbar_init(uA, 1);
        mbar_init(uB, 1);
        mbar_init(smem_u32(&barS), 1);
        mbar_init(smem_u32(&barE), 1);
        mbar_init(smem_u32(&bar), 1);
        mbar_init(smem_u32(&stall_bar), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tbase), 256);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tbase;
    MmaSync ms{smem_u32(&bar), smem_u32(p.stall ? &stall_bar : &bar), 0, p.wait_ns};
    const int row = tid & 127, half = tid >> 7;   // TMEM lane, and which 32 of each 64 columns
    const uint32_t trow = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const uint32_t Hh = (uint32_t)p.H;            // (unit indices fit 32 bits: the launcher checks)
    const bool Zg = p.Zb != nullptr;
    const bool mma2 = p.o || Zg;

    // a unit's slot, d and log-decays, requested a unit ahead
    auto fetch = [&](long long x, SlotInfo& si, float& d, float& g) {
        const uint32_t sl = (uint32_t)x / Hh;
        const int hx = (int)((uint32_t)x - sl * Hh);
        si = p.slot_info[sl];
        d = p.d[hx / p.vg];
        g = tid < 64 ? p.Gb[x * 64 + tid] : 0.f;
    };
    auto issue_qk = [&](long long t0x, int hkx) {   // thread 0
        mbar_expect_tx(uA, 32768u);
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
            tma_load_3d(smem_u32(sQK) + hh * 16384, &mp.q, 64 * hh, hkx, (int)t0x, uA);
            tma_load_3d(smem_u32(sQK) + 8192 + hh * 16384, &mp.k, 64 * hh, hkx, (int)t0x, uA);
        }
    };

    bool ok = true;
    uint32_t ph = 0;       // phase parity of ldA .. barE for the current unit
    bool pendA = false;    // thread 0: the coming unit's Q/K are requested already
    long long u = blockIdx.x;
    SlotInfo si{0, 0, 0, 0};
    float dh = 0.f, gv = 0.f;
    if (u < pairs) fetch(u, si, dh, gv);
    for (; u < pairs && ok; u += gridDim.x) {
        const SlotInfo sc = si;
        const float dhc = dh, gvc = gv;
        const long long un = u + gridDim.x;
        if (un < pairs) fetch(un, si, dh, gv);
        if (sc.len <= 0) continue;
        const int L = sc.len;
        const long long t0 = sc.start;
        const long long idx = u;
        const int h = (int)((uint32_t)u % Hh), hk = h / p.vg;

        if (tid == 0) {
            if (!pendA) issue_qk(t0, hk);
            pendA = false;
            bulk_wait_all_reads();   // the previous unit's stores have read W^T, U^T, H^T's tiles
            mbar_expect_tx(uB, 65536u);
            tma_load_2d(smem_u32(sWt), &mp.w, 0, (int)(idx * 128), uB);
            tma_load_2d(smem_u32(sUt), &mp.u, 0, (int)(idx * 128), uB);
#pragma unroll
            for (int hh = 0; hh < 2; ++hh)
                tma_load_2d(smem_u32(sHt) + hh * 16384, &mp.h, 64 * hh, (int)(idx * 128), uB);
        }
        if (tid < 64) sG[tid] = gvc;

        // Q and K in; rows past a short chunk hold the next sequence's tokens: zero them
        const bool okA = mbar_wait_polls(uA, ph, p.wait_ns);
        if (L < kChunk) {
            for (int e = tid; okA && e < (64 - L) * 16; e += NTH) {
                const int r = L + (e >> 4), ch = e & 15;
                *reinterpret_cast<uint4*>(sQK + sw128_offset(r, 8 * ch, 128)) = make_uint4(0, 0, 0, 0);
                *reinterpret_cast<uint4*>(sQK + sw128_offset(64 + r, 8 * ch, 128)) = make_uint4(0, 0, 0, 0);
            }
            __syncthreads();
        }
        // Q~ = Q - d K (rows < L)
        for (int e = tid; okA && e < L * 16; e += NTH) {
            const int r = e >> 4, ch = e & 15;
            uint4* qa = reinterpret_cast<uint4*>(sQK + sw128_offset(r, 8 * ch, 128));
            const uint4 ka = *reinterpret_cast<const uint4*>(sQK + sw128_offset(64 + r, 8 * ch, 128));
            float qv[8], kv[8];
            unpack8(*qa, qv);
            unpack8(ka, kv);
#pragma unroll
            for (int i = 0; i < 8; ++i) qv[i] -= dhc * kv[i];
            *qa = pack8(qv);
        }
        fence_async_smem();
        tc_fence_before();
        ok = !__syncthreads_or(!okA);
        tc_fence_after();

        // [Q~; K] K^T -> cols [0,64) (lanes 0-63: S = Q~ K^T; lanes 64-127 unused), then, once H^T,
        // W^T and U^T are in, E^T' = H^T W^T -> cols [64,128), each on its own barrier
        if (tid == 0) {
            if (ok) tc_gemm<false, false>(tmem, smem_u32(sQK), 128, smem_u32(sQK) + 64 * 128, 128, 64, D, false);
            tc_commit(smem_u32(&barS));
        }
        const bool okB = mbar_wait_polls(uB, ph, p.wait_ns);
        if (tid == 0) {
            if (ok && okB) tc_gemm<false, true>(tmem + 64, smem_u32(sHt), 128, smem_u32(sWt), 128, 64, D, false);
            tc_commit(smem_u32(&barE));
        }
        bf16* Eg = p.Eb ? (bf16*)p.Eb + idx * 64 * D : nullptr;
        uint32_t ev[16];   // this thread's 32 positions of row j of E^T, packed bf16 pairs
        const bool okS = mbar_wait_polls(smem_u32(&barS), ph, p.wait_ns);
        tc_fence_after();
        if (ok && okS) {
            if (row < 64) {
                // P = Tril(S * Gamma) into a K-major [64][64] tile (B operand of E^T P^T), over K
                float d[32], v[8];
                tmem_ld32(trow + half * 32, d);
                const float gr = sG[row];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const int i = 32 * half + 8 * q + e;
                        v[e] = (i <= row && row < L) ? d[8 * q + e] * __expf(gr - sG[i]) : 0.f;
                    }
                    *reinterpret_cast<uint4*>(sP + sw128_offset(row, 32 * half + 8 * q, 64)) = pack8(v);
                }
            } else {
                // the warps of TMEM lanes 64-127 (no S rows): Qhat = Diag(gamma) Q~ in place
                for (int e = (tid & 63) + 64 * half; e < 64 * 16; e += 128) {
                    const int r = e >> 4, ch = e & 15;
                    uint4* qa = reinterpret_cast<uint4*>(sQK + sw128_offset(r, 8 * ch, 128));
                    float qv[8];
                    unpack8(*qa, qv);
                    const float gr = __expf(sG[r]);
#pragma unroll
                    for (int i = 0; i < 8; ++i) qv[i] *= gr;
                    *qa = pack8(qv);
                }
            }
        }
        const bool okE = mbar_wait_polls(smem_u32(&barE), ph, p.wait_ns) && okB;
        tc_fence_after();
        if (ok && okE) {
            // E^T = U^T - H^T W^T  (half of row j of E^T per thread)
            float d[32], v[8];
            tmem_ld32(trow + 64 + half * 32, d);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                float uu[8];
                unpack8(*reinterpret_cast<const uint4*>(sUt + sw128_offset(row, 32 * half + 8 * q, 128)), uu);
#pragma unroll
                for (int e = 0; e < 8; ++e) v[e] = uu[e] - d[8 * q + e];
                // in place: each thread reads and then overwrites only these 16 bytes of its own row
                const uint4 pk = pack8(v);
                *reinterpret_cast<uint4*>(sEt + sw128_offset(row, 32 * half + 8 * q, 128)) = pk;
                const int b0 = 4 * q;
                ev[b0] = pk.x; ev[b0 + 1] = pk.y; ev[b0 + 2] = pk.z; ev[b0 + 3] = pk.w;
            }
        }
        fence_async_smem();
        tc_fence_before();
        ok = !__syncthreads_or(!(ok && okS && okE));
        tc_fence_after();

        // O^T = H^T Qhat^T + E^T P^T -> cols [128,192);  (P W)^T = W^T P^T -> cols [192,256)
        if (ok && tid == 0) {
            if (p.o) {
                tc_gemm<false, false>(tmem + 128, smem_u32(sHt), 128, smem_u32(sQK), 128, 64, D, false);
                tc_gemm<false, false>(tmem + 128, smem_u32(sEt), 128, smem_u32(sP), 64, 64, 64, true);
            }
            if (Zg) tc_gemm<false, false>(tmem + 192, smem_u32(sWt), 128, smem_u32(sP), 64, 64, 64, false);
        }
        if (mma2) ok = ok && ms.finish_warp(tid);   // (ok is block-uniform before it)
        // W^T, E^T and H^T are dead: E, Z^T and O are staged over them.
        if (ok && Eg) {
#pragma unroll
            for (int pp = 0; pp < 16; ++pp) {
                const __nv_bfloat162 two = *reinterpret_cast<const __nv_bfloat162*>(&ev[pp]);
                sE[(32 * half + 2 * pp) * D + row] = two.x;
                sE[(32 * half + 2 * pp + 1) * D + row] = two.y;
            }
        }
        if (ok && Zg) {
            // Z^T = Qhat^T - (P W)^T: row `row` (a key dimension), positions [32 half, +32); columns
            // past a short chunk are zero because Qhat and P rows past it are
            float d[32], v[8];
            tmem_ld32(trow + 192 + half * 32, d);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int t = 32 * half + 8 * q + e;
                    const float qh = __bfloat162float(*reinterpret_cast<const bf16*>(sQK + sw128_offset(t, row, 128)));
                    v[e] = qh - d[8 * q + e];
                }
                *reinterpret_cast<uint4*>(stZ + sw128_offset(row, 32 * half + 8 * q, 128)) = pack8(v);
            }
        }
        if (ok && p.o) {
            // O[t][j] for j = row, t in [32 half, +32): the [64][128] tile as two swizzled 64-column halves
            float d[32];
            tmem_ld32(trow + 128 + half * 32, d);
            uint8_t* oh = stO + (row >> 6) * 8192;
#pragma unroll
            for (int c = 0; c < 32; ++c)
                *reinterpret_cast<bf16*>(oh + sw128_offset(32 * half + c, row & 63, 64)) = __float2bfloat16_rn(d[c]);
        }
        fence_async_smem();
        tc_fence_before();   // every TMEM read of the unit is done: the next unit's products may follow
        ok = !__syncthreads_or(!ok);
        tc_fence_after();
        if (!ok) break;
        if (tid == 0) {
            if (Eg) bulk_copy_s2g(Eg, smem_u32(sE), 64 * D * 2);
            if (Zg) tma_store_2d(&mp.z, 0, (int)(idx * 128), smem_u32(stZ));
            if (p.o && L == kChunk)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) tma_store_3d(&mp.o, 64 * hh, h, (int)t0, smem_u32(stO) + hh * 8192);
            bulk_commit();
            // the next unit's Q and K (Qhat's last readers were the Z^T staging and the second products)
            if (un < pairs && si.len > 0) {
                issue_qk(si.start, (int)((uint32_t)un % Hh) / p.vg);
                pendA = true;
            }
        }
        if (p.o && L < kChunk) {
            // a short chunk by rows (a 64-row box would run into the next sequence)
            bf16* Og = (bf16*)p.o + (t0 * p.H + h) * D;
            for (int e = tid; e < L * 16; e += NTH) {
                const int r = e >> 4, ch = e & 15;
                *reinterpret_cast<uint4*>(Og + (long long)r * p.H * D + 8 * ch) =
                    *reinterpret_cast<const uint4*>(stO + (ch >> 3) * 8192 + sw128_offset(r, 8 * (ch & 7), 64));
            }
        }
        ph ^= 1;
        __syncthreads();   // the O rows above have read their staging before the next unit's H^T load
    }
    if (!ok) {
        if (tid == 0) {
            flag_error(p);
            // let the tile loads and every product end before the block's shared memory and TMEM go
            mbar_drain(uA, ph);
            mbar_drain(uB, ph);
            mbar_drain(smem_u32(&barS), ph);
            mbar_drain(smem_u32(&barE), ph);
        }
        ms.drain(tid);
    }
    if (tid == 0) bulk_wait_all_reads();   // the stores have read their staging before exit
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 256);
}

}  // namespace tc

// -------------------------------------------------------------- launchers

cudaError_t launch_prep_tc(const ChunkParams& p, cudaStream_t s) {
    const size_t sm = tc::PrepTcSmem::bytes();
    cudaError_t e = cudaFuncSetAttribute(tc::k_prep_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    if (p.slots <= 0) return cudaSuccess;
    const long long pairs = (long long)p.slots * p.H;
    if (pairs >= (1ll << 31)) return cudaErrorInvalidValue;   // unit indices are 32-bit in the kernel
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) || (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev))) return e;
    tc::PrepMaps mp;
    bool good = make_bf16_token_map(&mp.k, p.k, p.Ttot, p.H / p.vg, tc::D) &&
                make_bf16_token_map(&mp.v, p.v, p.Ttot, p.H, tc::D) && p.Wb && p.Ub && p.Usb && p.Ab &&
                make_bf16_map(&mp.w, p.Wb, pairs * tc::D, 64, tc::D) &&
                make_bf16_map(&mp.u, p.Ub, pairs * tc::D, 64, tc::D) &&
                make_bf16_map(&mp.us, p.Usb, pairs * tc::D, 64, tc::D) &&
                make_bf16_map(&mp.a, p.Ab, pairs * tc::D, tc::D, tc::D);
    if (good && p.p) good = make_bf16_token_map(&mp.p, p.p, p.Ttot, p.H / p.vg, tc::D);
    else mp.p = mp.k;   // not used
    if (!good) return cudaErrorInvalidValue;
    const long long cap = 2ll * nsm;   // two resident CTAs per SM (shared memory and TMEM)
    const int grid = (int)(pairs < cap ? pairs : cap);
    tc::k_prep_tc<<<grid, 256, sm, s>>>(p, pairs, mp);
    return cudaGetLastError();
}

cudaError_t launch_output_tc(const ChunkParams& p, cudaStream_t s) {
    const size_t sm = tc::OutTcSmem::bytes();
    cudaError_t e = cudaFuncSetAttribute(tc::k_output_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    if (p.slots <= 0) return cudaSuccess;
    const long long pairs = (long long)p.slots * p.H;
    if (pairs >= (1ll << 31)) return cudaErrorInvalidValue;   // unit indices are 32-bit in the kernel
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) || (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev))) return e;
    tc::OutMaps mp;
    bool good = make_bf16_token_map(&mp.q, p.q, p.Ttot, p.H / p.vg, tc::D) &&
                make_bf16_token_map(&mp.k, p.k, p.Ttot, p.H / p.vg, tc::D) &&
                make_bf16_map(&mp.w, p.Wb, pairs * tc::D, 64, tc::D) &&
                make_bf16_map(&mp.u, p.Ub, pairs * tc::D, 64, tc::D) &&
                make_bf16_map(&mp.h, p.Hb, pairs * tc::D, tc::D, tc::D);
    if (good && p.o) good = make_bf16_token_map(&mp.o, p.o, p.Ttot, p.H, tc::D);
    else mp.o = mp.q;   // not used
    if (good && p.Zb) good = make_bf16_map(&mp.z, p.Zb, pairs * tc::D, 64, tc::D);
    else mp.z = mp.w;   // not used
    if (!good) return cudaErrorInvalidValue;
    const long long cap = 2ll * nsm;   // two resident CTAs per SM (shared memory and TMEM)
    const int grid = (int)(pairs < cap ? pairs : cap);
    tc::k_output_tc<<<grid, 256, sm, s>>>(p, pairs, mp);
    return cudaGetLastError();
}

size_t tc_smem_bytes(int kernel) { return kernel == 0 ? tc::PrepTcSmem::bytes() : tc::OutTcSmem::bytes(); }

}  // namespace comba
