// Local chunk gradients on the tcgen05 path (bf16, dk = dv = 128).
//
// Same algebra as k_bwd_local (chunk_bwd.cu): given a chunk's K, Q, V, dO, its
// saved E = U - W H_n, chunk state H_n, incoming state gradient dH' and inverse
// M (and Comba-pk's feedback vectors P), form dq, dk, dv (and dp), the log-decay
// and beta gradients and the per-chunk db, dd partials.  The tile products are tcgen05.mma groups
// with M = 64 (the chunk rows), issued by one thread into TMEM; the warps wait
// on them six times a unit:
//
//   R0  S = Q~ K^T, dP = dO E^T      (its own barrier; R1 is issued right behind)
//   R1  dO H^T, E dH'^T, K dH'      (runs while the warps form P from R0)
//   R2  P^T dO                       (behind R1, one wait: dE = Kbar dH' + P^T dO)
//   R3  M^T dE, dPhat^T Q~
//   R4  (M^T dE) H^T = -M^T dW (dW = -dE H^T), K K^T, dPhat K
//   R5  (M^T dE) E^T                 (= M^T dM M^T: dM = dE (Diag(beta) V)^T + dW Ktilde^T with
//                                     dW = -dE H^T gives (M^T dE) U^T - (M^T dE) (W H)^T, and
//                                     U - W H = E; so dA needs neither dM, U, W nor a second
//                                     product with M)
//   R6  dG K + dG^T K onto dPhat^T Q~
//
// Each epilogue first forms what the next round reads and lets it be issued, then does the rest
// of its work while that round runs.
//
// An M = 64 accumulator read with tcgen05.ld.16x256b gives each warp the rows
// 16 (w & 3) .. + 15 in exactly the m16n8 accumulator fragment layout of
// mma.sync, so the epilogues (masks, decay factors, row and column partial
// sums) are fragment code.  Sixteen warps: w, w + 4, w + 8 and w + 12 share a
// TMEM lane quadrant and take the four column quarters of every accumulator
// (128 registers a thread, so the epilogues' register tiles stay small).
// Operands live in 128-byte-swizzled shared tiles (K-major or MN-major as
// each product needs; no transposed copies).  Outputs are staged in shared
// memory and written with coalesced 16-byte stores.
#include <cuda.h>

#include "tc_frag.cuh"

namespace comba {

bool make_bf16_token_map(CUtensorMap* m, const void* base, long long tokens, int heads, int cols);
bool make_bf16_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows);

namespace tc {

constexpr int kLocalThreads = 512;            // 16 warps: four per TMEM lane quadrant
constexpr int kQ = kLocalThreads / 128;        // column parts of each accumulator (one per warp of a quadrant)
constexpr int NK = 16 / kQ, NL = 8 / kQ;       // m16n8 fragments per warp of 128- and 64-wide results
constexpr int kTail = kLocalThreads - 64;     // the last two warps take the per-position tail

struct LocalTcSmem {
    static constexpr uint32_t OQK = 0;             // two [128][128] tiles (consecutive units alternate): rows 0-63
                                                   // Q -> Q~, rows 64-127 K; later dq, dk staging
    static constexpr uint32_t OV = OQK + 2 * 32768;  // V [64][128]
    static constexpr uint32_t ODO = OV + 16384;    // dO [64][128]
    static constexpr uint32_t OE = ODO + 16384;    // E [64][128] (read until R5)
    static constexpr uint32_t OH = OE + 16384;     // H^T [128][128]; later dPhat, dM, Y, dG [64][64]
    static constexpr uint32_t ODH = OH + 32768;    // dH'^T [128][128]; after R1 dE and the dv staging [64][128]
    static constexpr uint32_t OM = ODH + 32768;    // M [64][64]
    static constexpr uint32_t OP = OM + 8192;      // P [64][64]
    static constexpr uint32_t ODE = OP + 8192;     // dPhat [64][64] (R0 to R3); Comba-pk: dp staging [64][128]
    static constexpr uint32_t OF = ODE + 16384;    // fp32: 8 x 64 per-row vectors, row and column partials, reduction
    static constexpr uint32_t NF = 8 * 64 + 8 * kQ * 64 + 2 * 4 * 64 + 16;
    static constexpr uint32_t NX = 5 * 64 + 4;     // fp32: the next unit's scalars, copied in a unit ahead,
                                                   // and the current unit's b
    static constexpr size_t bytes() { return 1024 + OF + (NF + NX) * 4; }
};

// Row-major [64][128] bf16 staging with 16-byte chunks rotated by row (conflict-free fragment
// writes), and its coalesced copy of rows < L to a strided global matrix.
template <int NT>
__device__ __forceinline__ void frag_stage(uint8_t* st, int m0, int n0, const float (&acc)[NT][4]) {
    const int r = frag_mrow(m0);
#pragma unroll
    for (int t = 0; t < NT; t += 2)
        stsm_x4(st + r * 256 + ((((frag_mcol(n0, t) >> 3) + r) & 15) << 4), pack_bf2(acc[t][0], acc[t][1]),
                pack_bf2(acc[t][2], acc[t][3]), pack_bf2(acc[t + 1][0], acc[t + 1][1]),
                pack_bf2(acc[t + 1][2], acc[t + 1][3]));
}
// Bulk tensor store of a [64][64-column] swizzled tile to (columns x, head y, tokens z ..).
__device__ __forceinline__ void tma_store_rows(const void* tmap, int x, int y, int z, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];\n"
                 ::"l"(tmap), "r"(x), "r"(y), "r"(z), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit_rows() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_rows_read() { asm volatile("cp.async.bulk.wait_group.read 0;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_rows_done() { asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory"); }

// 4-byte global->shared copy that bypasses registers; zero-filled when `valid` is false.
__device__ __forceinline__ void cp_async4(float* s, const float* g, bool valid) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(smem_u32(s)), "l"(g), "r"(valid ? 4 : 0)
                 : "memory");
}

// Named barrier 1: the two tail warps only.
__device__ __forceinline__ void tail_sync() { asm volatile("bar.sync 1, 64;\n" ::: "memory"); }

__device__ __forceinline__ void copy_stage_rows(bf16* g, long long ld, const uint8_t* st, int L, int tid) {
    for (int e = tid; e < L * 16; e += kLocalThreads) {
        const int r = e >> 4, ch = e & 15;
        *reinterpret_cast<uint4*>(g + r * ld + ch * 8) =
            *reinterpret_cast<const uint4*>(st + r * 256 + (((ch + r) & 15) << 4));
    }
}

template <int NT>
__device__ __forceinline__ void rowdot(const float (&acc)[NT][4], float& s0, float& s1) {
    s0 = 0.f;
    s1 = 0.f;
#pragma unroll
    for (int t = 0; t < NT; ++t) {
        s0 += acc[t][0] + acc[t][1];
        s1 += acc[t][2] + acc[t][3];
    }
    s0 = quad_sum(s0);
    s1 = quad_sum(s1);
}

struct UnitRef {
    long long idx, t0;   // (slot, head) unit index, first token
    int L, h;
};
// (unit indices fit 32 bits: the launcher checks slots x heads; 64-bit division would cost the
// loop head several hundred cycles)
__device__ __forceinline__ UnitRef unit_ref(const ChunkParams& p, long long u) {
    const uint32_t uu = (uint32_t)u, hh = (uint32_t)p.H;
    const uint32_t slot = uu / hh;
    const SlotInfo si = p.slot_info[slot];
    return {u, si.start, si.len, (int)(uu - slot * hh)};
}

// Persistent: CTA b handles units b, b + G, b + 2G, ... (G = gridDim.x, about one CTA per SM).
// While unit u computes, the tiles of unit u + G stream into buffers as soon as their last
// reader in unit u has finished (M after R3, H^T after R4, E, dH'^T, dO and Q/K (into the second
// of two alternating tiles, which holds M^T dE until then) after R5, V after R6; the per-row and
// per-head scalars by asynchronous copies after R3), so the loads of consecutive units overlap the
// tensor-core and epilogue work instead of every SM loading at the same moment.  Once R1 has read
// the dH'^T tile it holds dE (until R3) and the dv staging.
//
// PK: Comba-pk feedback vectors P (p.p, shaped like K).  They replace K as the Gram's left factor
// (P K^T, formed in R5 here), in W = M Diag(btilde gamma_{-1}) P and in the correction q - d p
// (applied to q before the chunk kernels, which see d = 0): the W path and the Gram's left factor
// go to dp instead of dk (dp = dG K + Diag(btilde gamma_{-1}) M^T dW - d dq, finished from TMEM
// at the end), dk takes dG^T P, and the row dots of dd and of the W path take p.  The P tile
// lives over the M and P-matrix tiles from R3 to R6; the next unit's M then loads after R6.
// Tensor maps of the kernel's TMA traffic (128-byte swizzle, 64-column boxes): the dq, dk, dp
// stores and every tile load.  Token tensors [tokens][heads][128] take {64, 1, 64} boxes; the
// workspace tiles are 2D views [units * rows][cols] with boxes of a tile's rows.
struct LocalMaps {
    CUtensorMap dq, dk, dp;           // stores
    CUtensorMap q, k, p, v, dO;       // token tiles (q, k, p per key head; v, dO per value head)
    CUtensorMap e, h, dh, m;          // workspace: E [64][128], H^T, dH'^T [128][128], M [64][64]
};

template <bool PK>
__global__ void __launch_bounds__(kLocalThreads, 1)
    k_bwd_local_tc(ChunkParams p, long long units, const __grid_constant__ LocalMaps mp) {
    using S = LocalTcSmem;
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t bar, bar0, stall_bar;   // bar0: R0; stall_bar: nothing arrives (COMBA_DIAG_STALL)
    // TMA arrival: ldn[0..3] a unit's tiles, in the four groups the previous unit prefetches them in
    // (M; H^T; E, dH'^T, dO, Q/K; V, and with Comba-pk M), ldp its P (Comba-pk).  Each completes
    // one phase per unit that has rows.
    __shared__ uint64_t ldn[4], ldp;
    __shared__ uint32_t tbase;
    __shared__ int2 s_nslot;   // (start, length) of the unit after next, loaded during the tail
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wr = warp & 3, wc = warp >> 2, m0 = 16 * wr;
    uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sV = sm + S::OV;
    uint8_t* sdO = sm + S::ODO;
    uint8_t* sE = sm + S::OE;
    uint8_t* sHt = sm + S::OH;
    uint8_t* sdHt = sm + S::ODH;
    uint8_t* sM = sm + S::OM;
    uint8_t* sP = sm + S::OP;
    uint8_t* sdE = sm + S::ODE;
    uint8_t* sdPh = sdE;              // dPhat [64][64], from R0's epilogue until R3
    uint8_t* sdEt = sdHt;             // dE [64][128], after R1 (dH'^T's readers) until R3
    uint8_t* stV = sdHt + 16384;      // dv staging, after R3 (E itself is read once more, by R5)
    uint8_t* sdG = sV + 8192;         // dG [64][64], after R3 until R6
    uint8_t* sPf = sM;                // Comba-pk: P [64][128] over the M and P-matrix tiles, R3 to R6
    uint8_t* stP = sdE;               // Comba-pk: dp staging, at the end (dPhat is dead)
    float* sG = reinterpret_cast<float*>(sm + S::OF);
    float* sGm1 = sG + 64;
    float* sBe = sG + 128;
    float* sBt = sG + 192;
    float* sAl = sG + 256;
    float* sDg = sG + 320;
    float* sEm1 = sG + 384;           // gamma_{r-1}
    float* sWs = sG + 448;            // btilde_r gamma_{r-1}
    float* rowp = sG + 512;           // [kind][column quarter][row]
    float* colp = rowp + 8 * kQ * 64;  // [kind][row block][column]
    float* red = colp + 2 * 4 * 64;
    const uint32_t udO = smem_u32(sdO), uE = smem_u32(sE), uH = smem_u32(sHt), udH = smem_u32(sdHt),
                   uM = smem_u32(sM), uP = smem_u32(sP), udE = smem_u32(sdEt), udPh = smem_u32(sdPh),
                   udG = smem_u32(sdG), uPf = smem_u32(sPf);

    const int Hk = p.H / p.vg;   // key heads: q, k, alpha, beta, b, d of value head h are key head h / vg's
    // TMA issue (thread kTma).  Q rows 0-63 and K rows 64-127 of a 128-row tile: K halves 16 KB apart.
    constexpr int kTma = 32;
    auto tma_qk = [&](uint8_t* dst, const UnitRef& x, uint32_t mb) {
        const int hk = x.h / p.vg, t0x = (int)x.t0;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            tma_load_3d(smem_u32(dst) + half * 16384, &mp.q, 64 * half, hk, t0x, mb);
            tma_load_3d(smem_u32(dst) + 8192 + half * 16384, &mp.k, 64 * half, hk, t0x, mb);
        }
    };
    auto tma_tok = [&](uint8_t* dst, const CUtensorMap* m, int head, const UnitRef& x, uint32_t mb) {
#pragma unroll
        for (int half = 0; half < 2; ++half) tma_load_3d(smem_u32(dst) + half * 8192, m, 64 * half, head, (int)x.t0, mb);
    };
    auto tma_e = [&](const UnitRef& x, uint32_t mb) {
#pragma unroll
        for (int half = 0; half < 2; ++half) tma_load_2d(smem_u32(sE) + half * 8192, &mp.e, 64 * half, (int)(x.idx * 64), mb);
    };
    auto tma_sq = [&](uint8_t* dst, const CUtensorMap* m, const UnitRef& x, uint32_t mb) {   // H^T or dH'^T
#pragma unroll
        for (int half = 0; half < 2; ++half) tma_load_2d(smem_u32(dst) + half * 16384, m, 64 * half, (int)(x.idx * 128), mb);
    };
    auto tma_m = [&](const UnitRef& x, uint32_t mb) { tma_load_2d(smem_u32(sM), &mp.m, 0, (int)(x.idx * 64), mb); };
    // a unit's four tile groups (phase completions of ldn[0..3])
    auto issue_n0 = [&](const UnitRef& x, bool m_here) {
        const uint32_t mb = smem_u32(&ldn[0]);
        mbar_expect_tx(mb, m_here ? 8192u : 0u);
        if (m_here) tma_m(x, mb);
    };
    auto issue_n1 = [&](const UnitRef& x) {
        const uint32_t mb = smem_u32(&ldn[1]);
        mbar_expect_tx(mb, 32768u);
        tma_sq(sHt, &mp.h, x, mb);
    };
    auto issue_n2 = [&](uint8_t* qk, const UnitRef& x) {
        const uint32_t mb = smem_u32(&ldn[2]);
        mbar_expect_tx(mb, 16384u + 32768u + 16384u + 32768u);
        tma_e(x, mb);
        tma_sq(sdHt, &mp.dh, x, mb);
        tma_tok(sdO, &mp.dO, x.h, x, mb);
        tma_qk(qk, x, mb);
    };
    auto issue_n3 = [&](const UnitRef& x, bool m_here) {
        const uint32_t mb = smem_u32(&ldn[3]);
        mbar_expect_tx(mb, 16384u + (m_here ? 8192u : 0u));
        tma_tok(sV, &mp.v, x.h, x, mb);
        if (m_here) tma_m(x, mb);
    };
    // rows L..63 of a token tile hold the next sequence's tokens (or the zero fill past the tensor):
    // zeroed by all threads after the tile has landed (a sequence's last chunk only)
    auto zero_rows = [&](uint8_t* t, int rows, int L) {
        for (int e = tid; e < (64 - L) * 16; e += kLocalThreads) {
            const int r = L + (e >> 4), ch = e & 15;
            *reinterpret_cast<uint4*>(t + sw128_offset(r, 8 * ch, rows)) = make_uint4(0, 0, 0, 0);
        }
    };
    uint32_t pend = 0;   // thread kTma: barriers with loads issued and not yet waited on (bit i: ldn[i],
                         // 5: ldp), drained on the give-up path
    // A unit's scalars, copied into sNx a unit ahead (asynchronous 4-byte copies, which hold no
    // registers and wait behind no tile traffic): per row r (thread r < 64) the log-decays G_r and
    // G_{r-1}, beta, alpha and b; per head (thread 0) d and, with Comba-pk, the feedback d.
    float* sNx = sG + S::NF;
    auto issue_rows = [&](const UnitRef& x) {
        const int hk = x.h / p.vg;
        if (tid < 64) {
            const float* gb = p.Gb + x.idx * 64;
            cp_async4(sNx + tid, gb + tid, true);
            cp_async4(sNx + 64 + tid, gb + (tid > 0 ? tid - 1 : 0), tid > 0);
            cp_async4(sNx + 128 + tid, p.beta + (x.t0 + (tid < x.L ? tid : 0)) * Hk + hk, tid < x.L);
            cp_async4(sNx + 192 + tid, p.alpha + (x.t0 + (tid < x.L ? tid : 0)) * Hk + hk, tid < x.L);
            cp_async4(sNx + 256 + tid, p.b ? p.b + hk : p.d + hk, p.b != nullptr);
        }
        if (tid == 0) {
            cp_async4(sNx + 320, p.d + hk, true);
            cp_async4(sNx + 321, PK ? p.d_fb + hk : p.d + hk, PK);
        }
        cp_async_commit();
    };
    if (tid == 0) {
        mbar_init(smem_u32(&bar), 1);
        mbar_init(smem_u32(&bar0), 1);
        mbar_init(smem_u32(&stall_bar), 1);
        for (int i = 0; i < 4; ++i) mbar_init(smem_u32(&ldn[i]), 1);
        mbar_init(smem_u32(&ldp), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tbase), 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tbase;
    const uint32_t tq = tmem + ((uint32_t)(32 * wr) << 16);   // this warp's TMEM lanes
    MmaSync ms{smem_u32(&bar), smem_u32(p.stall ? &stall_bar : &bar), 0, p.wait_ns};
    // A round's wait: every thread on the commit's mbarrier, `ok` made uniform over the warp (warp-
    // collective TMEM and fragment instructions follow) and over the block at the next block-wide
    // barrier, which every round reaches before its next product is issued.
    auto mma_wait = [&]() { return ms.wait_warp(); };
    uint32_t ph0 = 0;   // phase of bar0 (R0, one commit per unit)
    const int nl0 = 8 * NL * wc, nk0 = 8 * NK * wc;   // this warp's columns of 64- and 128-wide results
    const int ra = m0 + frag_row(0), rb = m0 + frag_row(2);   // this lane's two rows
    auto put_rows = [&](int kind, float s0, float s1) {
        if ((lane & 3) == 0) { rowp[(kind * kQ + wc) * 64 + ra] = s0; rowp[(kind * kQ + wc) * 64 + rb] = s1; }
    };
    // row dot of a 128-wide fragment tile with the bf16 tile `t` (rows r at row offset roff)
    auto tile_rowdot = [&](const float (&acc)[NK][4], const uint8_t* t, int rows, int roff, float& s0, float& s1) {
        uint32_t w[2 * NK];
        frag_load_sw<NK>(t, rows, roff + m0, nk0, w);
        float prod[NK][4];
#pragma unroll
        for (int j = 0; j < NK; ++j)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh) {
                const float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[2 * j + hh]));
                prod[j][2 * hh] = acc[j][2 * hh] * v.x;
                prod[j][2 * hh + 1] = acc[j][2 * hh + 1] * v.y;
            }
        rowdot(prod, s0, s1);
    };

    bool ok = true;
    bool pre = false;   // this unit's tiles and row scalars were requested by the previous unit
    uint32_t lph = 0;   // phase parity of the TMA barriers for the current unit
    bool early = false; // thread 0: this unit's dP and R1 products were issued during the previous unit's tail
    long long u = blockIdx.x;
    UnitRef cur = u < units ? unit_ref(p, u) : UnitRef{0, 0, 0, 0};
    bool nslot = false;   // s_nslot holds the slot of unit u + G (the previous unit's tail loaded it)
    for (int it = 0; u < units && ok; ++it) {
        const long long un = u + gridDim.x;
        UnitRef nxt{0, 0, 0, 0};
        if (un < units) {   // used from the first prefetch point on
            if (nslot) {
                const int2 sl = s_nslot;
                nxt = UnitRef{un, sl.x, sl.y, (int)((uint32_t)un % (uint32_t)p.H)};
            } else {
                nxt = unit_ref(p, un);
            }
        }
        uint8_t* sQK = sm + S::OQK + (it & 1) * 32768;
        uint8_t* sQKn = sm + S::OQK + ((it + 1) & 1) * 32768;   // the next unit's Q/K tile
        if (cur.L <= 0) {
            if (tid == 0) { p.part[u * 2] = 0.f; p.part[u * 2 + 1] = 0.f; }
            pre = false;
            nslot = false;
            u = un;
            cur = nxt;
            continue;
        }
        uint8_t* sKt = sQK + 64 * 128;   // K: rows 64-127 of the 128-row tile
        const uint32_t uQK = smem_u32(sQK), uK = smem_u32(sKt);
        // M^T dE [64][128] (after R3 until R5) in the other Q/K tile, which takes the next unit's
        // Q and K only after R5
        uint8_t* sMdE = sQKn;
        const uint32_t uMdE = smem_u32(sMdE);
        const bool has_next = nxt.L > 0;
        const int L = cur.L, h = cur.h;
        const long long t0 = cur.t0, idx = cur.idx;

        if (!pre) {
            // a bulk store of dq, dk two units back may still read this tile
            if (tid == 0) bulk_wait_rows_read();
            __syncthreads();
            if (tid == kTma) {
                issue_n0(cur, true);
                issue_n1(cur);
                issue_n2(sQK, cur);
                issue_n3(cur, false);
                pend |= 15u;
            }
            issue_rows(cur);
        }
        cp_async_wait<0>();   // this thread's copies of the unit's scalars
        const float bh = tid < 64 ? (p.b ? sNx[256 + tid] : 1.f) : 1.f;
        if (tid < 64) {
            const float g = sNx[tid], gm1 = sNx[64 + tid], be = sNx[128 + tid];
            const float al = tid < L ? sNx[192 + tid] : 1.f;
            sG[tid] = g;
            sGm1[tid] = gm1;
            sBe[tid] = be;
            const float fsc = feedback_scale(p.iplr, al);
            sBt[tid] = bh * be * fsc;
            sAl[tid] = al;
            const float em1 = tid > 0 ? __expf(gm1) : 1.f;
            sEm1[tid] = em1;
            sWs[tid] = bh * be * fsc * em1;
            if (tid == 0) sNx[322] = bh;   // the unit's b for the tail (the next unit's copies miss this slot)
        }
        // the unit's tiles have landed (all four groups)
        {
            bool okl = true;
#pragma unroll
            for (int i = 0; i < 4; ++i) okl = mbar_wait_polls(smem_u32(&ldn[i]), lph, p.wait_ns) && okl;
            if (okl && tid == kTma) pend &= ~15u;
            ok = !__syncthreads_or(!okl);
            if (!ok) {   // give up on the unit: let its copies finish before leaving
                if (tid == kTma) {
                    for (int i = 0; i < 4; ++i)
                        if (pend & (1u << i)) mbar_drain(smem_u32(&ldn[i]), lph);
                    pend = 0;
                }
                if (tid == 0) {
                    if (early) {   // products issued ahead for this unit: track and drain them
                        tc_commit(smem_u32(&bar0));
                        mbar_drain(smem_u32(&bar0), ph0);
                    }
                    flag_error(p);
                }
                break;
            }
        }
        const float dh = sNx[320];                // thread 0's copies, published by the barrier above
        const float dfb = PK ? sNx[321] : 0.f;
        // rows past a short chunk: zero in Q, K, dO and V (Q~ below covers rows < L only)
        if (L < kChunk) {
            zero_rows(sQK, 128, L);
            zero_rows(sQK + 64 * 128, 128, L);
            zero_rows(sdO, 64, L);
            zero_rows(sV, 64, L);
        }
        // Q~ = Q - d K (rows < L)
        for (int e = tid; e < L * 16; e += kLocalThreads) {
            const int r = e >> 4, ch = e & 15;
            uint4* qa = reinterpret_cast<uint4*>(sQK + sw128_offset(r, 8 * ch, 128));
            const uint4 ka = *reinterpret_cast<const uint4*>(sQK + sw128_offset(64 + r, 8 * ch, 128));
            float qv[8], kv[8];
            unpack8(*qa, qv);
            unpack8(ka, kv);
#pragma unroll
            for (int i = 0; i < 8; ++i) qv[i] -= dh * kv[i];
            *qa = pack8(qv);
        }
        // the other Q/K tile (M^T dE from R3 on, then the next unit's Q/K) may still be the source
        // of the previous unit's bulk dq, dk stores
        if (tid == 0) bulk_wait_rows_read();
        publish_smem();

        const float gL = sG[L - 1];
        const float eGa = __expf(sG[ra]), eGb = __expf(sG[rb]);
        const float sKa = ra < L ? __expf(gL - sG[ra]) : 0.f, sKb = rb < L ? __expf(gL - sG[rb]) : 0.f;

        // ---------------- R0: S = Q~ K^T, dP = dO E^T (own barrier), and right behind them R1: dO H^T,
        // E dH'^T, K dH', so that the tensor core runs R1 while the warps form P from R0
        if (tid == 0) {
            tc_gemm_m64<false, false>(tmem + 0, uQK, 128, uK, 128, 64, D, false);      // S = Q~ K^T
            if (!early) tc_gemm_m64<false, false>(tmem + 64, udO, 64, uE, 64, 64, D, false);   // dP = dO E^T
            tc_commit(smem_u32(&bar0));   // (with products issued ahead, it covers those too)
            if (!early) {
                tc_gemm_m64<false, true>(tmem + 128, udO, 64, uH, 128, 128, D, false);     // dO H^T
                tc_gemm_m64<false, true>(tmem + 256, uE, 64, udH, 128, 128, D, false);     // E dH'^T
                tc_gemm_m64<false, false>(tmem + 384, uK, 128, udH, 128, 128, D, false);   // K dH'
            }
        }
        // While R0 runs: <H, dH'> (R1 reads the same two tiles; both only read them)
        {
            // the two tiles share one layout, so matching 16-byte chunks pair up
            float sacc = 0.f;
            for (int e = tid; e < 128 * 16; e += kLocalThreads) {
                float hv[8], gv[8];
                unpack8(reinterpret_cast<const uint4*>(sHt)[e], hv);
                unpack8(reinterpret_cast<const uint4*>(sdHt)[e], gv);
#pragma unroll
                for (int i = 0; i < 8; ++i) sacc = fmaf(hv[i], gv[i], sacc);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sacc += __shfl_xor_sync(0xffffffffu, sacc, o);
            if (lane == 0) red[warp] = sacc;
        }
        float acc_dq[NK][4], acc_dk[NK][4];
        {
            const bool ok0 = mbar_wait_polls(smem_u32(&bar0), ph0, p.wait_ns);
            ph0 ^= 1;
            ok = __all_sync(0xffffffffu, ok0);
            tc_fence_after();
        }
        // Each epilogue below first forms what the next round reads (P, dE, M^T dE, M^T dW, dG),
        // publishes it and lets thread 0 issue that round, then does the rest of its work (row and
        // column partials, dv, the dq / dk parts) while the tensor core runs.
        float sc[NL][4], ph[NL][4];
        if (ok) {
            // P = Tril(S * Gamma) (the R2 operand) and dPhat = dP * Gamma (an R3 operand); S and dP
            // arrive with one wait
            uint32_t rS[NL * 4], rP[NL * 4];
            tmem_issue<NL>(tq + 0 + nl0, rS);
            tmem_issue<NL>(tq + 64 + nl0, rP);
            tmem_wait();
            tmem_take<NL>(rS, sc);
            tmem_take<NL>(rP, ph);
            float pv[NL][4];
#pragma unroll
            for (int t = 0; t < NL; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = m0 + frag_row(i), c = nl0 + frag_col(t, i);
                    const float gam = (c <= r && r < L) ? __expf(sG[r] - sG[c]) : 0.f;
                    pv[t][i] = sc[t][i] * gam;
                    ph[t][i] *= gam;
                }
            frag_store_sw<NL>(sP, 64, m0, nl0, pv);
            frag_store_sw<NL>(sdPh, 64, m0, nl0, ph);
        }
        ok = publish_ok(ok);

        // ---------------- R2: P^T dO (dE = Kbar dH' + P^T dO) into the S and dP columns (read), behind
        // R1; one commit covers both.  The commit is made even when R0's wait gave up, so that the
        // give-up path finds R1 tracked on this barrier.
        if (tid == 0) {
            if (ok) tc_gemm_m64<true, true>(tmem + 0, uP, 64, udO, 64, 128, 64, false);
            tc_commit(smem_u32(&bar));
        }
        if (ok) {
            // dP * P = dPhat * S into the log-decay gradient; the diagonal's decay factor is exactly
            // 1 (no g-dependence), so it is left out rather than added and cancelled
            float rs0 = 0.f, rs1 = 0.f;
            float cs[NL][2];
#pragma unroll
            for (int t = 0; t < NL; ++t) {
                cs[t][0] = cs[t][1] = 0.f;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = m0 + frag_row(i), c = nl0 + frag_col(t, i);
                    const float w = c < r ? ph[t][i] * sc[t][i] : 0.f;
                    if (i < 2) rs0 += w; else rs1 += w;
                    cs[t][i & 1] += w;
                }
            }
            rs0 = quad_sum(rs0);
            rs1 = quad_sum(rs1);
            put_rows(3, rs0, rs1);
#pragma unroll
            for (int t = 0; t < NL; ++t)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const float v = col_sum8(cs[t][e]);
                    if ((lane >> 2) == 0) colp[(0 * 4 + wr) * 64 + nl0 + 8 * t + 2 * (lane & 3) + e] = v;
                }
        }
        {
            const bool ok2 = mma_wait();
            ok = ok && ok2;
        }
        if (ok) {
            // dE = Kbar dH' + P^T dO (over the dead dH'^T tile: an R3 operand)
            float de[NK][4], t2[NK][4];
            uint32_t re[NK * 4], rt[NK * 4];
            tmem_issue<NK>(tq + 384 + nk0, re);
            tmem_issue<NK>(tq + 0 + nk0, rt);
            tmem_wait();
            tmem_take<NK>(re, de);
            tmem_take<NK>(rt, t2);
#pragma unroll
            for (int t = 0; t < NK; ++t) {
                de[t][0] = fmaf(de[t][0], sKa, t2[t][0]); de[t][1] = fmaf(de[t][1], sKa, t2[t][1]);
                de[t][2] = fmaf(de[t][2], sKb, t2[t][2]); de[t][3] = fmaf(de[t][3], sKb, t2[t][3]);
            }
            frag_store_sw<NK>(sdEt, 64, m0, nk0, de);
        }
        ok = publish_ok(ok);

        // ---------------- R3: M^T dE, dPhat^T Q~ (into the columns dE was read from)
        if (tid == 0) {
            if (ok) {
                tc_gemm_m64<true, true>(tmem + 0, uM, 64, udE, 64, 128, 64, false);        // M^T dE
                tc_gemm_m64<true, true>(tmem + 384, udPh, 64, uQK, 128, 128, 64, false);   // dPhat^T Q~
            }
            tc_commit(smem_u32(&bar));
        }
        if (ok) {
            // the other two R1 products: dQ~ part Diag(gamma) dO H^T and dK from Kbar,
            // Diag(gamma_C / gamma_r) E dH'^T, with their row dots with Q~ and with K (used by the
            // per-position tail only)
            uint32_t rq[NK * 4], rk[NK * 4];
            tmem_issue<NK>(tq + 128 + nk0, rq);
            tmem_issue<NK>(tq + 256 + nk0, rk);
            tmem_wait();
            tmem_take<NK>(rq, acc_dq);
            tmem_take<NK>(rk, acc_dk);
#pragma unroll
            for (int t = 0; t < NK; ++t) {
                acc_dq[t][0] *= eGa; acc_dq[t][1] *= eGa; acc_dq[t][2] *= eGb; acc_dq[t][3] *= eGb;
                acc_dk[t][0] *= sKa; acc_dk[t][1] *= sKa; acc_dk[t][2] *= sKb; acc_dk[t][3] *= sKb;
            }
            float s0, s1;
            tile_rowdot(acc_dq, sQK, 128, 0, s0, s1);
            put_rows(0, s0, s1);
            tile_rowdot(acc_dk, sQK, 128, 64, s0, s1);
            put_rows(1, s0, s1);
        }
        {
            const bool ok3 = mma_wait();
            ok = ok && ok3;
        }
        if (ok && tid == kTma) {
            if constexpr (PK) {
                // this unit's P over M (its last reader was R3) and the P matrix; the next unit's M
                // comes after R6
                const uint32_t mb = smem_u32(&ldp);
                mbar_expect_tx(mb, 16384u);
                tma_tok(sPf, &mp.p, h / p.vg, cur, mb);
                pend |= 32u;
            }
            if (has_next) { issue_n0(nxt, !PK); pend |= 1u; }   // M's last reader was R3
        }
        if (ok && has_next) issue_rows(nxt);   // sNx was last read at this unit's start
        if (ok) {
            // M^T dE, unscaled and in bf16, over the dead dE tile: the R4 / R5 operand; and
            // dV = Diag(beta) M^T dE staged over the dead E tile, direct dbeta = v . (M^T dE)
            float t3[NK][4], s0, s1;
            tmem_frag<NK>(tq + 0 + nk0, t3);
            frag_store_sw<NK>(sMdE, 64, m0, nk0, t3);
            tile_rowdot(t3, sV, 64, 0, s0, s1);
            put_rows(2, s0, s1);
            const float ba = sBe[ra], bb = sBe[rb];
#pragma unroll
            for (int t = 0; t < NK; ++t) { t3[t][0] *= ba; t3[t][1] *= ba; t3[t][2] *= bb; t3[t][3] *= bb; }
            frag_stage<NK>(stV, m0, nk0, t3);
        }
        ok = publish_ok(ok);

        // ---------------- R4: (M^T dE) H^T = -M^T dW (dW = -dE H^T) into M^T dE's columns (read), and
        // K K^T, dPhat K into the columns of the two R1 products read above
        if (tid == 0) {
            if (ok) {
                tc_gemm_m64<false, true>(tmem + 0, uMdE, 64, uH, 128, 128, D, false);
                if constexpr (!PK) tc_gemm_m64<false, false>(tmem + 128, uK, 128, uK, 128, 64, D, false);   // K K^T
                tc_gemm_m64<false, true>(tmem + 256, udPh, 64, uK, 128, 128, 64, false);   // dPhat K
            }
            tc_commit(smem_u32(&bar));
        }
        if (ok) copy_stage_rows((bf16*)p.dvv + (t0 * p.H + h) * D, (long long)p.H * D, stV, L, tid);   // dv rows
        {
            const bool ok4 = mma_wait();
            ok = ok && ok4;
        }
        if (ok && has_next && tid == kTma) { issue_n1(nxt); pend |= 2u; }   // R4 was H^T's last reader
        float t4[NK][4];
        if (ok) {
            // M^T dW = -(M^T dE) H^T, for dk (the W path) and its row dots
            tmem_frag<NK>(tq + 0 + nk0, t4);
#pragma unroll
            for (int t = 0; t < NK; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) t4[t][i] = -t4[t][i];
        }
        // every thread's dv rows are copied (the next unit's dH'^T loads over their staging after R5),
        // and with Comba-pk P has landed (its rows past a short chunk zeroed)
        {
            bool okl = ok;
            if constexpr (PK) okl = okl && mbar_wait_polls(smem_u32(&ldp), lph, p.wait_ns);
            if (okl && tid == kTma) pend &= ~32u;
            if constexpr (PK)
                if (okl && L < kChunk) zero_rows(sPf, 64, L);
            fence_async_smem();
            tc_fence_before();
            ok = !__syncthreads_or(!okl);   // okl is false wherever ok is
            tc_fence_after();
        }

        // ---------------- R5: M^T dM M^T = (M^T dE) E^T.  With dM = dE (Diag(beta) V)^T + dW (Diag(btilde
        // gamma_{-1}) K)^T, U = M Diag(beta) V and W = M Diag(btilde gamma_{-1}) K it is (M^T dE) U^T +
        // (M^T dW) W^T, and dW = -dE H^T turns the second term into -(M^T dE) (W H)^T; E = U - W H.
        if (tid == 0) {
            if (ok) {
                tc_gemm_m64<false, false>(tmem + 192, uMdE, 64, uE, 64, 64, D, false);
                if constexpr (PK) tc_gemm_m64<false, false>(tmem + 128, uPf, 64, uK, 128, 64, D, false);   // P K^T
            }
            tc_commit(smem_u32(&bar));
        }
        if (ok) {
            // W path: M^T dW scaled by btilde gamma_{r-1} goes to dk; its row dot with k feeds dbtilde
            // and d g_{r-1}
            float s0, s1;
            if constexpr (PK) {
                tile_rowdot(t4, sPf, 64, 0, s0, s1);   // with p; M^T dW stays in TMEM for dp
            } else {
                tile_rowdot(t4, sQK, 128, 64, s0, s1);
                const float wa = sWs[ra], wb = sWs[rb];
#pragma unroll
                for (int t = 0; t < NK; ++t) {
                    acc_dk[t][0] += wa * t4[t][0]; acc_dk[t][1] += wa * t4[t][1];
                    acc_dk[t][2] += wb * t4[t][2]; acc_dk[t][3] += wb * t4[t][3];
                }
            }
            put_rows(7, s0, s1);
            // dq = dQ~ complete (dPhat K from R4): dd partial = -k . dQ~ ; dk -= d dQ~
            tmem_frag<NK>(tq + 256 + nk0, t4);
#pragma unroll
            for (int t = 0; t < NK; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    acc_dq[t][i] += t4[t][i];
                    if constexpr (!PK) acc_dk[t][i] -= dh * acc_dq[t][i];
                }
            if constexpr (PK) tile_rowdot(acc_dq, sPf, 64, 0, s0, s1);   // dd = -p . dq
            else tile_rowdot(acc_dq, sQK, 128, 64, s0, s1);
            put_rows(6, s0, s1);
        }
        {
            const bool ok5 = mma_wait();
            ok = ok && ok5;
        }
        // the next unit's E (R5 was its last reader), dH'^T (dE and the dv rows staged over it are
        // dead: the rows were copied before R4's wait), dO and Q/K (M^T dE is dead; the previous
        // unit's dq, dk stores have read this tile: the prologue waited for them)
        if (ok && has_next && tid == kTma) { issue_n2(sQKn, nxt); pend |= 4u; }
        if (ok) {
            // dA = -(M^T dM M^T) on the strict lower triangle -> dG (the R6 operand)
            float dA[NL][4];
            tmem_frag<NL>(tq + 192 + nl0, dA);
            float g4[NL][4];
#pragma unroll
            for (int t = 0; t < NL; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = m0 + frag_row(i), c = nl0 + frag_col(t, i);
                    const bool strict = c < r && r < L;
                    const float gm = strict ? __expf(sGm1[r] - sG[c]) : 0.f;
                    g4[t][i] = -dA[t][i] * sBt[r] * gm;
                }
            frag_store_sw<NL>(sdG, 64, m0, nl0, g4);
        }
        ok = publish_ok(ok);

        // ---------------- R6: dK += dPhat^T Q~ (already in TMEM) + dG K + dG^T K; with Comba-pk dG K is
        // dp's (into the dPhat K columns, read) and dk takes dG^T P
        if (tid == 0) {
            if (ok) {
                if constexpr (PK) {
                    tc_gemm_m64<false, true>(tmem + 256, udG, 64, uK, 128, 128, 64, false);
                    tc_gemm_m64<true, true>(tmem + 384, udG, 64, uPf, 64, 128, 64, true);
                } else {
                    tc_gemm_m64<false, true>(tmem + 384, udG, 64, uK, 128, 128, 64, true);
                    tc_gemm_m64<true, true>(tmem + 384, udG, 64, uK, 128, 128, 64, true);
                }
            }
            tc_commit(smem_u32(&bar));
        }
        if (ok) {
            // the R5 epilogue's partials, from dA and K K^T read again (R6 writes neither's
            // columns): dA * Gram into dbtilde_r, dA * Aval into the log-decay gradient (on the
            // first sub-diagonal the decay factor gamma_{r-1}/gamma_c is exactly 1, so it is left
            // out: it would cancel)
            float dA[NL][4], gr[NL][4];
            {
                uint32_t ra_[NL * 4], rg[NL * 4];
                tmem_issue<NL>(tq + 192 + nl0, ra_);
                tmem_issue<NL>(tq + 128 + nl0, rg);
                tmem_wait();
                tmem_take<NL>(ra_, dA);
                tmem_take<NL>(rg, gr);
            }
            float rb0 = 0.f, rb1 = 0.f, ra0 = 0.f, ra1 = 0.f;
            float cs[NL][2];
#pragma unroll
            for (int t = 0; t < NL; ++t) {
                cs[t][0] = cs[t][1] = 0.f;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int r = m0 + frag_row(i), c = nl0 + frag_col(t, i);
                    const bool strict = c < r && r < L;
                    const float gm = strict ? __expf(sGm1[r] - sG[c]) : 0.f;
                    const float uu = -dA[t][i] * gm * gr[t][i];   // contributes to dbtilde_r
                    const float w = c + 1 < r ? uu * sBt[r] : 0.f;
                    if (i < 2) { rb0 += uu; ra0 += w; } else { rb1 += uu; ra1 += w; }
                    cs[t][i & 1] += w;
                }
            }
            rb0 = quad_sum(rb0); rb1 = quad_sum(rb1);
            ra0 = quad_sum(ra0); ra1 = quad_sum(ra1);
            put_rows(4, rb0, rb1);
            put_rows(5, ra0, ra1);
#pragma unroll
            for (int t = 0; t < NL; ++t)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const float v = col_sum8(cs[t][e]);
                    if ((lane >> 2) == 0) colp[(1 * 4 + wr) * 64 + nl0 + 8 * t + 2 * (lane & 3) + e] = v;
                }
        }
        {
            const bool ok6 = mma_wait();
            ok = ok && ok6;
        }
        if (ok && has_next) {
            if (tid == kTma) { issue_n3(nxt, PK); pend |= 8u; }   // dG (over V) is dead, and P (over M)
        }
        if (ok) {
            float t6[NK][4];
            tmem_frag<NK>(tq + 384 + nk0, t6);
#pragma unroll
            for (int t = 0; t < NK; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc_dk[t][i] += t6[t][i];
        }
        // dq, dk staged over the Q~/K tile: its last readers were R6 (complete for every warp that saw
        // the wait end) and the row dots of R5's epilogue (before the block-wide barrier ahead of R6)
        if (ok) {
            // a full chunk leaves by bulk tensor stores from swizzled tiles, which run behind the
            // per-position tail; a partial one by row copies (a 64-row box would pass its end)
            if (L == kChunk) {
                frag_store_sw<NK>(sQK, 64, m0, nk0, acc_dq);
                frag_store_sw<NK>(sQK + 16384, 64, m0, nk0, acc_dk);
            } else {
                frag_stage<NK>(sQK, m0, nk0, acc_dq);
                frag_stage<NK>(sQK + 16384, m0, nk0, acc_dk);
            }
            if constexpr (PK) {
                // dp = dG K + Diag(btilde gamma_{-1}) M^T dW - d dq, the first two still in TMEM (R4 left
                // (M^T dE) H^T = -M^T dW there)
                float dpv[NK][4], t7[NK][4];
                uint32_t rg[NK * 4], rw[NK * 4];
                tmem_issue<NK>(tq + 256 + nk0, rg);
                tmem_issue<NK>(tq + 0 + nk0, rw);
                tmem_wait();
                tmem_take<NK>(rg, dpv);
                tmem_take<NK>(rw, t7);
                const float wa = sWs[ra], wb = sWs[rb];
#pragma unroll
                for (int t = 0; t < NK; ++t)
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        dpv[t][i] -= (i < 2 ? wa : wb) * t7[t][i] + dfb * acc_dq[t][i];
                if (L == kChunk) frag_store_sw<NK>(stP, 64, m0, nk0, dpv);
                else frag_stage<NK>(stP, m0, nk0, dpv);
            }
        }
        if (L == kChunk) fence_async_smem();
        tc_fence_before();   // every TMEM read of this unit is done: the next unit's products may follow
        ok = !__syncthreads_or(!ok);
        tc_fence_after();
        if (ok) {
            if (L == kChunk) {
                if (tid == 0) {
#pragma unroll
                    for (int half = 0; half < 2; ++half) {
                        tma_store_rows(&mp.dq, 64 * half, h, (int)t0, smem_u32(sQK) + half * 8192);
                        tma_store_rows(&mp.dk, 64 * half, h, (int)t0, smem_u32(sQK + 16384) + half * 8192);
                        if constexpr (PK) tma_store_rows(&mp.dp, 64 * half, h, (int)t0, smem_u32(stP) + half * 8192);
                    }
                    bulk_commit_rows();
                }
            } else {
                const long long ld = (long long)p.H * D;
                copy_stage_rows((bf16*)p.dq + (t0 * p.H + h) * D, ld, sQK, L, tid);
                copy_stage_rows((bf16*)p.dkk + (t0 * p.H + h) * D, ld, sQK + 16384, L, tid);
                if constexpr (PK) copy_stage_rows((bf16*)p.dpp + (t0 * p.H + h) * D, ld, stP, L, tid);
            }
        }
        // The next unit's dP = dO E^T and R1 products (their tiles are in), issued while the tensor core
        // would idle through this unit's tail, which the last two warps run; warp 0 may wait here
        // for room in the tensor core's queue.  A short next chunk (rows to zero first) waits for its
        // own prologue.
        if (tid == 0) {
            early = false;
            if (ok && has_next && nxt.L == kChunk && mbar_wait_polls(smem_u32(&ldn[1]), lph ^ 1, p.wait_ns) &&
                mbar_wait_polls(smem_u32(&ldn[2]), lph ^ 1, p.wait_ns)) {
                const uint32_t uKn = smem_u32(sQKn) + 64 * 128;
                tc_gemm_m64<false, false>(tmem + 64, udO, 64, uE, 64, 64, D, false);       // dP = dO E^T
                tc_gemm_m64<false, true>(tmem + 128, udO, 64, uH, 128, 128, D, false);     // dO H^T
                tc_gemm_m64<false, true>(tmem + 256, uE, 64, udH, 128, 128, D, false);     // E dH'^T
                tc_gemm_m64<false, false>(tmem + 384, uKn, 128, udH, 128, 128, D, false);  // K dH'
                early = true;
            }
        }

        // ---------------- per-position scalars (rows 0..63, one thread each of the last two warps,
        // which meet alone at named barrier 1; the rest of the block goes on to the unit's end)
        auto rsum = [&](int kind, int r) {
            float v = 0.f;
#pragma unroll
            for (int j = 0; j < kQ; ++j) v += rowp[(kind * kQ + j) * 64 + r];
            return v;
        };
        auto csum = [&](int kind, int c) {
            return colp[(kind * 4 + 0) * 64 + c] + colp[(kind * 4 + 1) * 64 + c] + colp[(kind * 4 + 2) * 64 + c] +
                   colp[(kind * 4 + 3) * 64 + c];
        };
        if (tid >= kTail) {
            const int r = tid - kTail;
            // the slot of the unit after next, for the next unit's loop head (the load's latency,
            // behind this unit's bulk traffic, would otherwise open that unit)
            const long long unn = un + gridDim.x;
            SlotInfo ns{0, 0, 0, 0};
            if (r == 0 && unn < units) ns = p.slot_info[(uint32_t)unn / (uint32_t)p.H];
            if (ok) {
                float g = 0.f;
                if (r < L) {
                    g = rsum(0, r) + rsum(3, r) - csum(0, r) - csum(1, r);   // Kbar terms: prefix sum below
                    if (r + 1 < L) {
                        g += rsum(5, r + 1);
                        g += sWs[r + 1] * rsum(7, r + 1);
                    }
                }
                sDg[r] = g;
            }
            tail_sync();
            if (ok && warp == kTail / 32) {
                // d log alpha_j = sum_{r >= j} dg_r (a suffix sum inside the chunk) plus gamma_C <H, dH'> at the
                // last position; the Kbar terms, which reach it as (their total - their suffix), are
                // added as the exclusive prefix sum_{r < j} instead, so nothing cancels.
                float k0 = lane < L ? rsum(1, lane) : 0.f, k1 = lane + 32 < L ? rsum(1, lane + 32) : 0.f;
                float hd = lane < kLocalThreads / 32 ? red[lane] : 0.f;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) hd += __shfl_xor_sync(0xffffffffu, hd, o);
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {   // inclusive prefix sums of the Kbar terms
                    const float y0 = __shfl_up_sync(0xffffffffu, k0, o);
                    const float y1 = __shfl_up_sync(0xffffffffu, k1, o);
                    if (lane >= o) { k0 += y0; k1 += y1; }
                }
                const float half0 = __shfl_sync(0xffffffffu, k0, 31);
                k1 += half0;
                const float e0p = __shfl_up_sync(0xffffffffu, k0, 1), e1p = __shfl_up_sync(0xffffffffu, k1, 1);
                const float e0 = lane == 0 ? 0.f : e0p, e1 = lane == 0 ? half0 : e1p;   // exclusive prefixes
                float x0 = sDg[lane], x1 = sDg[lane + 32];   // zero past L
                const float last = __expf(gL) * hd;
                if (L - 1 == lane) x0 += last;
                if (L - 1 == lane + 32) x1 += last;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const float y0 = __shfl_down_sync(0xffffffffu, x0, o);
                    const float y1 = __shfl_down_sync(0xffffffffu, x1, o);
                    if (lane + o < 32) { x0 += y0; x1 += y1; }
                }
                x0 += __shfl_sync(0xffffffffu, x1, 0);
                sDg[lane] = x0 + e0;
                sDg[lane + 32] = x1 + e1;
            }
            tail_sync();
            if (ok) {
                float dbt = 0.f, db_c = 0.f, dd_c = 0.f;
                if (r < L) {
                    dbt = rsum(4, r) + sEm1[r] * rsum(7, r);
                    // dbt is the gradient of btilde_r = b beta_r f_r (f_r = 1, or 2 alpha_r for iplr)
                    const float fr = feedback_scale(p.iplr, sAl[r]);
                    const float bh = sNx[322];
                    p.dalpha[(t0 + r) * p.H + h] = sDg[r] / sAl[r] + (p.iplr ? 2.f * bh * sBe[r] * dbt : 0.f);
                    p.dbeta[(t0 + r) * p.H + h] = rsum(2, r) + bh * fr * dbt;
                    db_c = sBe[r] * fr * dbt;
                    dd_c = -rsum(6, r);
                }
                // fixed-order reduction of the two per-chunk partials over 64 rows
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    db_c += __shfl_xor_sync(0xffffffffu, db_c, o);
                    dd_c += __shfl_xor_sync(0xffffffffu, dd_c, o);
                }
                if (lane == 0) { red[(warp - kTail / 32) * 2] = db_c; red[(warp - kTail / 32) * 2 + 1] = dd_c; }
            }
            tail_sync();
            if (r == 0) {
                if (ok) {
                    p.part[idx * 2] = red[0] + red[2];
                    p.part[idx * 2 + 1] = red[1] + red[3];
                } else {
                    flag_error(p);
                }
                s_nslot = make_int2(ns.start, ns.len);
            }
        }
        ok = !__syncthreads_or(!ok);   // the staging tile read above takes the Q/K copies of the unit after next
        pre = has_next;
        nslot = true;
        lph ^= 1;
        u = un;
        cur = nxt;
    }
    cp_async_wait<0>();   // no scalar copy is still writing shared memory at exit
    // no tile copy is still writing shared memory at exit (after a give-up, the next unit's tiles are
    // in the phase after this one's, P in this one's)
    if (tid == kTma && pend) {
        for (int i = 0; i < 4; ++i)
            if (pend & (1u << i)) mbar_drain(smem_u32(&ldn[i]), lph);
        if (pend & 32u) mbar_drain(smem_u32(&ldp), lph ^ 1);
    }
    if (tid == 0) bulk_wait_rows_done();   // and no bulk store is still reading it
    if (!ok) ms.drain(tid);               // nor a product still writing TMEM after a wait gave up
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
}

}  // namespace tc

cudaError_t launch_bwd_local_tc(const ChunkParams& p, cudaStream_t s) {
    const size_t sm = tc::LocalTcSmem::bytes();
    const bool pk = p.p != nullptr;
    auto kern = pk ? tc::k_bwd_local_tc<true> : tc::k_bwd_local_tc<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    int dev = 0, nsm = 0;
    if ((e = cudaGetDevice(&dev)) || (e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev))) return e;
    const long long units = (long long)p.slots * p.H;
    if (units >= (1ll << 31)) return cudaErrorInvalidValue;   // unit indices are 32-bit in the kernel
    const int grid = (int)(units < nsm ? units : nsm);   // one resident CTA per SM
    tc::LocalMaps mp;
    const int Hk = p.H / p.vg;
    bool good = make_bf16_token_map(&mp.dq, p.dq, p.Ttot, p.H, tc::D) &&
                make_bf16_token_map(&mp.dk, p.dkk, p.Ttot, p.H, tc::D) &&
                make_bf16_token_map(&mp.q, p.q, p.Ttot, Hk, tc::D) &&
                make_bf16_token_map(&mp.k, p.k, p.Ttot, Hk, tc::D) &&
                make_bf16_token_map(&mp.v, p.v, p.Ttot, p.H, tc::D) &&
                make_bf16_token_map(&mp.dO, p.dO, p.Ttot, p.H, tc::D) &&
                make_bf16_map(&mp.e, p.Eb, units * 64, tc::D, 64) &&
                make_bf16_map(&mp.h, p.Hb, units * tc::D, tc::D, tc::D) &&
                make_bf16_map(&mp.dh, p.dHb, units * tc::D, tc::D, tc::D) &&
                make_bf16_map(&mp.m, p.Mb, units * 64, 64, 64);
    if (pk) {
        good = good && p.dpp && make_bf16_token_map(&mp.dp, p.dpp, p.Ttot, p.H, tc::D) &&
               make_bf16_token_map(&mp.p, p.p, p.Ttot, Hk, tc::D);
    } else {
        mp.dp = mp.dq;   // not used
        mp.p = mp.q;
    }
    if (!good) return cudaErrorInvalidValue;
    if (grid > 0) kern<<<grid, tc::kLocalThreads, sm, s>>>(p, units, mp);
    return cudaGetLastError();
}

size_t local_tc_smem_bytes() { return tc::LocalTcSmem::bytes(); }

}  // namespace comba
