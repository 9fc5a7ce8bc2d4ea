// M = 64 accumulators read in the mma.sync m16n8 fragment layout, and fragment tiles moved to
// and from 128-byte-swizzled shared tiles (tcgen05 kernels whose epilogues are fragment code).
//
// An M = 64 accumulator row m lives in TMEM lane 32 (m / 16) + m % 16, so warp w, which may read
// only the lane quadrant w % 4, reads the rows 16 (w % 4) .. + 15; tcgen05.ld.16x256b hands them
// out as m16n8 accumulator fragments (thread l: rows l / 4 and + 8, columns 2 (l % 4) and + 1 of
// each 8-column tile).
#pragma once

#include "tc_tiles.cuh"

namespace comba {
namespace tc {

// M = 64 accumulator columns [taddr, +8 NT) of this warp's 16 rows as m16n8 fragments (NT = 4, 2).
__device__ __forceinline__ void tmem_frag4(uint32_t taddr, float (&a)[4][4]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) a[i >> 2][i & 3] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_frag2(uint32_t taddr, float (&a)[2][4]) {
    uint32_t r[8];
    asm volatile("tcgen05.ld.sync.aligned.16x256b.x2.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
    for (int i = 0; i < 8; ++i) a[i >> 2][i & 3] = __uint_as_float(r[i]);
}

__device__ __forceinline__ uint32_t pack_bf2(float x, float y) {
    __nv_bfloat162 v = __floats2bfloat162_rn(x, y);
    return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ void stsm_x4(const void* p, uint32_t r0, uint32_t r1, uint32_t r2, uint32_t r3) {
    asm volatile("stmatrix.sync.aligned.m8n8.x4.shared.b16 [%0], {%1,%2,%3,%4};\n" ::"r"(smem_u32(p)), "r"(r0),
                 "r"(r1), "r"(r2), "r"(r3)
                 : "memory");
}
// The m16n8 accumulator fragment is the layout of four 8 x 8 b16 matrices of ldmatrix / stmatrix
// (thread l: row l / 4, columns 2 (l % 4) and + 1), so a warp moves its 16 rows x 16 columns of a
// fragment tile with one x4 instruction: matrices (rows 0-7, n8 tile t), (rows 8-15, t), (rows
// 0-7, t + 1), (rows 8-15, t + 1), lane l addressing row (l & 7) + 8 ((l >> 3) & 1) of matrix
// l >> 3 (a 16-byte chunk, which the swizzle or the staging rotation keeps whole).
__device__ __forceinline__ int frag_mrow(int m0) { return m0 + (threadIdx.x & 7) + (((threadIdx.x >> 3) & 1) << 3); }
__device__ __forceinline__ int frag_mcol(int n0, int t) { return n0 + 8 * (t + ((threadIdx.x >> 4) & 1)); }
// Fragment tile into a K-major swizzled tile (columns n0 + 8 t + ...).
template <int NT>
__device__ __forceinline__ void frag_store_sw(uint8_t* tile, int rows, int m0, int n0, const float (&acc)[NT][4]) {
    static_assert(NT % 2 == 0, "pairs of n8 tiles");
    const int mr = frag_mrow(m0);
#pragma unroll
    for (int t = 0; t < NT; t += 2)
        stsm_x4(tile + sw128_offset(mr, frag_mcol(n0, t), rows), pack_bf2(acc[t][0], acc[t][1]),
                pack_bf2(acc[t][2], acc[t][3]), pack_bf2(acc[t + 1][0], acc[t + 1][1]),
                pack_bf2(acc[t + 1][2], acc[t + 1][3]));
}
// The same tile read back as packed bf16 pairs: w[2 t] = (row g, tile t), w[2 t + 1] = (row g + 8, t).
template <int NT>
__device__ __forceinline__ void frag_load_sw(const uint8_t* tile, int rows, int m0, int n0, uint32_t (&w)[2 * NT]) {
    static_assert(NT % 2 == 0, "pairs of n8 tiles");
    const int mr = frag_mrow(m0);
#pragma unroll
    for (int t = 0; t < NT; t += 2) {
        uint32_t r[4];
        ldsm_x4(r, tile + sw128_offset(mr, frag_mcol(n0, t), rows));
        w[2 * t] = r[0]; w[2 * t + 1] = r[1]; w[2 * t + 2] = r[2]; w[2 * t + 3] = r[3];
    }
}
template <int NT>
__device__ __forceinline__ void tmem_frag(uint32_t taddr, float (&a)[NT][4]) {
    static_assert(NT == 2 || NT == 4, "column quarters of 64- and 128-wide accumulators");
    if constexpr (NT == 2) tmem_frag2(taddr, a);
    else tmem_frag4(taddr, a);
}
// Several accumulators read with one wait: tmem_issue() starts a load, tmem_wait() completes
// every load issued before it, and tmem_take() then moves the words into floats behind an empty
// asm per register, so that no use of them is scheduled ahead of the wait.
template <int NT>
__device__ __forceinline__ void tmem_issue(uint32_t taddr, uint32_t (&r)[NT * 4]) {
    static_assert(NT == 2 || NT == 4, "column quarters of 64- and 128-wide accumulators");
    if constexpr (NT == 2) {
        asm volatile("tcgen05.ld.sync.aligned.16x256b.x2.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];\n"
                     : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                     : "r"(taddr));
    } else {
        asm volatile(
            "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
              "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
            : "r"(taddr));
    }
}
__device__ __forceinline__ void tmem_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }
template <int NT>
__device__ __forceinline__ void tmem_take(uint32_t (&r)[NT * 4], float (&a)[NT][4]) {
#pragma unroll
    for (int i = 0; i < NT * 4; ++i) {
        asm volatile("" : "+r"(r[i]));
        a[i >> 2][i & 3] = __uint_as_float(r[i]);
    }
}

}  // namespace tc
}  // namespace comba
