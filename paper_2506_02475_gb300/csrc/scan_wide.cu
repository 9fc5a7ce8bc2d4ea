// Sequential inter-chunk scan for head dim dk = 256.
//
// At dk = 256 a chunk's folded map Atilde = -Kbar^T W is 256 x 256 (128 KB in
// bf16): writing and reading it per (chunk, head) would cost twice W and K
// together.  So this scan applies section 3.2's chunk equations directly, two
// products per chunk:
//     forward:   E = U - W H,            H' = gamma_C H + Kbar^T E
//     backward:  R = Kbar dH',           dH = gamma_C dH' + C - W^T R,   C = Z^T dO
// with Kbar = Diag(s) K, s_r = gamma_C / gamma_r for positions r < L (zero past
// the chunk).  Both run transposed over one value head's 64 state rows (dv):
//     Pt = (Z - S^T F1^T) Diag(s),       S^T <- gamma_C S^T + Pt F2 + Y
// forward:  F1 = W, F2 = K, Z = U^T, Y = 0 (Pt = E^T Diag(s));
// backward: F1 = K, F2 = W, Z = 0,   Y = C^T (Pt = -R^T).
// The backward forms Y itself: C^T = dO^T Z (M = 64, N = 256, K = 64) from the
// chunk's Z = Diag(gamma) Q~ - P W (saved by the forward's output kernel once per
// key head) and this value head's dO, issued right after the first product into
// the second product's accumulator, so it runs while Pt is formed and the second
// product accumulates onto it.
// W rows past the chunk are zero (prep zero-fills its key rows).  Key rows past
// a short chunk (the next sequence's tokens, or the fill value past the tensor)
// meet s_r = 0, but are zeroed in shared memory all the same, so that a
// non-finite key elsewhere cannot reach this sequence (0 * inf); so are the dO
// rows there in the backward.
//
// One CTA per (sequence, value head), 256 threads.  Both products run on the
// tensor core (tcgen05, M = 64): S^T F1^T (N = 64, K = 256) and Pt F2 (N = 256,
// K = 64; F2 is read MN-major from the same [64][256] tile layout that serves
// as the K-major F1).  The accumulators are read with tcgen05.ld.16x256b, which
// gives each warp 16 rows in the m16n8 fragment layout: warp (wr, wc) keeps
// state rows 16 wr + g (+ 8) and columns 128 wc + 8 t + 2 q (+ 1) in registers
// (64 fp32 values a thread) across the whole sequence.  One thread issues the
// MMAs; another issues the TMA traffic: F1 single-buffered and refilled as soon
// as the first product has read it, F2 and Z / Y double-buffered a chunk
// ahead (the backward's stage also holds Z and the dO tile), and each chunk's
// starting state (H_n^T, or dH_{n+1}^T in the backward) stored in bf16 by a bulk
// tensor copy from the A-operand tile.
#include <cuda.h>

#include "params.cuh"

namespace comba {

bool make_bf16_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows);
bool make_bf16_token_map(CUtensorMap* m, const void* base, long long tokens, int heads, int cols);

namespace {

constexpr int kWideDK = 256, kWideDV = 64;


struct WideSmem {
    static constexpr uint32_t T_BYTES = 64 * kWideDK * 2;   // a [64][256] bf16 tile: four 64-column halves
    static constexpr uint32_t OA = 0;                       // S^T: A operand of the first product, stored state
    static constexpr uint32_t OP = OA + T_BYTES;            // Pt: A operand of the second product [64][64]
    static constexpr uint32_t OF1 = OP + 8192;              // F1 (one buffer)
    static constexpr uint32_t OST = OF1 + T_BYTES;          // two stages: F2, then U [64][64] (forward) or
                                                            // Z [64][256] and dO [64][64] (backward)
    __host__ __device__ static constexpr uint32_t z_bytes(bool reverse) { return reverse ? T_BYTES + 8192 : 8192; }
    __host__ __device__ static constexpr uint32_t stage_bytes(bool reverse) { return T_BYTES + z_bytes(reverse); }
    __host__ __device__ static constexpr size_t bytes(bool reverse) { return 1024 + OST + 2 * stage_bytes(reverse); }
};

__device__ __forceinline__ void wide_seq_range(const ScanArgs& a, int n, long long& start, long long& len) {
    long long s = a.cu ? a.cu[n] : (long long)n * a.T;
    long long e = a.cu ? a.cu[n + 1] : (long long)(n + 1) * a.T;
    s = s < 0 ? 0 : (s > a.Ttot ? a.Ttot : s);
    e = e < s ? s : (e > a.Ttot ? a.Ttot : e);
    start = s;
    len = e - s;
}

__device__ __forceinline__ void tma_store_tile(const void* tmap, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];\n"
                 ::"l"(tmap), "r"(x), "r"(y), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit_group() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read_all() { asm volatile("cp.async.bulk.wait_group.read 0;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all_groups() { asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory"); }

// TMEM loads of M = 64 accumulator columns in the m16n8 fragment layout: NT 8-column tiles.
template <int NT>
__device__ __forceinline__ void tmem_frags(uint32_t taddr, uint32_t (&r)[NT * 4]) {
    static_assert(NT == 4 || NT == 16, "the two accumulator widths read here");
    if constexpr (NT == 4) {
        asm volatile(
            "tcgen05.ld.sync.aligned.16x256b.x4.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
            : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
              "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
            : "r"(taddr));
    } else {
#pragma unroll
        for (int q = 0; q < 2; ++q)
            asm volatile(
                "tcgen05.ld.sync.aligned.16x256b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
                "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
                : "=r"(r[32 * q + 0]), "=r"(r[32 * q + 1]), "=r"(r[32 * q + 2]), "=r"(r[32 * q + 3]),
                  "=r"(r[32 * q + 4]), "=r"(r[32 * q + 5]), "=r"(r[32 * q + 6]), "=r"(r[32 * q + 7]),
                  "=r"(r[32 * q + 8]), "=r"(r[32 * q + 9]), "=r"(r[32 * q + 10]), "=r"(r[32 * q + 11]),
                  "=r"(r[32 * q + 12]), "=r"(r[32 * q + 13]), "=r"(r[32 * q + 14]), "=r"(r[32 * q + 15]),
                  "=r"(r[32 * q + 16]), "=r"(r[32 * q + 17]), "=r"(r[32 * q + 18]), "=r"(r[32 * q + 19]),
                  "=r"(r[32 * q + 20]), "=r"(r[32 * q + 21]), "=r"(r[32 * q + 22]), "=r"(r[32 * q + 23]),
                  "=r"(r[32 * q + 24]), "=r"(r[32 * q + 25]), "=r"(r[32 * q + 26]), "=r"(r[32 * q + 27]),
                  "=r"(r[32 * q + 28]), "=r"(r[32 * q + 29]), "=r"(r[32 * q + 30]), "=r"(r[32 * q + 31])
                : "r"(taddr + 64 * q));
    }
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
    for (int i = 0; i < NT * 4; ++i) asm volatile("" : "+r"(r[i]));
}

__global__ void __launch_bounds__(256, 1)
    k_scan_wide(ScanArgs a, const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmZ, const __grid_constant__ CUtensorMap tmS,
                const __grid_constant__ CUtensorMap tmO) {
    using S = WideSmem;
    constexpr int DK = kWideDK, DV = kWideDV, NT = DK / 16;   // 16 8-column state tiles a thread
    constexpr int kTma = 32;                                  // the thread that issues the TMA traffic
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t full_f1, full_st[2], mma1_bar, mma2_bar;
    __shared__ uint32_t tmem_base;
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wr = warp & 3, wc = warp >> 2;
    const int n = blockIdx.x, h = blockIdx.y;
    const bool rev = a.reverse != 0;
    const int Hk = a.H / a.vg, hk = h / a.vg;
    const int r0 = 16 * wr + (lane >> 2);       // state rows r0, r0 + 8 (value columns of the head)
    const int cq = 128 * wc + 2 * (lane & 3);   // state columns cq + 8 t, + 1 (key rows)
    const int pc = 32 * wc + 2 * (lane & 3);    // Pt columns pc + 8 t, + 1 (chunk positions)
    const uint32_t su = smem_u32(smem);
    const uint32_t uA = su + S::OA, uP = su + S::OP, uF1 = su + S::OF1;
    const uint32_t stb = S::stage_bytes(rev);
    auto uF2 = [&](int it) { return su + S::OST + (uint32_t)(it & 1) * stb; };
    auto uZ = [&](int it) { return uF2(it) + S::T_BYTES; };

    float st[NT][4];
    const long long soff = ((long long)n * Hk + hk) * DK * ((long long)a.vg * DV) + (long long)(h - hk * a.vg) * DV;
    const long long sld = (long long)a.vg * DV;   // stride between state rows (key index) of init / fin
#pragma unroll
    for (int t = 0; t < NT; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i)
            st[t][i] = a.init ? a.init[soff + (long long)(cq + 8 * t + (i & 1)) * sld + r0 + 8 * (i >> 1)] : 0.f;

    long long start, len;
    wide_seq_range(a, n, start, len);
    const int s0 = a.seq_first[n];
    int nch = (int)((len + kChunk - 1) / kChunk);
    if (s0 + nch > a.slots) nch = a.slots - s0 > 0 ? a.slots - s0 : 0;
    auto chunk_of = [&](int it) { return rev ? nch - 1 - it : it; };
    auto unit_of = [&](int it) { return (long long)(s0 + chunk_of(it)) * a.H + h; };
    // W and the log-decays are stored once per key head, at its first value head's unit: the
    // key head's value-head CTAs read the same tiles (and so share them in L2)
    auto kunit_of = [&](int it) { return (long long)(s0 + chunk_of(it)) * a.H + hk * a.vg; };
    auto len_of = [&](int it) {
        const long long rest = len - (long long)chunk_of(it) * kChunk;
        return (int)(rest < kChunk ? rest : kChunk);
    };

    if (tid == 0) {
        mbar_init(smem_u32(&full_f1), 1);
        mbar_init(smem_u32(&full_st[0]), 1);
        mbar_init(smem_u32(&full_st[1]), 1);
        mbar_init(smem_u32(&mma1_bar), 1);
        mbar_init(smem_u32(&mma2_bar), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tmem_base), 512);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;
    const uint32_t tq = tmem + ((uint32_t)(32 * wr) << 16);   // this warp's TMEM lane quadrant

    // TMA: a chunk's W (its 64 stored rows) or its key rows (tokens t0 .., key head hk)
    auto load_w = [&](uint32_t dst, int it, uint32_t bar) {
#pragma unroll
        for (int half = 0; half < 4; ++half) tma_load_2d(dst + half * 8192, &tmW, 64 * half, (int)(kunit_of(it) * 64), bar);
    };
    auto load_k = [&](uint32_t dst, int it, uint32_t bar) {
        const int t0 = (int)(start + (long long)chunk_of(it) * kChunk);
#pragma unroll
        for (int half = 0; half < 4; ++half) tma_load_2d(dst + half * 8192, &tmK, hk * DK + 64 * half, t0, bar);
    };
    int nf1 = 0, nst = 0;   // F1 loads and stages issued (thread kTma)
    auto issue_f1 = [&](int it) {
        const uint32_t bar = smem_u32(&full_f1);
        mbar_expect_tx(bar, S::T_BYTES);
        if (rev) load_k(uF1, it, bar);
        else load_w(uF1, it, bar);
        ++nf1;
    };
    auto issue_stage = [&](int it) {
        const uint32_t bar = smem_u32(&full_st[it & 1]);
        mbar_expect_tx(bar, stb);
        if (rev) {
            load_w(uF2(it), it, bar);
#pragma unroll
            for (int half = 0; half < 4; ++half)   // Z, stored at the key head's unit
                tma_load_2d(uZ(it) + half * 8192, &tmZ, 64 * half, (int)(kunit_of(it) * 64), bar);
            tma_load_3d(uZ(it) + S::T_BYTES, &tmO, 0, h, (int)(start + (long long)chunk_of(it) * kChunk), bar);   // dO
        } else {
            load_k(uF2(it), it, bar);
            tma_load_2d(uZ(it), &tmZ, 0, (int)(unit_of(it) * 64), bar);                              // U
        }
        ++nst;
    };
    if (tid == kTma && nch > 0) {
        issue_f1(0);
        issue_stage(0);
        if (nch > 1) issue_stage(1);
    }

    // the chunk's log-decays at this thread's Pt columns and at its last position, a chunk ahead
    float gc[8], gl = 0.f;
    auto load_g = [&](int it) {
        const float* G = a.Gb + kunit_of(it) * 64;
        gl = __ldg(G + len_of(it) - 1);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
            gc[2 * t] = __ldg(G + pc + 8 * t);
            gc[2 * t + 1] = __ldg(G + pc + 8 * t + 1);
        }
    };
    if (nch > 0) load_g(0);

    bool failed = false;
    int n2 = 0;   // thread 0: commits to mma2_bar so far
    for (int it = 0; it < nch; ++it) {
        const int L = len_of(it);
        float g[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) g[e] = gc[e];
        const float gL = gl;
        if (it + 1 < nch) load_g(it + 1);

        // the state this chunk starts from, as the first product's A operand (the previous chunk's
        // bulk store from this tile has finished reading it)
        if (tid == kTma) bulk_wait_read_all();
        __syncthreads();
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh)
                *reinterpret_cast<__nv_bfloat162*>(smem + S::OA + sw128_offset(r0 + 8 * hh, cq + 8 * t, 64)) =
                    __floats2bfloat162_rn(st[t][2 * hh], st[t][2 * hh + 1]);
        fence_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();

        int bad = 0;
        if (tid == 0) {
            if (mbar_wait(smem_u32(&full_f1), it & 1, a.wait_ns)) {
                // backward: F1 holds the keys; the first chunk of the reverse scan may be short
                if (rev && it == 0 && L < kChunk) zero_tile_rows(smem + S::OF1, L, 4);
                tc_gemm_m64<false, false>(tmem, uA, 64, uF1, 64, 64, DK, false);
            } else {
                bad = 1;
            }
            tc_commit(smem_u32(&mma1_bar));
            if (rev && !bad) {
                // C^T = dO^T Z into the second product's columns (read back in the previous chunk's update)
                if (mbar_wait(smem_u32(&full_st[it & 1]), (it >> 1) & 1, a.wait_ns)) {
                    // the reverse scan's first chunk is a sequence's last and may be short: its dO rows
                    // past the sequence end (the next sequence's, or past the tensor) must not enter
                    if (it == 0 && L < kChunk) zero_tile_rows(smem + (uZ(it) - su) + S::T_BYTES, L, 1);
                    tc_gemm_m64<true, true>(tmem + 64, uZ(it) + S::T_BYTES, 64, uZ(it), 64, DK, 64, false);
                } else {
                    bad = 1;
                }
            }
        } else if (tid == kTma) {
#pragma unroll
            for (int half = 0; half < 4; ++half) tma_store_tile(&tmS, 64 * half, (int)(unit_of(it) * 64), uA + half * 8192);
            bulk_commit_group();
        }
        if (!mbar_wait(smem_u32(&mma1_bar), it & 1, a.wait_ns)) bad = 1;
        if (!mbar_wait(smem_u32(&full_st[it & 1]), (it >> 1) & 1, a.wait_ns)) bad = 1;
        if (__syncthreads_or(bad)) {
            failed = true;
            break;
        }
        tc_fence_after();
        if (tid == kTma && it + 1 < nch) issue_f1(it + 1);   // the first product has read F1

        // Pt = (Z - S^T F1^T) Diag(s): this warp's 16 rows, columns 32 wc .. + 31
        {
            uint32_t d[16];
            tmem_frags<4>(tq + 32 * wc, d);
            const uint8_t* z = smem + (uZ(it) - su);
#pragma unroll
            for (int t = 0; t < 4; ++t) {
                const int r = pc + 8 * t;
                const float sa = r < L ? __expf(gL - g[2 * t]) : 0.f;
                const float sb = r + 1 < L ? __expf(gL - g[2 * t + 1]) : 0.f;
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                    const int j = r0 + 8 * hh;
                    float za = 0.f, zb = 0.f;
                    if (!rev) {   // U^T
                        za = __bfloat162float(*reinterpret_cast<const bf16*>(z + sw128_offset(r, j, 64)));
                        zb = __bfloat162float(*reinterpret_cast<const bf16*>(z + sw128_offset(r + 1, j, 64)));
                    }
                    const float va = sa * (za - __uint_as_float(d[4 * t + 2 * hh]));
                    const float vb = sb * (zb - __uint_as_float(d[4 * t + 2 * hh + 1]));
                    *reinterpret_cast<__nv_bfloat162*>(smem + S::OP + sw128_offset(j, r, 64)) =
                        __floats2bfloat162_rn(va, vb);
                }
            }
        }
        fence_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();
        if (tid == 0) {
            // forward: F2 holds the keys; the last chunk may be short
            if (!rev && it + 1 == nch && L < kChunk) zero_tile_rows(smem + (uF2(it) - su), L, 4);
            tc_gemm_m64<false, true>(tmem + 64, uP, 64, uF2(it), 64, DK, 64, rev);   // onto C^T (backward)
            tc_commit(smem_u32(&mma2_bar));
            ++n2;
        }
        if (!mbar_wait(smem_u32(&mma2_bar), it & 1, a.wait_ns)) bad = 1;
        tc_fence_after();

        // S^T <- gamma_C S^T + Pt F2 + Y  (the accumulator holds Y as well)
        if (!bad) {
            uint32_t d[4 * NT];
            tmem_frags<NT>(tq + 64 + 128 * wc, d);
            const float gam = __expf(gL);
#pragma unroll
            for (int t = 0; t < NT; ++t)
#pragma unroll
                for (int i = 0; i < 4; ++i) st[t][i] = fmaf(gam, st[t][i], __uint_as_float(d[4 * t + i]));
        }
        tc_fence_before();
        if (__syncthreads_or(bad)) {   // this stage and Pt are fully read
            failed = true;
            break;
        }
        if (tid == kTma && it + 2 < nch) issue_stage(it + 2);
    }

    if (failed && tid == 0) {
        // every product finishes before TMEM is released: first the last committed phase of the
        // second barrier (it may be the pending one; a parity wait is only exact on that phase),
        // then one more commit covers the first product and a C^T product issued since
        if (n2 > 0) mbar_drain(smem_u32(&mma2_bar), (n2 - 1) & 1);
        tc_commit(smem_u32(&mma2_bar));
        mbar_drain(smem_u32(&mma2_bar), n2 & 1);
    }
    if (failed && tid == kTma) {
        // a bounded wait gave up: record it, and let the last load issued to each barrier land
        // (bounded waits again) before this CTA's shared memory is released
        if (a.err) atomicExch(a.err, 1);
        if (nf1 > 0) mbar_drain(smem_u32(&full_f1), (nf1 - 1) & 1);
        for (int b = 0; b < 2; ++b) {
            const int k = nst - 1 - ((nst - 1 - b) & 1);   // the latest stage issued to barrier b
            if (k >= 0) mbar_drain(smem_u32(&full_st[b]), (k >> 1) & 1);
        }
    }
    if (tid == kTma) bulk_wait_all_groups();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 512);
    if (a.fin) {
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i)
                a.fin[soff + (long long)(cq + 8 * t + (i & 1)) * sld + r0 + 8 * (i >> 1)] = st[t][i];
    }
}

}  // namespace

cudaError_t launch_scan_wide(const ScanArgs& a, cudaStream_t s) {
    const bool rev = a.reverse != 0;
    const long long pairs = (long long)a.slots * a.H;
    const int Hk = a.H / a.vg;
    CUtensorMap tw, tk, tz, ts, to;
    const long long krows = a.Ttot > 0 ? a.Ttot : 1;   // a valid view even when no token exists
    const long long prow = pairs > 0 ? pairs * 64 : 64;
    // backward: Z [pairs * 64][dk] (key-head units) and dO [tokens][value heads][64]; forward: U
    if (rev && (a.ym != 1 || !a.F || !a.tok)) return cudaErrorInvalidValue;
    if (!make_bf16_map(&tw, a.W, prow, kWideDK, 64) || !make_bf16_map(&tk, a.K, krows, Hk * kWideDK, 64) ||
        !make_bf16_map(&tz, rev ? a.F : a.Y, prow, rev ? kWideDK : kWideDV, 64) ||
        !make_bf16_map(&ts, a.Sout, prow, kWideDK, 64))
        return cudaErrorInvalidValue;
    if (rev) {
        if (!make_bf16_token_map(&to, a.tok, krows, a.H, kWideDV)) return cudaErrorInvalidValue;
    } else {
        to = tz;   // not read
    }
    const size_t sm = WideSmem::bytes(rev);
    cudaError_t e = cudaFuncSetAttribute(k_scan_wide, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e) return e;
    if (a.N > 0 && a.H > 0) k_scan_wide<<<dim3(a.N, a.H), 256, sm, s>>>(a, tw, tk, tz, ts, to);
    return cudaGetLastError();
}

size_t scan_wide_smem_bytes() { return WideSmem::bytes(true); }

}  // namespace comba
