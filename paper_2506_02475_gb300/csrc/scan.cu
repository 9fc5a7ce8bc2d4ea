// Sequential inter-chunk scan, shared by the forward and the backward.
//
// Folding each chunk of section 3.2's state equation into one affine map,
//     H_{n+1} = gamma_n H_n + Atilde_n H_n + B_n,
//     Atilde_n = -Kbar_n^T W_n,  B_n = Kbar_n^T U_n,  gamma_n = gamma_C of chunk n,
// leaves a single dense product on the sequential path.  The backward's
// reverse recurrence has the same form,
//     dH_n = gamma_n dH_{n+1} + Atilde_n^T dH_{n+1} + C_n,  C_n = (Qhat_n - P_n W_n)^T dO_n.
// Both are evaluated transposed, one state row (a dv index) per thread:
//     S^T <- gamma S^T + S^T X^T + Y,
// with X = Atilde (forward; row-major [dk][dk], read K-major) or, in the
// backward, Atilde read as an MN-major operand (bf16 path) or Atilde^T
// (fp32 path); Y = B^T or C^T stored [dv][dk].  Each chunk stores the state it started
// from (H_n^T, or dH_{n+1}^T in the backward) for the parallel kernels.  The
// tcgen05 path reads no Y: its scans form B^T = U_s^T K (U_s = Diag(s) U, saved
// by prep) and C^T = dO^T Z (Z^T saved by the forward's output kernel)
// themselves, one product per chunk issued ahead of the sequential one (see
// k_scan_tc_split).
//
// bf16 storage: one CTA per (sequence, head), 256 threads (two per state row,
// each holding half of the row's dk columns); the fp32 state stays in registers.
// Each chunk, S^T (bf16) is written into one of two 128-byte-swizzled K-major
// shared tiles: it is the MMA's A operand and, by a bulk tensor store issued
// right after the MMAs, the chunk's stored starting state (one SM writes
// global memory at only a few tens of bytes per cycle, so the store must not
// sit on the chunk-to-chunk path; it drains while the next chunks compute).
// X and Y stream in by TMA through mbarrier pipelines (3 and 2 stages); one
// thread issues the tcgen05 MMAs (M = 128, N = dk, K = dk) into a TMEM
// accumulator that all threads read back with tcgen05.ld (shapes other than
// dk = dv = 128; that one runs the row-split kernel below).
// fp32 storage: the same recurrence with FMA tile products (tolerance 1e-4).
#include <cuda.h>

#include "params.cuh"

namespace comba {

// Offset of the initial / final state of (sequence n, value head h): states are [N, H / vg, dk,
// vg * dv], so value head h holds the dv-column block h % vg of key head h / vg's rows.
__device__ __forceinline__ long long state_off(const ScanArgs& a, int n, int h, int DK, int DV) {
    const int hk = h / a.vg, j = h - hk * a.vg;
    return ((long long)n * (a.H / a.vg) + hk) * DK * ((long long)a.vg * DV) + (long long)j * DV;
}

__device__ __forceinline__ void scan_seq_range(const ScanArgs& a, int n, long long& start, long long& len) {
    long long s = a.cu ? a.cu[n] : (long long)n * a.T;
    long long e = a.cu ? a.cu[n + 1] : (long long)(n + 1) * a.T;
    s = s < 0 ? 0 : (s > a.Ttot ? a.Ttot : s);
    e = e < s ? s : (e > a.Ttot ? a.Ttot : e);
    start = s;
    len = e - s;
}

// ------------------------------------------------------------ tcgen05 path

template <int DK, int DV>
struct ScanTcSmem {
    static constexpr int SX = 3;                          // X stages (refilled once the MMA that read them is done)
    static constexpr int SY = 2;                          // Y stages (refilled once the epilogue that read them is done)
    static constexpr uint32_t A_BYTES = 128 * DK * 2;     // S^T tile, M = 128 rows (rows >= DV are zero); two buffers
    static constexpr uint32_t X_BYTES = DK * DK * 2;
    static constexpr uint32_t Y_BYTES = DV * DK * 2;
    static constexpr uint32_t OX = 2 * A_BYTES;
    static constexpr uint32_t OY = OX + SX * X_BYTES;
    static constexpr size_t bytes() { return 1024 + OY + (size_t)SY * Y_BYTES; }
};

__device__ __forceinline__ void tma_store_2d(const void* tmap, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];\n"
                 ::"l"(tmap), "r"(x), "r"(y), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }
// Wait until at most N bulk groups still read shared memory (resp. are incomplete).
template <int N>
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read %0;\n" ::"n"(N) : "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory"); }

template <int DK, int DV, bool XMN>
__global__ void __launch_bounds__(256, 1)
    k_scan_tc(ScanArgs a, const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmY,
              const __grid_constant__ CUtensorMap tmS) {
    using S = ScanTcSmem<DK, DV>;
    constexpr int HC = DK / 2;  // state columns per thread: two threads per state row
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t full_x[S::SX], full_y[S::SY];
    __shared__ uint64_t mma_bar;
    __shared__ uint32_t tmem_base;
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5;
    const int n = blockIdx.x, h = blockIdx.y;
    const int j = tid & 127;           // state row (dv index); warps w and w+4 share TMEM lanes
    const int c0 = (tid >> 7) * HC;    // first state column of this thread
    const bool live = j < DV;
    const uint32_t smem_u = smem_u32(smem);

    float st[HC];
    const float* init = a.init ? a.init + state_off(a, n, h, DK, DV) : nullptr;
#pragma unroll
    for (int m = 0; m < HC; ++m) st[m] = (init && live) ? init[(long long)(c0 + m) * a.vg * DV + j] : 0.f;

    long long start, len;
    scan_seq_range(a, n, start, len);
    const int s0 = a.seq_first[n];
    int nch = (int)((len + kChunk - 1) / kChunk);
    if (s0 + nch > a.slots) nch = a.slots - s0 > 0 ? a.slots - s0 : 0;

    if (tid == 0) {
        for (int s = 0; s < S::SX; ++s) mbar_init(smem_u32(&full_x[s]), 1);
        for (int s = 0; s < S::SY; ++s) mbar_init(smem_u32(&full_y[s]), 1);
        mbar_init(smem_u32(&mma_bar), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tmem_base), DK);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;
    const uint32_t tlane = tmem + ((uint32_t)((warp & 3) * 32) << 16);

    auto chunk_of = [&](int it) { return a.reverse ? nch - 1 - it : it; };
    auto unit_of = [&](int it) { return (long long)(s0 + chunk_of(it)) * a.H + h; };
    auto a_buf = [&](int it) { return smem_u + (uint32_t)(it & 1) * S::A_BYTES; };
    auto x_buf = [&](int it) { return smem_u + S::OX + (uint32_t)(it % S::SX) * S::X_BYTES; };
    auto y_off = [&](int it) { return S::OY + (uint32_t)(it % S::SY) * S::Y_BYTES; };
    auto issue_x = [&](int it) {
        const uint32_t fb = smem_u32(&full_x[it % S::SX]);
        mbar_expect_tx(fb, S::X_BYTES);
#pragma unroll
        for (int half = 0; half < DK / 64; ++half)
            tma_load_2d(x_buf(it) + half * DK * 128, &tmX, half * 64, (int)(unit_of(it) * DK), fb);
    };
    auto issue_y = [&](int it) {
        const uint32_t fb = smem_u32(&full_y[it % S::SY]);
        mbar_expect_tx(fb, S::Y_BYTES);
#pragma unroll
        for (int half = 0; half < DK / 64; ++half)
            tma_load_2d(smem_u + y_off(it) + half * DV * 128, &tmY, half * 64, (int)(unit_of(it) * DV), fb);
    };
    int nx = 0, ny = 0;   // chunks whose X / Y loads have been issued (thread 0)
    if (tid == 0) {
        for (; nx < S::SX - 1 && nx < nch; ++nx) issue_x(nx);
        for (; ny < S::SY - 1 && ny < nch; ++ny) issue_y(ny);
    }

    constexpr uint32_t idesc = idesc_bf16_f32(128, DK) | (XMN ? 1u << 16 : 0u);
    // log gamma_C of the chunk processed at step `it` (loaded one step ahead so the load latency hides)
    auto log_decay = [&](int it) {
        const int c = chunk_of(it);
        const int L = (int)(len - (long long)c * kChunk < kChunk ? len - (long long)c * kChunk : kChunk);
        return __ldg(a.Gb + unit_of(it) * 64 + L - 1);
    };
    float g_next = nch > 0 ? log_decay(0) : 0.f;
    for (int it = 0; it < nch; ++it) {
        const float gam = expf(g_next);
        if (it + 1 < nch) g_next = log_decay(it + 1);

        // The state this chunk starts from, as the MMA's A operand (bf16, swizzled, buffer it % 2;
        // the bulk store that read this buffer two chunks ago has finished reading it).
        uint8_t* sA = smem + (it & 1) * S::A_BYTES;
#pragma unroll
        for (int q = 0; q < HC / 8; ++q) {
            __nv_bfloat162 v0 = __floats2bfloat162_rn(st[8 * q + 0], st[8 * q + 1]);
            __nv_bfloat162 v1 = __floats2bfloat162_rn(st[8 * q + 2], st[8 * q + 3]);
            __nv_bfloat162 v2 = __floats2bfloat162_rn(st[8 * q + 4], st[8 * q + 5]);
            __nv_bfloat162 v3 = __floats2bfloat162_rn(st[8 * q + 6], st[8 * q + 7]);
            uint4 pk;
            pk.x = *reinterpret_cast<uint32_t*>(&v0);
            pk.y = *reinterpret_cast<uint32_t*>(&v1);
            pk.z = *reinterpret_cast<uint32_t*>(&v2);
            pk.w = *reinterpret_cast<uint32_t*>(&v3);
            *reinterpret_cast<uint4*>(sA + sw128_offset(j, c0 + 8 * q, 128)) = pk;
        }
        fence_async_smem();
        tc_fence_before();
        __syncthreads();
        tc_fence_after();

        int bad = 0;
        if (tid == 0) {
            if (mbar_wait(smem_u32(&full_x[it % S::SX]), (it / S::SX) & 1, a.wait_ns)) {
                const uint64_t a0 = desc_kmajor(a_buf(it), 128, 0);
                const uint64_t b0 = XMN ? desc_mnmajor(x_buf(it), DK, 0) : desc_kmajor(x_buf(it), DK, 0);
#pragma unroll
                for (int ks = 0; ks < DK / 16; ++ks)
                    tc_mma_bf16(tmem, a0 + desc_step<false>(128, ks), b0 + desc_step<XMN>(DK, ks), idesc,
                                ks > 0 ? 1u : 0u);
            } else {
                bad = 1;
            }
            tc_commit(smem_u32(&mma_bar));
            // The chunk's starting state goes out by one bulk tensor store from the same tile,
            // asynchronously: rows >= DV of the tile are not part of the box.
#pragma unroll
            for (int half = 0; half < DK / 64; ++half)
                tma_store_2d(&tmS, half * 64, (int)(unit_of(it) * DV), a_buf(it) + half * 128 * 128);
            bulk_commit();
            // Refill the stages chunk it-1 used: its MMA (X) and its epilogue (Y) are done.
            if (nx < nch) issue_x(nx++);
            if (ny < nch) issue_y(ny++);
        }
        if (!mbar_wait(smem_u32(&mma_bar), it & 1, a.wait_ns)) bad = 1;
        if (!mbar_wait(smem_u32(&full_y[it % S::SY]), (it / S::SY) & 1, a.wait_ns)) bad = 1;
        // Before the next chunk packs into the other A buffer, the store issued one chunk ago
        // (from that buffer) must have finished reading it.
        if (tid == 0) bulk_wait_read<1>();
        if (__syncthreads_or(bad)) {
            if (tid == 0) {
                if (a.err) atomicExch(a.err, 1);
                // drain the loads still in flight into this CTA's shared memory, and the chunk's
                // product (its commit, phase it, is the last) before TMEM is released
                for (int c = it; c < nx; ++c) mbar_drain(smem_u32(&full_x[c % S::SX]), (c / S::SX) & 1);
                for (int c = it; c < ny; ++c) mbar_drain(smem_u32(&full_y[c % S::SY]), (c / S::SY) & 1);
                mbar_drain(smem_u32(&mma_bar), it & 1);
            }
            break;
        }
        tc_fence_after();

        // S^T <- gamma S^T + (S^T X^T) + Y   (this thread's HC columns; all TMEM loads in flight at once)
        const uint8_t* sY = smem + y_off(it);
        uint32_t d[HC / 16][16];
#pragma unroll
        for (int g = 0; g < HC / 16; ++g) tmem_ld16_async(tlane + c0 + g * 16, d[g]);
        uint4 yv[HC / 8];
#pragma unroll
        for (int q = 0; q < HC / 8; ++q)
            yv[q] = live ? *reinterpret_cast<const uint4*>(sY + sw128_offset(j, c0 + 8 * q, DV)) : make_uint4(0, 0, 0, 0);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < HC / 8; ++q) {
            const __nv_bfloat162* y2 = reinterpret_cast<const __nv_bfloat162*>(&yv[q]);
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float2 yf = __bfloat1622float2(y2[e]);
                const int m = 8 * q + 2 * e;
                st[m] = fmaf(gam, st[m], __uint_as_float(d[m >> 4][m & 15]) + yf.x);
                st[m + 1] = fmaf(gam, st[m + 1], __uint_as_float(d[(m + 1) >> 4][(m + 1) & 15]) + yf.y);
            }
        }
        tc_fence_before();
    }

    // every bulk store of this CTA completes before its shared memory is released
    if (tid == 0) bulk_wait_all();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, DK);
    if (a.fin && live) {
        float* fin = a.fin + state_off(a, n, h, DK, DV);
#pragma unroll
        for (int m = 0; m < HC; ++m) fin[(long long)(c0 + m) * a.vg * DV + j] = st[m];
    }
}

// Row-split variant (dk = dv = 128, the tcgen05 path): two CTAs per (sequence, head), each
// owning 64 of the state's dv rows (rows are independent under S^T <- gamma S^T + S^T X^T + Y).
// The MMA is M = 64 (this CTA's rows) x N = dk x K = dk against the full X; read back with
// tcgen05.ld.16x256b, the accumulator arrives in the m16n8 fragment layout, so each thread
// keeps 32 state values (rows 16 (w & 3) + g, + 8; columns 64 (w >> 2) + 8 t + 2 q, + 1).
// Per chunk each SM loads X and stores half of the chunk state, and the epilogue is half as
// long.  One thread issues the MMAs while another issues the TMA stores and loads, so a
// step's critical path is the MMA, not the issue sequence.
//
// The additive term Y is not read: this kernel forms its rows as one more product per chunk,
// K = 64 positions, from a workspace factor F and a token tensor T of the chunk:
//   forward (YM = 2):  B^T = U_s^T K,  F = U_s^T = (Diag(s) U)^T [dv][64] (this CTA's 64 rows,
//                      K-major A), T = the chunk's keys [64][dk] (MN-major B);
//   reverse (YM = 1):  C^T = dO^T Z,   F = Z^T [dk][64] (K-major B), T = this CTA's 64 columns
//                      of dO [64][64] (MN-major A).
// F and T stream in four chunks deep.  Each chunk's product is issued right after the previous
// chunk's state product, into the other of two TMEM accumulators, so it runs while that
// chunk's epilogue does; the state product then accumulates onto it.  The rows of T past a
// short chunk's end (the next sequence's tokens, or past the tensor) are zeroed first, so
// nothing from outside the sequence enters its sums.
template <int DK, int DV, int YM>
struct ScanSplitSmem {
    static constexpr int SX = 3, SF = 4;
    static constexpr uint32_t A_BYTES = 64 * DK * 2;                 // this CTA's 64 rows of S^T; two buffers
    static constexpr uint32_t X_BYTES = DK * DK * 2;
    static constexpr uint32_t F_BYTES = (YM == 1 ? DK : 64) * 64 * 2;   // Z^T, or this CTA's rows of U_s^T
    static constexpr uint32_t T_BYTES = 64 * (YM == 1 ? 64 : DK) * 2;   // this CTA's dO columns, or K
    static constexpr uint32_t OX = 2 * A_BYTES;
    static constexpr uint32_t OF = OX + SX * X_BYTES;
    static constexpr uint32_t OT = OF + SF * F_BYTES;
    static constexpr size_t bytes() { return 1024 + OT + (size_t)SF * T_BYTES; }
};

template <int DK, int DV, bool XMN, int YM>
__global__ void __launch_bounds__(256, 1)
    k_scan_tc_split(ScanArgs a, const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmF,
                    const __grid_constant__ CUtensorMap tmS, const __grid_constant__ CUtensorMap tmT) {
    static_assert(DK == 128 && DV == 128, "row split is laid out for dk = dv = 128");
    static_assert(YM == 1 || YM == 2, "the additive term is formed in the scan");
    using S = ScanSplitSmem<DK, DV, YM>;
    constexpr int NT = DK / 16;   // 8-column tiles per thread (half of the columns)
    extern __shared__ uint8_t smem_raw[];
    __shared__ uint64_t full_x[S::SX], full_f[S::SF];
    __shared__ uint64_t mma_bar;
    __shared__ uint32_t tmem_base;
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n = blockIdx.x >> 1, rhalf = blockIdx.x & 1, h = blockIdx.y;
    const int wr = warp & 3, wc = warp >> 2;
    const int r0 = 16 * wr + (lane >> 2);          // local rows r0, r0 + 8
    const int cq = 64 * wc + 2 * (lane & 3);       // columns cq + 8 t, + 1
    const uint32_t smem_u = smem_u32(smem);

    float st[NT][4];
    {
        const float* init = a.init ? a.init + state_off(a, n, h, DK, DV) : nullptr;
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int j = 64 * rhalf + r0 + 8 * (i >> 1), m = cq + 8 * t + (i & 1);
                st[t][i] = init ? init[(long long)m * a.vg * DV + j] : 0.f;
            }
    }

    long long start, len;
    scan_seq_range(a, n, start, len);
    const int s0 = a.seq_first[n];
    int nch = (int)((len + kChunk - 1) / kChunk);
    if (s0 + nch > a.slots) nch = a.slots - s0 > 0 ? a.slots - s0 : 0;

    if (tid == 0) {
        for (int s = 0; s < S::SX; ++s) mbar_init(smem_u32(&full_x[s]), 1);
        for (int s = 0; s < S::SF; ++s) mbar_init(smem_u32(&full_f[s]), 1);
        mbar_init(smem_u32(&mma_bar), 1);
        mbar_fence_init();
    }
    if (warp == 0) tmem_alloc(smem_u32(&tmem_base), 2 * DK);   // two accumulators: chunk it in (it & 1)
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base;
    const uint32_t tq = tmem + ((uint32_t)(32 * wr) << 16) + 64 * wc;
    auto acc_col = [&](int it) { return (uint32_t)(it & 1) * DK; };

    auto chunk_of = [&](int it) { return a.reverse ? nch - 1 - it : it; };
    auto unit_of = [&](int it) { return (long long)(s0 + chunk_of(it)) * a.H + h; };
    auto a_buf = [&](int it) { return smem_u + (uint32_t)(it & 1) * S::A_BYTES; };
    auto x_buf = [&](int it) { return smem_u + S::OX + (uint32_t)(it % S::SX) * S::X_BYTES; };
    auto f_off = [&](int it) { return S::OF + (uint32_t)(it % S::SF) * S::F_BYTES; };
    auto t_off = [&](int it) { return S::OT + (uint32_t)(it % S::SF) * S::T_BYTES; };
    auto issue_x = [&](int it) {
        const uint32_t fb = smem_u32(&full_x[it % S::SX]);
        mbar_expect_tx(fb, S::X_BYTES);
#pragma unroll
        for (int half = 0; half < DK / 64; ++half)
            tma_load_2d(x_buf(it) + half * DK * 128, &tmX, half * 64, (int)(unit_of(it) * DK), fb);
    };
    auto issue_f = [&](int it) {   // F and T of the chunk
        const uint32_t fb = smem_u32(&full_f[it % S::SF]);
        mbar_expect_tx(fb, S::F_BYTES + S::T_BYTES);
        const int tok = (int)(start + (long long)chunk_of(it) * kChunk);
        if constexpr (YM == 1) {
            tma_load_2d(smem_u + f_off(it), &tmF, 0, (int)(unit_of(it) * DK), fb);
            tma_load_3d(smem_u + t_off(it), &tmT, 64 * rhalf, h, tok, fb);
        } else {
            tma_load_2d(smem_u + f_off(it), &tmF, 0, (int)(unit_of(it) * DV + 64 * rhalf), fb);
#pragma unroll
            for (int half = 0; half < DK / 64; ++half)   // the key head's keys, two 64-column halves
                tma_load_3d(smem_u + t_off(it) + half * 64 * 128, &tmT, 64 * half, h / a.vg, tok, fb);
        }
    };
    // Thread 0 issues the MMAs; thread 32 (warp 1) the TMA traffic: the chunk-state stores, the
    // X / F / T loads and the bulk-group waits, so neither waits for the other's issue sequence.
    constexpr int kTma = 32;
    int nx = 0, nf = 0;
    if (tid == kTma) {
        for (; nx < S::SX - 1 && nx < nch; ++nx) issue_x(nx);
        for (; nf < S::SF - 1 && nf < nch; ++nf) issue_f(nf);
    }

    constexpr uint32_t idesc = idesc_bf16_f32(64, DK) | (XMN ? 1u << 16 : 0u);
    // additive-term product: A = dO^T (MN-major) for YM = 1, U_s^T (K-major) for YM = 2; B = Z^T
    // (K-major) for YM = 1, K (MN-major) for YM = 2
    constexpr uint32_t idesc_y = idesc_bf16_f32(64, DK) | (YM == 1 ? 1u << 15 : 1u << 16);
    // Thread 0: the rows of T past a short chunk's end are zeroed before its product is issued.
    // Only a sequence's last chunk can be short: the reverse scan's first step, the forward's last.
    auto zero_tail = [&](int it) {
        zero_tile_rows(smem + t_off(it), (int)(len - (long long)chunk_of(it) * kChunk), YM == 1 ? 1 : DK / 64);
    };
    auto issue_y = [&](int it) {
        const uint32_t fa = smem_u + f_off(it), ta = smem_u + t_off(it);
        const uint64_t a0 = YM == 1 ? desc_mnmajor(ta, 64, 0) : desc_kmajor(fa, 64, 0);
        const uint64_t b0 = YM == 1 ? desc_kmajor(fa, DK, 0) : desc_mnmajor(ta, 64, 0);
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
            tc_mma_bf16(tmem + acc_col(it), a0 + desc_step<YM == 1>(64, ks), b0 + desc_step<YM != 1>(DK, ks), idesc_y,
                        ks > 0 ? 1u : 0u);
    };
    auto wait_f = [&](int it) { return mbar_wait(smem_u32(&full_f[it % S::SF]), (it / S::SF) & 1, a.wait_ns); };
    const bool tail_short = (len & (kChunk - 1)) != 0;
    int ybad = 0;   // thread 0: a chunk's F / T never arrived
    if (tid == 0 && nch > 0) {
        if (!wait_f(0)) {
            ybad = 1;
        } else {
            if (tail_short && (YM == 1 || nch == 1)) zero_tail(0);
            issue_y(0);
        }
    }

    auto log_decay = [&](int it) {
        const int c = chunk_of(it);
        const int L = (int)(len - (long long)c * kChunk < kChunk ? len - (long long)c * kChunk : kChunk);
        return __ldg(a.Gb + unit_of(it) * 64 + L - 1);
    };
    // A give-up (a wait that ran out, or thread 0's missing F / T) reaches the whole block at the
    // next chunk's barrier, which every warp passes before thread 0 issues another product: each
    // warp waits for the products on its own and reads its accumulator rows without a block-wide
    // barrier in between.  `wbad` is uniform over the warp.
    auto give_up = [&](int it) {   // the block's failure, seen at chunk it's barrier (it <= nch)
        if (tid == kTma) {
            if (a.err) atomicExch(a.err, 1);
            // chunk it - 1's loads may still be in flight when its waits ran out; later stages were
            // not re-armed yet
            for (int c = it > 0 ? it - 1 : 0; c < nx; ++c) mbar_drain(smem_u32(&full_x[c % S::SX]), (c / S::SX) & 1);
            for (int c = it > 0 ? it - 1 : 0; c < nf; ++c) mbar_drain(smem_u32(&full_f[c % S::SF]), (c / S::SF) & 1);
        }
        if (tid == 0 && it > 0) {
            // chunk it - 1's products (phase (it - 1) & 1, which may still be pending: a parity wait
            // is only exact on the pending phase), then one more commit for an additive term issued
            // after them
            mbar_drain(smem_u32(&mma_bar), (it - 1) & 1);
            tc_commit(smem_u32(&mma_bar));
            mbar_drain(smem_u32(&mma_bar), it & 1);
        }
    };
    int wbad = 0;
    bool gave_up = false;
    float g_next = nch > 0 ? log_decay(0) : 0.f;
    for (int it = 0; it < nch; ++it) {
        const float gam = expf(g_next);
        if (it + 1 < nch) g_next = log_decay(it + 1);

        // this CTA's rows of the chunk's starting state: bf16 A operand in buffer it % 2
        uint8_t* sA = smem + (it & 1) * S::A_BYTES;
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int hh = 0; hh < 2; ++hh)
                *reinterpret_cast<__nv_bfloat162*>(sA + sw128_offset(r0 + 8 * hh, cq + 8 * t, 64)) =
                    __floats2bfloat162_rn(st[t][2 * hh], st[t][2 * hh + 1]);
        // the previous chunk's state store (issued a step ago) has read its buffer, which the next
        // chunk's state overwrites once this barrier is passed
        if (tid == kTma) bulk_wait_read<0>();
        fence_async_smem();
        tc_fence_before();
        if (__syncthreads_or(wbad)) {
            give_up(it);
            gave_up = true;
            break;
        }
        tc_fence_after();

        int bad = ybad;
        if (tid == 0) {
            if (!ybad && mbar_wait(smem_u32(&full_x[it % S::SX]), (it / S::SX) & 1, a.wait_ns)) {
                const uint64_t a0 = desc_kmajor(a_buf(it), 64, 0);
                const uint64_t b0 = XMN ? desc_mnmajor(x_buf(it), DK, 0) : desc_kmajor(x_buf(it), DK, 0);
#pragma unroll
                for (int ks = 0; ks < DK / 16; ++ks)   // onto the additive term
                    tc_mma_bf16(tmem + acc_col(it), a0 + desc_step<false>(64, ks), b0 + desc_step<XMN>(DK, ks), idesc,
                                1u);
            } else {
                bad = 1;
            }
            tc_commit(smem_u32(&mma_bar));
        } else if (tid == kTma) {
#pragma unroll
            for (int half = 0; half < DK / 64; ++half)
                tma_store_2d(&tmS, half * 64, (int)(unit_of(it) * DV + 64 * rhalf), a_buf(it) + half * 64 * 128);
            bulk_commit();
            if (nx < nch) issue_x(nx++);
            // its stage last held chunk it - 1, whose product the commit of chunk it - 1 covered
            if (nf < nch) issue_f(nf++);
        }
        if (!mbar_wait(smem_u32(&mma_bar), it & 1, a.wait_ns)) bad = 1;
        wbad = __any_sync(0xffffffffu, bad);
        tc_fence_after();

        // S^T <- gamma S^T + (Y + S^T X^T)  on this thread's 32 values
        uint32_t d[32];
        asm volatile(
            "tcgen05.ld.sync.aligned.16x256b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
            "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
            : "=r"(d[0]), "=r"(d[1]), "=r"(d[2]), "=r"(d[3]), "=r"(d[4]), "=r"(d[5]), "=r"(d[6]), "=r"(d[7]),
              "=r"(d[8]), "=r"(d[9]), "=r"(d[10]), "=r"(d[11]), "=r"(d[12]), "=r"(d[13]), "=r"(d[14]), "=r"(d[15]),
              "=r"(d[16]), "=r"(d[17]), "=r"(d[18]), "=r"(d[19]), "=r"(d[20]), "=r"(d[21]), "=r"(d[22]), "=r"(d[23]),
              "=r"(d[24]), "=r"(d[25]), "=r"(d[26]), "=r"(d[27]), "=r"(d[28]), "=r"(d[29]), "=r"(d[30]), "=r"(d[31])
            : "r"(tq + acc_col(it)));
        tmem_wait_ld();
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) st[t][i] = fmaf(gam, st[t][i], __uint_as_float(d[4 * t + i]));
        tc_fence_before();
        // The next chunk's additive term, into the other accumulator (read back a chunk ago), once
        // this chunk's products are done: issued behind them it would hold every warp at the
        // barrier above while thread 0 waits for room in the tensor core's queue.
        if (tid == 0 && !ybad && it + 1 < nch) {
            if (!wait_f(it + 1)) {
                ybad = 1;
            } else {
                if constexpr (YM == 2)
                    if (tail_short && it + 2 == nch) zero_tail(it + 1);
                issue_y(it + 1);
            }
        }
    }

    // the last chunk's waits, unless the loop has given up already
    if (__syncthreads_or(wbad) && !gave_up) give_up(nch);
    if (tid == kTma) bulk_wait_all();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 2 * DK);
    if (a.fin) {
        float* fin = a.fin + state_off(a, n, h, DK, DV);
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int j = 64 * rhalf + r0 + 8 * (i >> 1), m = cq + 8 * t + (i & 1);
                fin[(long long)m * a.vg * DV + j] = st[t][i];
            }
    }
}

// ------------------------------------------------------------- fp32 path

template <int DK>
struct ScanSimtSmem {
    static constexpr int PK = pitch<float>(DK);
    static constexpr size_t OS = 0;                                       // state tile [64][DK]
    static constexpr size_t OX = align128(OS + sizeof(float) * 64 * PK);  // X [DK][DK]
    static constexpr size_t OY = align128(OX + sizeof(float) * DK * PK);  // Y tile [64][DK]
    static constexpr size_t bytes() { return OY + sizeof(float) * 64 * PK; }
};

// One CTA per (sequence x 64-row dv tile, head); warp w owns state rows 16w..16w+15.
template <int DK, int DV>
__global__ void __launch_bounds__(128) k_scan_simt(ScanArgs a) {
    using S = ScanSimtSmem<DK>;
    constexpr int NT = DK / 8;
    const int jt = blockIdx.x % (DV / 64), n = blockIdx.x / (DV / 64), h = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5;
    const int j0 = jt * 64;
    extern __shared__ __align__(128) char smem[];
    float* sS = reinterpret_cast<float*>(smem + S::OS);
    float* sX = reinterpret_cast<float*>(smem + S::OX);
    float* sY = reinterpret_cast<float*>(smem + S::OY);

    float acc[NT][4];
    const float* init = a.init ? a.init + state_off(a, n, h, DK, DV) : nullptr;
#pragma unroll
    for (int t = 0; t < NT; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int r = j0 + 16 * warp + frag_row(i), m = frag_col(t, i);
            acc[t][i] = init ? init[(long long)m * a.vg * DV + r] : 0.f;
        }

    long long start, len;
    scan_seq_range(a, n, start, len);
    const int s0 = a.seq_first[n];
    int nch = (int)((len + kChunk - 1) / kChunk);
    if (s0 + nch > a.slots) nch = a.slots - s0 > 0 ? a.slots - s0 : 0;

    for (int it = 0; it < nch; ++it) {
        const int c = a.reverse ? nch - 1 - it : it;
        const long long idx = (long long)(s0 + c) * a.H + h;
        const int L = (int)(len - (long long)c * kChunk < kChunk ? len - (long long)c * kChunk : kChunk);
        const float gam = expf(__ldg(a.Gb + idx * 64 + L - 1));
        load_tile_async<float>(sX, S::PK, reinterpret_cast<const float*>(a.X) + idx * DK * DK, DK, DK, DK, DK, tid,
                               128);
        load_tile_async<float>(sY, S::PK, reinterpret_cast<const float*>(a.Y) + (idx * DV + j0) * DK, DK, 64, DK, 64,
                               tid, 128);
        cp_async_commit();
        frag_store<float, NT>(sS, S::PK, 16 * warp, 0, acc);
        float* out = reinterpret_cast<float*>(a.Sout) + (idx * DV + j0) * DK;
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i)
                out[(long long)(16 * warp + frag_row(i)) * DK + frag_col(t, i)] = acc[t][i];
        cp_async_wait<0>();
        __syncthreads();
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i)
                acc[t][i] = fmaf(gam, acc[t][i], sY[(16 * warp + frag_row(i)) * S::PK + frag_col(t, i)]);
        warp_gemm<true, true, NT>(acc, sS, S::PK, sX, S::PK, 16 * warp, 0, DK);
        __syncthreads();
    }
    if (a.fin) {
        float* fin = a.fin + state_off(a, n, h, DK, DV);
#pragma unroll
        for (int t = 0; t < NT; ++t)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = j0 + 16 * warp + frag_row(i), m = frag_col(t, i);
                fin[(long long)m * a.vg * DV + r] = acc[t][i];
            }
    }
}

// ---------------------------------------------------------------- launcher

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    if (!fn) {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// 2D bf16 view [rows][cols] with 128-byte swizzle and a [box_rows][64] box.
static bool make_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t gstride[1] = {(cuuint64_t)cols * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same view for other kernels (scan_wide.cu).
bool make_bf16_map(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows) {
    return make_map(m, base, rows, cols, box_rows);
}

// A [tokens][heads][cols] bf16 token tensor as a 3D view with a {64 columns, 1 head, 64 tokens}
// box (one head's 64-token chunk, 128-byte rows, 128-byte swizzle).
bool make_bf16_token_map(CUtensorMap* m, const void* base, long long tokens, int heads, int cols) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t gdim[3] = {(cuuint64_t)cols, (cuuint64_t)heads, (cuuint64_t)(tokens > 0 ? tokens : 1)};
    cuuint64_t gstride[2] = {(cuuint64_t)cols * 2, (cuuint64_t)heads * cols * 2};
    cuuint32_t box[3] = {64, 1, 64};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), gdim, gstride, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DK, int DV, bool XMN, int YM>
static cudaError_t run_scan_tc_split(const ScanArgs& a, long long pairs, cudaStream_t s) {
    using S = ScanSplitSmem<DK, DV, YM>;
    CUtensorMap tx, tf, ts, tt;
    if (!a.F || !a.tok || !make_map(&tx, a.X, pairs * DK, DK, DK) || !make_map(&ts, a.Sout, pairs * DV, DK, 64))
        return cudaErrorInvalidValue;
    if (YM == 1) {
        // Z^T [pairs * dk][64] with a [dk][64] box; dO [tokens][heads][dv], {64, 1, 64} boxes
        if (!make_map(&tf, a.F, pairs * DK, 64, DK) || !make_bf16_token_map(&tt, a.tok, a.Ttot, a.H, DV))
            return cudaErrorInvalidValue;
    } else {
        // U_s^T [pairs * dv][64] with a [64][64] box; keys [tokens][key heads][dk], {64, 1, 64} boxes
        if (!make_map(&tf, a.F, pairs * DV, 64, 64) || !make_bf16_token_map(&tt, a.tok, a.Ttot, a.H / a.vg, DK))
            return cudaErrorInvalidValue;
    }
    cudaError_t e = cudaFuncSetAttribute(k_scan_tc_split<DK, DV, XMN, YM>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)S::bytes());
    if (e) return e;
    k_scan_tc_split<DK, DV, XMN, YM><<<dim3(2 * a.N, a.H), 256, S::bytes(), s>>>(a, tx, tf, ts, tt);
    return cudaGetLastError();
}

template <int DK, int DV, bool XMN>
static cudaError_t run_scan_tc(const ScanArgs& a, long long pairs, cudaStream_t s) {
    if constexpr (DK == 128 && DV == 128) {
        // the tcgen05 path forms its additive term in the scan: C^T = dO^T Z (reverse, Atilde read
        // MN-major) or B^T = U_s^T K (forward)
        if (a.ym != (XMN ? 1 : 2)) return cudaErrorInvalidValue;
        return run_scan_tc_split<DK, DV, XMN, XMN ? 1 : 2>(a, pairs, s);
    }
    if (a.ym) return cudaErrorInvalidValue;
    using S = ScanTcSmem<DK, DV>;
    CUtensorMap tx, ty, ts;
    if (!make_map(&tx, a.X, pairs * DK, DK, DK) || !make_map(&ty, a.Y, pairs * DV, DK, DV) ||
        !make_map(&ts, a.Sout, pairs * DV, DK, DV))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_scan_tc<DK, DV, XMN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)S::bytes());
    if (e) return e;
    k_scan_tc<DK, DV, XMN><<<dim3(a.N, a.H), 256, S::bytes(), s>>>(a, tx, ty, ts);
    return cudaGetLastError();
}

template <int DK, int DV>
static cudaError_t run_scan_simt(const ScanArgs& a, cudaStream_t s) {
    using S = ScanSimtSmem<DK>;
    cudaError_t e = cudaFuncSetAttribute(k_scan_simt<DK, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)S::bytes());
    if (e) return e;
    k_scan_simt<DK, DV><<<dim3((DV / 64) * a.N, a.H), 128, S::bytes(), s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_scan(const ScanArgs& a, bool is_bf16, int dk, int dv, long long pairs, cudaStream_t s) {
    if (dk == 256) return is_bf16 && dv == 64 ? launch_scan_wide(a, s) : cudaErrorInvalidValue;
#define COMBA_SCAN(DK, DV)                                                                          \
    if (dk == DK && dv == DV)                                                                        \
        return !is_bf16 ? run_scan_simt<DK, DV>(a, s)                                                \
                        : (a.x_mn ? run_scan_tc<DK, DV, true>(a, pairs, s) : run_scan_tc<DK, DV, false>(a, pairs, s));
    COMBA_SCAN(128, 128) COMBA_SCAN(128, 64) COMBA_SCAN(64, 128) COMBA_SCAN(64, 64)
#undef COMBA_SCAN
    return cudaErrorInvalidValue;
}

size_t scan_smem_bytes(bool is_bf16, int dk, int dv) {
    if (dk == 256) return is_bf16 && dv == 64 ? scan_wide_smem_bytes() : 0;
    if (is_bf16) {
        if (dk == 128)   // both directions of the row split take the same shared memory
            return dv == 128 ? ScanSplitSmem<128, 128, 1>::bytes() : ScanTcSmem<128, 64>::bytes();
        return dv == 128 ? ScanTcSmem<64, 128>::bytes() : ScanTcSmem<64, 64>::bytes();
    }
    return dk == 128 ? ScanSimtSmem<128>::bytes() : ScanSimtSmem<64>::bytes();
}

}  // namespace comba
