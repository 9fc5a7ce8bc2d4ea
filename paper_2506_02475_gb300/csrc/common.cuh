// Shared device helpers for the Comba chunk kernels (sm_103a).
//
// Tiles live in shared memory in the storage type T of the call (bf16 or
// fp32), row-major with a 16-byte pad per row.  Products of tiles are formed
// warp by warp on 16 x (8*NT) output blocks held in registers in the
// accumulator-fragment layout of the m16n8k16 tensor-core MMA:
//   lane = 4*g + q;  element i of n-tile t sits at
//   row  m0 + g + 8*(i >> 1),  column  n0 + 8*t + 2*q + (i & 1).
// For bf16 tiles the product runs on the tensor cores (ldmatrix + mma.sync,
// fp32 accumulation).  For fp32 tiles the same fragment positions are
// accumulated with fp32 FMAs, so every kernel has one body for both types.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace comba {

typedef __nv_bfloat16 bf16;

constexpr int kChunk = 64;  // chunk length C

// Feedback strength btilde_t relative to b beta_t: 1 (SPLR), or 2 alpha_t for the
// Comba-iplr transition alpha_t (I - 2 btilde_t k_t k_t^T).
__host__ __device__ __forceinline__ float feedback_scale(int iplr, float alpha) { return iplr ? 2.f * alpha : 1.f; }

// ------------------------------------------------------------------ scalars

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(bf16 x) { return __bfloat162float(x); }

template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float x) { return __float2bfloat16_rn(x); }

// Row pitch (elements) of a shared tile with `cols` columns: 16 bytes of pad
// keep ldmatrix row addresses and FMA-path row reads on distinct banks.
template <typename T> __host__ __device__ constexpr int pitch(int cols) { return cols + 16 / (int)sizeof(T); }

// ------------------------------------------------------------ copy helpers

// Copy `rows` x `cols` elements of a strided global matrix into a shared tile,
// zero-filling rows >= valid_rows.  16-byte vectors; cols * sizeof(T) % 16 == 0.
template <typename T>
__device__ __forceinline__ void load_tile(T* s, int sp, const T* g, long long gstride, int rows, int cols,
                                          int valid_rows, int tid, int nthreads) {
    constexpr int V = 16 / sizeof(T);
    const int vpr = cols / V;
    for (int idx = tid; idx < rows * vpr; idx += nthreads) {
        const int r = idx / vpr, c = (idx % vpr) * V;
        uint4 val = make_uint4(0, 0, 0, 0);
        if (r < valid_rows) val = *reinterpret_cast<const uint4*>(g + (long long)r * gstride + c);
        *reinterpret_cast<uint4*>(s + r * sp + c) = val;
    }
}

// ---------------------------------------------------- tensor-core fragments

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------ asynchronous copies

// 16-byte global->shared copy that bypasses registers (cp.async); when
// `valid` is false nothing is read and the 16 bytes are zero-filled.
__device__ __forceinline__ void cp_async16(void* s, const void* g, bool valid) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(smem_u32(s)), "l"(g),
                 "r"(valid ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// Asynchronous version of load_tile (rows >= valid_rows are zero-filled);
// completes at the caller's cp_async_wait + __syncthreads.
template <typename T>
__device__ __forceinline__ void load_tile_async(T* s, int sp, const T* g, long long gstride, int rows, int cols,
                                                int valid_rows, int tid, int nthreads) {
    constexpr int V = 16 / sizeof(T);
    const int vpr = cols / V;
    for (int idx = tid; idx < rows * vpr; idx += nthreads) {
        const int r = idx / vpr, c = (idx % vpr) * V;
        const bool ok = r < valid_rows;
        cp_async16(s + r * sp + c, ok ? (const void*)(g + (long long)r * gstride + c) : (const void*)g, ok);
    }
}

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(smem_u32(p)));
}

__device__ __forceinline__ void mma_bf16(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// acc[NT][4] += A(m0.., 0..K) * B(0..K, n0..)
//   AK: A is stored [m][k] (k contiguous); otherwise stored transposed [k][m].
//   BK: B is stored [n][k] (k contiguous); otherwise stored [k][n].
//   lda/ldb are row pitches in elements.  K % 16 == 0, NT even.
template <bool AK, bool BK, int NT>
__device__ __forceinline__ void warp_gemm(float (&acc)[NT][4], const bf16* sA, int lda, const bf16* sB, int ldb,
                                          int m0, int n0, int K) {
    static_assert(NT % 2 == 0, "NT must be even");
    const int lane = threadIdx.x & 31;
    const int j = lane >> 3, r = lane & 7;
#pragma unroll 2
    for (int k0 = 0; k0 < K; k0 += 16) {
        uint32_t a[4];
        if (AK) {
            ldsm_x4(a, sA + (m0 + (lane & 15)) * lda + k0 + ((lane >> 4) << 3));
        } else {
            ldsm_x4_t(a, sA + (k0 + r + ((j >> 1) << 3)) * lda + m0 + ((j & 1) << 3));
        }
#pragma unroll
        for (int t = 0; t < NT; t += 2) {
            uint32_t b[4];
            if (BK) {
                ldsm_x4(b, sB + (n0 + 8 * t + r + ((j >> 1) << 3)) * ldb + k0 + ((j & 1) << 3));
            } else {
                ldsm_x4_t(b, sB + (k0 + r + ((j & 1) << 3)) * ldb + n0 + 8 * t + ((j >> 1) << 3));
            }
            mma_bf16(acc[t], a, b[0], b[1]);
            mma_bf16(acc[t + 1], a, b[2], b[3]);
        }
    }
}

// fp32 tiles: same fragment positions, fp32 FMAs.
template <bool AK, bool BK, int NT>
__device__ __forceinline__ void warp_gemm(float (&acc)[NT][4], const float* sA, int lda, const float* sB, int ldb,
                                          int m0, int n0, int K) {
    const int lane = threadIdx.x & 31;
    const int g = lane >> 2, q = lane & 3;
    const int r0 = m0 + g, r1 = r0 + 8;
#pragma unroll 4
    for (int k = 0; k < K; ++k) {
        const float a0 = AK ? sA[r0 * lda + k] : sA[k * lda + r0];
        const float a1 = AK ? sA[r1 * lda + k] : sA[k * lda + r1];
#pragma unroll
        for (int t = 0; t < NT; ++t) {
            const int c = n0 + 8 * t + 2 * q;
            const float b0 = BK ? sB[c * ldb + k] : sB[k * ldb + c];
            const float b1 = BK ? sB[(c + 1) * ldb + k] : sB[k * ldb + c + 1];
            acc[t][0] = fmaf(a0, b0, acc[t][0]);
            acc[t][1] = fmaf(a0, b1, acc[t][1]);
            acc[t][2] = fmaf(a1, b0, acc[t][2]);
            acc[t][3] = fmaf(a1, b1, acc[t][3]);
        }
    }
}

template <int NT>
__device__ __forceinline__ void zero(float (&acc)[NT][4]) {
#pragma unroll
    for (int t = 0; t < NT; ++t) acc[t][0] = acc[t][1] = acc[t][2] = acc[t][3] = 0.f;
}

// Fragment coordinates (relative to the block origin).
__device__ __forceinline__ int frag_row(int i) { return ((threadIdx.x & 31) >> 2) + ((i >> 1) << 3); }
__device__ __forceinline__ int frag_col(int t, int i) { return 8 * t + 2 * (threadIdx.x & 3) + (i & 1); }

// Write a fragment block into a shared tile of type T.
template <typename T, int NT>
__device__ __forceinline__ void frag_store(T* s, int sp, int m0, int n0, const float (&acc)[NT][4]) {
#pragma unroll
    for (int t = 0; t < NT; ++t)
#pragma unroll
        for (int i = 0; i < 4; ++i) s[(m0 + frag_row(i)) * sp + n0 + frag_col(t, i)] = from_f<T>(acc[t][i]);
}

// Sum over the 4 lanes of a quad (lanes sharing fragment rows).
__device__ __forceinline__ float quad_sum(float x) {
    x += __shfl_xor_sync(0xffffffffu, x, 1);
    x += __shfl_xor_sync(0xffffffffu, x, 2);
    return x;
}
// Sum over the 8 lanes sharing a quad position (lanes sharing fragment columns).
__device__ __forceinline__ float col_sum8(float x) {
    x += __shfl_xor_sync(0xffffffffu, x, 4);
    x += __shfl_xor_sync(0xffffffffu, x, 8);
    x += __shfl_xor_sync(0xffffffffu, x, 16);
    return x;
}

// ----------------------------------------------------------------- chunks

// Per chunk slot: first token, length (0 = unused slot), sequence, chunk index.
struct SlotInfo {
    int start;
    int len;
    int seq;
    int idx;
};

// Shared-memory carve-up: bump allocator with 128-byte alignment.
struct SmemCarver {
    char* base;
    size_t off;
    __device__ explicit SmemCarver(void* b) : base(static_cast<char*>(b)), off(0) {}
    template <typename T>
    __device__ T* take(size_t n) {
        off = (off + 127) & ~size_t(127);
        T* p = reinterpret_cast<T*>(base + off);
        off += n * sizeof(T);
        return p;
    }
};
__host__ __device__ constexpr size_t carve_bytes(size_t off, size_t bytes) { return ((off + 127) & ~size_t(127)) + bytes; }
__host__ __device__ constexpr size_t align128(size_t off) { return (off + 127) & ~size_t(127); }

// Inclusive prefix sum of log(alpha) over a chunk (warp-wide; the lane passes its
// alpha values at positions lane and lane + 32, already loaded).  Positions >= L
// contribute 0, so G stays finite there.  Writes G[p] and Gm1[p] = G[p-1] (Gm1[0] = 0).
__device__ __forceinline__ void chunk_log_cumsum_vals(float a0, float a1, int L, float* G, float* Gm1) {
    const int lane = threadIdx.x & 31;
    float x0 = lane < L ? logf(a0) : 0.f;
    float x1 = lane + 32 < L ? logf(a1) : 0.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y0 = __shfl_up_sync(0xffffffffu, x0, o);
        const float y1 = __shfl_up_sync(0xffffffffu, x1, o);
        if (lane >= o) { x0 += y0; x1 += y1; }
    }
    const float tot0 = __shfl_sync(0xffffffffu, x0, 31);
    x1 += tot0;
    G[lane] = x0;
    G[lane + 32] = x1;
    const float p0 = __shfl_up_sync(0xffffffffu, x0, 1);
    const float p1 = __shfl_up_sync(0xffffffffu, x1, 1);
    Gm1[lane] = lane == 0 ? 0.f : p0;
    Gm1[lane + 32] = lane == 0 ? tot0 : p1;
}

// ------------------------------------------- sm_100-family async primitives
// mbarrier, TMA (cp.async.bulk.tensor), and tcgen05 (5th-generation tensor
// cores with TMEM accumulators).  Every wait is bounded in time (%globaltimer,
// nanoseconds) and reports failure instead of hanging.  A kernel's own waits
// take the per-call limit of its launch parameters (kDefaultWaitNs unless the
// caller sets one, at most kMaxWaitNs); a kernel that gave up then lets every copy and product it
// has in flight finish with mbar_drain, whose limit is fixed, so that nothing
// still writes its shared memory or TMEM when the kernel releases them.

constexpr uint32_t kDefaultWaitNs = 1000000000u;   // 1 s
constexpr uint32_t kDrainWaitNs = 2000000000u;     // 2 s
// Limits are at most kMaxWaitNs, so that the low 32 bits of %globaltimer measure them
// without ambiguity (they wrap every 4.29 s).
constexpr uint32_t kMaxWaitNs = 4000000000u;

__device__ __forceinline__ uint32_t global_ns_lo() {
    uint32_t t;
    asm volatile("{\n .reg .u64 t64;\n mov.u64 t64, %%globaltimer;\n cvt.u32.u64 %0, t64;\n}\n" : "=r"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t mbar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(mbar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_fence_init() { asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory"); }
__device__ __forceinline__ void mbar_expect_tx(uint32_t mbar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(mbar), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t mbar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(mbar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Wait for the phase of parity `parity` to complete; false once `limit_ns` have passed without it.
// The clock is first read after 64 polls (a wait that ends sooner never touches it), then every 64
// polls, which keeps both the fast path and the loop's registers lean.
__device__ __forceinline__ bool mbar_wait(uint32_t mbar, uint32_t parity, uint32_t limit_ns) {
    uint32_t t0 = 0;
    for (uint32_t i = 1;; ++i) {
        if (mbar_try(mbar, parity)) return true;
        if ((i & 63) == 0) {
            const uint32_t t = global_ns_lo();
            if (i == 64)
                t0 = t;
            else if (t - t0 > limit_ns)
                return false;
        }
    }
}
// A wait bounded by a poll count instead of the clock, for the tensor-core completion waits of the
// chunk kernels (prep, output, local gradients), where reading %globaltimer anywhere in the loop
// measurably slows the kernel: one try_wait takes at least ~16 ns, so `limit_ns / 16` polls
// last no less than the limit.
__device__ __forceinline__ bool mbar_wait_polls(uint32_t mbar, uint32_t parity, uint32_t limit_ns) {
    const long long polls = (long long)(limit_ns >> 4) + 1;
    for (long long it = 0; it < polls; ++it)
        if (mbar_try(mbar, parity)) return true;
    return false;
}
// The wait of a kernel's give-up path: its copies and products in flight must land first.
__device__ __forceinline__ bool mbar_drain(uint32_t mbar, uint32_t parity) {
    return mbar_wait(mbar, parity, kDrainWaitNs);
}

// 2D tiled TMA load of box (x, y) into shared memory, completing on `mbar`.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int x, int y, uint32_t mbar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n"
        ::"r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(mbar)
        : "memory");
}

// 3D tiled TMA load of box (x, y, z) into shared memory, completing on `mbar`.
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const void* tmap, int x, int y, int z, uint32_t mbar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];\n"
        ::"r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(z), "r"(mbar)
        : "memory");
}

__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }

// Zero rows [from, 64) of `halves` consecutive [64][128 B] tiles and make the writes visible to
// the tensor core (one thread; kept out of line, off the scans' per-chunk issue path).
static __device__ __noinline__ void zero_tile_rows(uint8_t* tile, int from, int halves) {
    for (int half = 0; half < halves; ++half)
        for (int e = from * 8; e < 64 * 8; ++e)
            *reinterpret_cast<uint4*>(tile + half * 64 * 128 + e * 16) = make_uint4(0, 0, 0, 0);
    fence_async_smem();
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

// TMEM allocation (whole warp): writes the base address to shared memory.
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(dst_smem), "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols) : "memory");
}

// Instruction descriptor, kind::f16: bf16 x bf16 -> fp32, both operands K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem]^T, issued by one thread.
__device__ __forceinline__ void tc_mma_bf16(uint32_t tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                            uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n"
        ::"r"(tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t mbar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(mbar)
                 : "memory");
}

// 32 consecutive fp32 accumulator columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Descriptors of the 16-deep K step `ks` of a bf16 operand tile in the 128-byte
// swizzle layout.  K-major tile: K split in 64-element halves, each a
// [rows][128 B] block (rows = the tile's allocated M or N extent).  MN-major
// tile: M/N split in 64-element halves, each a [krows][128 B] block (krows =
// the tile's allocated K extent); consecutive K rows are 128 B apart.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFF);
    d |= (uint64_t)((lbo >> 4) & 0x3FFF) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFF) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
__device__ __forceinline__ uint64_t desc_kmajor(uint32_t base, int rows, int ks) {
    return smem_desc(base + (ks >> 2) * rows * 128 + (ks & 3) * 32, 16, 1024);
}
__device__ __forceinline__ uint64_t desc_mnmajor(uint32_t base, int krows, int ks) {
    return smem_desc(base + ks * 2048, krows * 128, 1024);
}

// Step from the k-step-0 descriptor of a tile to that of k-step ks, in the descriptor's
// address units (16 bytes): a K-major tile advances 32 B inside a 64-element K half and
// rows x 128 B from one half to the next; an MN-major one advances 16 K-rows x 128 B.  Adding
// it to the 64-bit descriptor touches only the 14-bit start-address field, which cannot carry
// out: shared-memory addresses stay below 2^18 bytes.  With the descriptors formed once per
// product, issuing a k-step costs two 64-bit adds instead of rebuilding both descriptors.
template <bool MN>
__device__ __forceinline__ uint64_t desc_step(int ext, int ks) {
    return MN ? (uint64_t)(ks * 128) : (uint64_t)((ks >> 2) * ext * 8 + (ks & 3) * 2);
}

// D[tmem, M x N fp32] (+)= A[M x K] * B[K x N] on bf16 smem tiles, issued by one thread.
// AMN/BMN select MN-major operand tiles; a_ext/b_ext are the tiles' allocated row counts (see
// above).  K % 16 == 0.
template <int M, bool AMN, bool BMN>
__device__ __forceinline__ void tc_gemm_mk(uint32_t tmem, uint32_t a, int a_ext, uint32_t b, int b_ext, int N, int K,
                                           bool accumulate) {
    const uint32_t idesc = idesc_bf16_f32(M, N) | (AMN ? 1u << 15 : 0u) | (BMN ? 1u << 16 : 0u);
    const uint64_t a0 = AMN ? desc_mnmajor(a, a_ext, 0) : desc_kmajor(a, a_ext, 0);
    const uint64_t b0 = BMN ? desc_mnmajor(b, b_ext, 0) : desc_kmajor(b, b_ext, 0);
#pragma unroll
    for (int ks = 0; ks < K / 16; ++ks)
        tc_mma_bf16(tmem, a0 + desc_step<AMN>(a_ext, ks), b0 + desc_step<BMN>(b_ext, ks), idesc,
                    (accumulate || ks > 0) ? 1u : 0u);
}
// M = 128: D row m in TMEM lane m.
template <bool AMN, bool BMN>
__device__ __forceinline__ void tc_gemm(uint32_t tmem, uint32_t a, int a_ext, uint32_t b, int b_ext, int N, int K,
                                        bool accumulate) {
    tc_gemm_mk<128, AMN, BMN>(tmem, a, a_ext, b, b_ext, N, K, accumulate);
}
// M = 64: D row m lives in TMEM lane 32*(m/16) + m%16 (lanes 0-15 of each warp's quadrant),
// column n in column n.
template <bool AMN, bool BMN>
__device__ __forceinline__ void tc_gemm_m64(uint32_t tmem, uint32_t a, int a_ext, uint32_t b, int b_ext, int N, int K,
                                            bool accumulate) {
    tc_gemm_mk<64, AMN, BMN>(tmem, a, a_ext, b, b_ext, N, K, accumulate);
}

// 16 consecutive fp32 accumulator columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Issue a 16-column TMEM load without waiting; complete with tmem_wait_ld().
__device__ __forceinline__ void tmem_ld16_async(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory"); }

// Byte offset of element (row, k) of a K-major bf16 tile in the 128-byte swizzle
// layout: K is split in halves of 64 elements, each a [rows][128 B] block.
__host__ __device__ constexpr uint32_t sw128_offset(int row, int k, int rows) {
    return (uint32_t)((k >> 6) * rows * 128 + row * 128 + ((((k & 63) >> 3) ^ (row & 7)) << 4) + (k & 7) * 2);
}

// (I + A)^{-1} for a 64 x 64 strictly-lower A (fp32, pitch 65), by blocks of 16:
// the four diagonal blocks by forward substitution (one lane per column), then
// the off-diagonal blocks level by level, X_ij = -X_ii sum_{k=j}^{i-1} A_ik X_kj.
// 128 threads; `tmp` holds 3 x 16 x 17 floats.  Rows past a short chunk have
// A = 0 and come out as identity rows.
__device__ __forceinline__ void unit_lower_inverse64(const float* A, float* M, float* tmp, int tid) {
    for (int e = tid; e < 64 * 64; e += 128) {
        const int r = e >> 6, c = e & 63;
        M[r * 65 + c] = (r == c) ? 1.f : 0.f;
    }
    __syncthreads();
    if (tid < 64) {
        const int cj = tid, end = (tid & ~15) + 16;
        for (int r = cj + 1; r < end; ++r) {
            float s = 0.f;
            for (int i = cj; i < r; ++i) s = fmaf(A[r * 65 + i], M[i * 65 + cj], s);
            M[r * 65 + cj] = -s;
        }
    }
    __syncthreads();
    for (int lvl = 1; lvl < 4; ++lvl) {
        const int nb = 4 - lvl;
        for (int e = tid; e < nb * 256; e += 128) {
            const int blk = e >> 8, r = (e >> 4) & 15, c = e & 15;
            const int bj = blk, bi = blk + lvl;
            float s = 0.f;
            for (int i = 16 * bj; i < 16 * bi; ++i) s = fmaf(A[(16 * bi + r) * 65 + i], M[i * 65 + 16 * bj + c], s);
            tmp[blk * 272 + r * 17 + c] = s;
        }
        __syncthreads();
        for (int e = tid; e < nb * 256; e += 128) {
            const int blk = e >> 8, r = (e >> 4) & 15, c = e & 15;
            const int bj = blk, bi = blk + lvl;
            float s = 0.f;
#pragma unroll 4
            for (int i = 0; i < 16; ++i) s = fmaf(M[(16 * bi + r) * 65 + 16 * bi + i], tmp[blk * 272 + i * 17 + c], s);
            M[(16 * bi + r) * 65 + 16 * bj + c] = -s;
        }
        __syncthreads();
    }
}

// Row pitches (floats) of the tcgen05 prep kernel's inverse: A transposed (At) and M.  At's
// pitch is 8 (mod 32) and M's 4 (mod 32), so the tf32 fragment loads below (lanes g = 0..7 along
// one index, q = 0..3 along the other) fall in distinct banks: At and M as A operands, M as a B
// operand in two lanes per bank at most.
constexpr int kAtPitch = 72, kMPitch = 68;

// Column j (of 16) of (I + A_bb)^{-1} for the 16 x 16 diagonal block starting at B0, by
// forward substitution in registers: M[r2][j] = delta - sum_{r < r2} A[r2][r] M[r][j].
// At is A transposed (pitch kAtPitch): its row r holds column r of A, zero at and above r.
template <int B0>
__device__ __forceinline__ void unit_lower_inverse_diag16(const float* At, float* M, int pm, int j) {
    float s[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) s[r] = 0.f;
#pragma unroll
    for (int r = 0; r < 16; ++r) {
        const float x = r == j ? 1.f : (r < j ? 0.f : -s[r]);
        M[(B0 + r) * pm + B0 + j] = x;
#pragma unroll
        for (int g = (r + 1) >> 2; g < 4; ++g) {
            const float4 a = *reinterpret_cast<const float4*>(At + (B0 + r) * kAtPitch + B0 + 4 * g);
            s[4 * g + 0] = fmaf(a.x, x, s[4 * g + 0]);
            s[4 * g + 1] = fmaf(a.y, x, s[4 * g + 1]);
            s[4 * g + 2] = fmaf(a.z, x, s[4 * g + 2]);
            s[4 * g + 3] = fmaf(a.w, x, s[4 * g + 3]);
        }
    }
}

// fp32 -> tf32 (round to nearest, ties away) for the tf32 tile products below.
__device__ __forceinline__ uint32_t to_tf32(float x) {
    uint32_t r;
    asm("cvt.rna.tf32.f32 %0, %1;\n" : "=r"(r) : "f"(x));
    return r;
}
// d += a b on one m16n8k8 tile, tf32 operands and fp32 accumulators.  Fragments (g = lane / 4,
// q = lane % 4): a = A[g][q], A[g + 8][q], A[g][q + 4], A[g + 8][q + 4]; b = B[q][g], B[q + 4][g];
// d = D[g][2 q], D[g][2 q + 1], D[g + 8][2 q], D[g + 8][2 q + 1].
__device__ __forceinline__ void mma_tf32(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k8.row.col.f32.tf32.tf32.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// (I + A)^{-1} for a strictly lower 64 x 64 A over 256 threads, in three levels: the four
// 16 x 16 diagonal blocks by forward substitution (warps 0..3, one block each, a column per
// lane, fp32), then the 32 x 32 blocks M10 = -M11 (A10 M00) of both halves, then the 64 x 64
// M21 = -M22 (A21 M11).  The two off-diagonal levels are tile products on the tensor cores
// (mma.sync m16n8k8, tf32 operands rounded to nearest, fp32 accumulation): four warps, each
// owning an 8-column block of the level's result, form its block of the inner product, pass it
// from the accumulator layout to the operand layout through a warp-private scratch tile and
// finish the outer product, so each level ends at a single block-wide barrier.  The tf32
// operand rounding (relative 2^-11) lies well below that of the bf16 copies every consumer of M
// takes (2^-8).  At is A transposed with pitch kAtPitch; M has pitch kMPitch and is written in
// full (zeros above the diagonal); T holds 1024 floats of scratch.
__device__ __forceinline__ void unit_lower_inverse64_h16(const float* At, float* M, float* T, int tid) {
    constexpr int pm = kMPitch, pa = kAtPitch;
    if (tid < 128) {
        // warp b solves diagonal block b (lanes 0..15, one column each): no divergence between blocks
        const int j = tid & 31;
        if (j < 16) {
            switch (tid >> 5) {
                case 0: unit_lower_inverse_diag16<0>(At, M, pm, j); break;
                case 1: unit_lower_inverse_diag16<16>(At, M, pm, j); break;
                case 2: unit_lower_inverse_diag16<32>(At, M, pm, j); break;
                default: unit_lower_inverse_diag16<48>(At, M, pm, j); break;
            }
        }
    } else {
        // zeros above the diagonal blocks: rows 0..47, columns past each row's block
        for (int e = tid - 128; e < 64 * 64; e += 128) {
            const int r = e >> 6, c = e & 63;
            if ((c >> 4) > (r >> 4)) M[r * pm + c] = 0.f;
        }
    }
    __syncthreads();
    const int warp = tid >> 5, g = (tid >> 2) & 7, q = tid & 3;
    if (warp < 4) {
        // level 1: half h (rows and columns o1 .. o1 + 31), column block nt of M10 (8 columns)
        const int o1 = 32 * (warp >> 1), nt = warp & 1, c0 = o1 + 8 * nt;
        float* Tw = T + warp * 128;   // [16][8]: T1's column block
        float d[4] = {0.f, 0.f, 0.f, 0.f};
        // T1 = A10 M00; M00 is lower, so its rows above the block's first column are zero
        for (int ks = nt; ks < 2; ++ks) {
            const int k = o1 + 8 * ks + q;
            const uint32_t a[4] = {to_tf32(At[k * pa + o1 + 16 + g]), to_tf32(At[k * pa + o1 + 24 + g]),
                                   to_tf32(At[(k + 4) * pa + o1 + 16 + g]), to_tf32(At[(k + 4) * pa + o1 + 24 + g])};
            mma_tf32(d, a, to_tf32(M[k * pm + c0 + g]), to_tf32(M[(k + 4) * pm + c0 + g]));
        }
        *reinterpret_cast<float2*>(Tw + g * 8 + 2 * q) = make_float2(d[0], d[1]);
        *reinterpret_cast<float2*>(Tw + (g + 8) * 8 + 2 * q) = make_float2(d[2], d[3]);
        __syncwarp();
        // M10 = -M11 T1
        float e[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int ks = 0; ks < 2; ++ks) {
            const int k = o1 + 16 + 8 * ks + q;
            const uint32_t a[4] = {to_tf32(M[(o1 + 16 + g) * pm + k]), to_tf32(M[(o1 + 24 + g) * pm + k]),
                                   to_tf32(M[(o1 + 16 + g) * pm + k + 4]), to_tf32(M[(o1 + 24 + g) * pm + k + 4])};
            mma_tf32(e, a, to_tf32(Tw[(8 * ks + q) * 8 + g]), to_tf32(Tw[(8 * ks + q + 4) * 8 + g]));
        }
        const int c = c0 + 2 * q;
        M[(o1 + 16 + g) * pm + c] = -e[0];
        M[(o1 + 16 + g) * pm + c + 1] = -e[1];
        M[(o1 + 24 + g) * pm + c] = -e[2];
        M[(o1 + 24 + g) * pm + c + 1] = -e[3];
    }
    __syncthreads();
    if (warp < 4) {
        // level 2: column block nt of M21 (rows 32..63, columns 8 nt .. + 7), both 16-row tiles
        const int nt = warp;
        float* Tw = T + warp * 256;   // [32][8]: T's column block
        float d[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
        // T = A21 M11; M11 (the top-left 32 x 32 inverse) is lower: rows k < 8 nt of the block are zero
        for (int ks = nt; ks < 4; ++ks) {
            const int k = 8 * ks + q;
            const uint32_t b0 = to_tf32(M[k * pm + 8 * nt + g]), b1 = to_tf32(M[(k + 4) * pm + 8 * nt + g]);
#pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
                const int r = 32 + 16 * mt + g;
                const uint32_t a[4] = {to_tf32(At[k * pa + r]), to_tf32(At[k * pa + r + 8]),
                                       to_tf32(At[(k + 4) * pa + r]), to_tf32(At[(k + 4) * pa + r + 8])};
                mma_tf32(d[mt], a, b0, b1);
            }
        }
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
            *reinterpret_cast<float2*>(Tw + (16 * mt + g) * 8 + 2 * q) = make_float2(d[mt][0], d[mt][1]);
            *reinterpret_cast<float2*>(Tw + (16 * mt + g + 8) * 8 + 2 * q) = make_float2(d[mt][2], d[mt][3]);
        }
        __syncwarp();
        // M21 = -M22 T; M22 is lower: rows 16 mt .. + 15 of it reach column 16 mt + 15 at most
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
            float e[4] = {0.f, 0.f, 0.f, 0.f};
            const int r = 32 + 16 * mt + g;
#pragma unroll
            for (int ks = 0; ks < 2 + 2 * mt; ++ks) {
                const int k = 32 + 8 * ks + q;
                const uint32_t a[4] = {to_tf32(M[r * pm + k]), to_tf32(M[(r + 8) * pm + k]),
                                       to_tf32(M[r * pm + k + 4]), to_tf32(M[(r + 8) * pm + k + 4])};
                mma_tf32(e, a, to_tf32(Tw[(8 * ks + q) * 8 + g]), to_tf32(Tw[(8 * ks + q + 4) * 8 + g]));
            }
            const int c = 8 * nt + 2 * q;
            M[r * pm + c] = -e[0];
            M[r * pm + c + 1] = -e[1];
            M[(r + 8) * pm + c] = -e[2];
            M[(r + 8) * pm + c + 1] = -e[3];
        }
    }
}

}  // namespace comba
