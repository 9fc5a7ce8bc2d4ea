// Shared-memory tile helpers of the tcgen05 kernels (bf16, 128-byte swizzle).
#pragma once

#include "params.cuh"

namespace comba {
namespace tc {

constexpr int D = 128;  // head dim of this path

__device__ __forceinline__ uint4 pack8(const float* v) {
    uint4 r;
    __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]);
    __nv_bfloat162 b = __floats2bfloat162_rn(v[2], v[3]);
    __nv_bfloat162 c = __floats2bfloat162_rn(v[4], v[5]);
    __nv_bfloat162 d = __floats2bfloat162_rn(v[6], v[7]);
    r.x = *reinterpret_cast<uint32_t*>(&a);
    r.y = *reinterpret_cast<uint32_t*>(&b);
    r.z = *reinterpret_cast<uint32_t*>(&c);
    r.w = *reinterpret_cast<uint32_t*>(&d);
    return r;
}
__device__ __forceinline__ void unpack8(uint4 u, float* v) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(h[i]);
        v[2 * i] = f.x;
        v[2 * i + 1] = f.y;
    }
}

// One-barrier MMA completion tracker (all threads keep the same phase).
struct MmaSync {
    uint32_t bar;        // the barrier the products commit to
    uint32_t wbar;       // the barrier waited on: `bar`, or (COMBA_DIAG_STALL) one nothing arrives at
    uint32_t phase;
    uint32_t limit_ns;
    // Thread 0 has issued MMAs; commit, wait everywhere, and report failure uniformly.
    __device__ __forceinline__ bool finish(int tid) {
        if (tid == 0) tc_commit(bar);
        return wait(tid);
    }
    // The same when thread 0 has committed already (tc_commit(bar) right behind its products).
    __device__ __forceinline__ bool wait(int tid) {
        const bool ok = mbar_wait_polls(wbar, phase, limit_ns);
        phase ^= 1;
        const bool any_bad = __syncthreads_or(!ok);
        tc_fence_after();
        return !any_bad;
    }
    // The same two without a block-wide barrier: `ok` comes out uniform over the warp only (the
    // warp-collective TMEM reads that follow need that much), and the caller makes it uniform over
    // the block at its next block-wide barrier, before it issues another product.
    __device__ __forceinline__ bool finish_warp(int tid) {
        if (tid == 0) tc_commit(bar);
        return wait_warp();
    }
    __device__ __forceinline__ bool wait_warp() {
        const bool ok = mbar_wait_polls(wbar, phase, limit_ns);
        phase ^= 1;
        const bool all = __all_sync(0xffffffffu, ok);
        tc_fence_after();
        return all;
    }
    // After a failed finish (the kernel then issues no further product): the commit whose wait
    // gave up covers every product thread 0 has issued, so waiting (again) for that phase means
    // nothing writes TMEM once the kernel releases it.  `phase` has moved past it, and a parity
    // wait on the phase still pending is the right one.  Called by every thread ahead of the
    // kernel's exit barrier.
    __device__ __forceinline__ void drain(int tid) {
        if (tid == 0) mbar_drain(bar, phase ^ 1);
    }
};

// Hand the tiles written so far to the tensor core, with `ok` made uniform over the block.
__device__ __forceinline__ bool publish_ok(bool ok) {
    fence_async_smem();
    tc_fence_before();
    const bool bad = __syncthreads_or(!ok);
    tc_fence_after();
    return !bad;
}

__device__ __forceinline__ void flag_error(const ChunkParams& p) {
    if (p.err) atomicExch(p.err, 1);
}

// Make generic-proxy shared-memory writes visible to the tensor core and order
// prior TMEM reads before the next MMA.
__device__ __forceinline__ void publish_smem() {
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
}

__device__ __forceinline__ void bulk_copy_s2g(void* g, uint32_t s, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;\n" ::"l"(g), "r"(s), "r"(bytes) : "memory");
    asm volatile("cp.async.bulk.commit_group;\n" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all_reads() { asm volatile("cp.async.bulk.wait_group.read 0;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all_done() { asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory"); }
// Bulk tensor stores of a swizzled shared tile (2D: columns x, rows y; 3D: columns x, head y,
// tokens z), completed as one bulk group by bulk_commit.
__device__ __forceinline__ void tma_store_2d(const void* tmap, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];\n"
                 ::"l"(tmap), "r"(x), "r"(y), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void tma_store_3d(const void* tmap, int x, int y, int z, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];\n"
                 ::"l"(tmap), "r"(x), "r"(y), "r"(z), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }

}  // namespace tc
}  // namespace comba
