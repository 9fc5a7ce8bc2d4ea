// Launch parameters shared by the chunk kernels and the C-ABI layer.
#pragma once

#include <stddef.h>
#include <stdint.h>

#include "common.cuh"

namespace comba {

struct ChunkParams {
    // problem
    int B, T, H, dk, dv, N;
    long long Ttot;          // packed tokens (B*T, or T when varlen)
    const int32_t* cu;       // device [N+1] or null (dense: sequence n starts at n*T)
    int slots;               // chunk slots (upper bound on the number of chunks)

    // forward inputs / outputs
    const void* q;
    const void* k;
    const void* v;
    const float* alpha;
    const float* beta;
    const float* b;          // [H] or null (b = 1)
    const float* d;          // [H]
    const float* h0;         // [N,H,dk,dv] or null
    void* o;
    float* hT;

    // backward inputs / outputs
    const void* dO;
    const float* dhT;
    void* dq;
    void* dkk;
    void* dvv;
    float* dalpha;
    float* dbeta;
    float* db;
    float* dd;
    float* dh0;

    // workspace views (per (slot, head) pair idx = slot*H + h)
    SlotInfo* slot_info;     // [slots]
    int* seq_first;          // [N+1] first slot of each sequence
    void* Wb;                // [pairs][64][dk]  storage type
    void* Ub;                // [pairs][64][dv]
    float* Gb;               // [pairs][64]      chunk-local log-cumsum of alpha
    void* Mb;                // [pairs][64][64]  UT inverse, storage type (backward only)
    void* Hb;                // [pairs][dk][dv]  state at chunk start (storage type)
    void* Eb;                // [pairs][64][dv]  U - W H
    void* dHb;               // [pairs][dk][dv]  dL/dH at chunk end
    void* dEb;               // [pairs][64][dv]
    float* part;             // [pairs][2]       per-chunk db, dd partial sums

    // optional stage-boundary events (instrumentation)
    cudaEvent_t* ev;
    int nev;
};

// Record stage-boundary event i on stream s when instrumentation is on.
inline void mark(const ChunkParams& p, int i, cudaStream_t s) {
    if (p.ev && i < p.nev) cudaEventRecord(p.ev[i], s);
}

// Kernel launchers (one translation unit each); return cudaGetLastError().
cudaError_t launch_chunk_map(const ChunkParams& p, cudaStream_t s);
// Stage events: launch_fwd marks ev0 before prep, ev0+1 before the scan, ev0+2 before the
// output (forward only) and ev0+3 after the last kernel; launch_bwd marks ev0 before the
// reverse scan, ev0+1 before the local gradients, ev0+2 before the head reduction, ev0+3 after.
cudaError_t launch_fwd(const ChunkParams& p, bool is_bf16, bool for_backward, cudaStream_t s, int ev0);
cudaError_t launch_bwd(const ChunkParams& p, bool is_bf16, cudaStream_t s, int ev0);
size_t fwd_smem_bytes(int kernel, bool is_bf16, int dk, int dv);
size_t bwd_smem_bytes(int kernel, bool is_bf16, int dk, int dv);
cudaError_t launch_recurrent_step(int Bd, int H, int dk, int dv, bool is_bf16, const void* q, const void* k,
                                  const void* v, const float* alpha, const float* beta, const float* b,
                                  const float* d, float* state, void* o, cudaStream_t s);

}  // namespace comba
