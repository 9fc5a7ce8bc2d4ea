// Launch parameters shared by the chunk kernels and the C-ABI layer.
#pragma once

#include <stddef.h>
#include <stdint.h>

#include "common.cuh"

namespace comba {

struct ChunkParams {
    // problem
    int B, T, H, dk, dv, N;  // H: value heads; dk, dv: one head's widths
    int vg;                  // value heads per key head (>= 1): head h takes q, k, p, alpha, beta, b, d
                             // of key head h / vg; v, o, dO, dv and the chunk states are per value head
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
    int iplr;                // Comba-iplr: feedback strength 2 alpha b beta instead of b beta
    const float* d;          // [H]
    const void* p;           // Comba-pk feedback vectors [tokens,H,dk] (storage type), or null (p = k)
    const float* d_fb;       // Comba-pk: the per-head d of the correction q - d p, applied to q before
                             // the chunk kernels (which then see d = 0); its share of dp is -d dq
    const float* h0;         // [N,H,dk,dv] or null
    void* o;
    float* hT;

    // backward inputs / outputs
    const void* dO;
    const float* dhT;
    void* dq;
    void* dkk;
    void* dvv;
    void* dpp;               // Comba-pk: dL/dp [tokens,H,dk]
    float* dalpha;
    float* dbeta;
    float* db;
    float* dd;
    float* dh0;

    // workspace views (per (slot, head) pair idx = slot*H + h; with value-head groups on the
    // mma.sync path, W, G and M are stored once per key head, at its first value head's pair)
    SlotInfo* slot_info;     // [slots]
    int* seq_first;          // [N+1] first slot of each sequence
    void* Wb;                // [pairs][64][dk]  WY factor W (storage type)
    void* Ub;                // [pairs][64][dv]  WY factor U
    float* Gb;               // [pairs][64]      chunk-local log-cumsum of alpha
    void* Ab;                // [pairs][dk][dk]  Atilde = -Kbar^T W (forward scan operand)
    void* Bb;                // [pairs][dv][dk]  (Kbar^T U)^T (forward scan additive term; off the
                             //                  tcgen05 path)
    void* Usb;               // [pairs][dv][64]  U_s^T = (Diag(s) U)^T, s_r = gamma_C / gamma_r (tcgen05
                             //                  path: the forward scan forms B^T = U_s^T K itself)
    void* Hb;                // [pairs][dv][dk]  chunk-start state, transposed
    void* Eb;                // [pairs][64][dv]  E = U - W H (saved for the backward)
    void* Mb;                // [pairs][64][64]  UT inverse M (saved for the backward)
    void* ATb;               // [pairs][dk][dk]  Atilde^T (backward scan operand)
    void* Cb;                // [pairs][dv][dk]  ((Qhat - P W)^T dO)^T (backward scan additive term;
                             //                  off the tcgen05 path)
    void* Zb;                // [pairs][dk][64]  Z^T = (Qhat - P W)^T (tcgen05 path), or [pairs][64][dk]
                             //                  Z at head dim 256 (once per key head, at its first value
                             //                  head's pair): the reverse scan forms C^T = dO^T Z itself
    void* dHb;               // [pairs][dv][dk]  dL/dH at chunk end, transposed
    float* part;             // [pairs][2]       per-chunk db, dd partial sums
    int* err;                // device status word (nonzero: a bounded wait gave up)
    uint32_t wait_ns;        // limit of each device-side wait (kDefaultWaitNs unless set)
    int stall;               // COMBA_DIAG_STALL: the tcgen05 chunk kernels' first completion wait runs out

    // optional stage-boundary events (instrumentation)
    cudaEvent_t* ev;
    int nev;
};

// Gate and normalisation prologue / epilogue (gates.cu): raw inputs, the prologue's outputs
// in the workspace, and (backward) the chunk backward's gradients mapped to the raw inputs.
struct GateParams {
    long long rows;          // tokens * H
    int H;
    float eps;
    const void* q;           // raw q, k [tokens, H, dk]
    const void* k;
    const float* g_alpha;    // [tokens, H] gate pre-activations
    const float* g_beta;
    const float* a;          // [H] per-head scalars
    const float* c;
    const float* b_raw;
    void* qh;                // prologue outputs
    void* kh;
    float* alpha;
    float* beta;
    float* bgate;            // [H] sigmoid(b_raw)
    const void* dqh;         // chunk backward outputs (gradients w.r.t. the prologue outputs)
    const void* dkh;
    const float* dalpha;
    const float* dbeta;
    const float* db;
    void* dq;                // gradients w.r.t. the raw inputs
    void* dk;
    float* dg_alpha;
    float* dg_beta;
    float* da;
    float* dc;
    float* db_raw;
    float* da_rows;          // [tokens, H] per-row contributions, summed per head in a fixed order
    float* dc_rows;
    float* da_part;          // [H, ceil(tokens / 64)] token-block sums of da_rows, dc_rows
    float* dc_part;
};
cudaError_t launch_gate_prologue(const GateParams& g, bool is_bf16, int dk, cudaStream_t s);
cudaError_t launch_gate_epilogue(const GateParams& g, bool is_bf16, int dk, cudaStream_t s);

// Key-side row of (token t, value head h): q, k, p, alpha, beta (and their gradients' scratch
// indexing stays per value head).
__host__ __device__ __forceinline__ long long krow(const ChunkParams& p, long long t, int h) {
    return t * (p.H / p.vg) + h / p.vg;
}

// Record stage-boundary event i on stream s when instrumentation is on.
inline void mark(const ChunkParams& p, int i, cudaStream_t s) {
    if (p.ev && i < p.nev) cudaEventRecord(p.ev[i], s);
}

// Arguments of the sequential scan S^T <- gamma S^T + S^T X^T + Y (see scan.cu).
struct ScanArgs {
    int H, N, T, slots;
    long long Ttot;
    const int32_t* cu;
    const int* seq_first;
    const float* Gb;         // chunk log-decays: gamma_n = exp(G[L-1])
    const float* init;       // [N,H,dk,dv] initial state (h0 or dhT) or null
    float* fin;              // [N,H,dk,dv] final state (hT or dh0) or null
    void* Sout;              // [pairs][dv][dk] state each chunk starts from (storage type)
    const void* X;           // [pairs][dk][dk] row-major
    const void* Y;           // [pairs][dv][dk]; at dk = 256 the forward's is U [pairs][64][dv] instead
    const void* W;           // dk = 256: the chunks' W [pairs][64][dk] and the keys [tokens, H / vg, dk]
    const void* K;           //           (the scan applies E = U - W H per chunk instead of Atilde)
    int reverse;
    int x_mn;                // X is read as an MN-major operand ([k][m] row-major, no transpose)
    int vg;                  // value heads per key head: init/fin are [N, H / vg, dk, vg * dv]
    int* err;
    uint32_t wait_ns;        // limit of each device-side wait
    // tcgen05 path (dk = dv = 128): the scan forms each chunk's additive term itself instead of
    // reading Y, as a product of a workspace factor F and a token tensor `tok`:
    //   ym = 2 (forward):  B^T = U_s^T K,  F = U_s^T [pairs][dv][64], tok = keys [tokens, H / vg, dk]
    //   ym = 1 (reverse):  C^T = dO^T Z,   F = Z^T [pairs][dk][64],   tok = dO [tokens, H, dv]
    // and at dk = 256 (k_scan_wide) ym = 1 with F = Z [pairs][64][dk] (key-head pairs).
    int ym = 0;
    const void* F = nullptr;
    const void* tok = nullptr;
};
cudaError_t launch_scan(const ScanArgs& a, bool is_bf16, int dk, int dv, long long pairs, cudaStream_t s);
size_t scan_smem_bytes(bool is_bf16, int dk, int dv);
// dk = 256 (bf16, value heads 64 wide): the scan of scan_wide.cu
cudaError_t launch_scan_wide(const ScanArgs& a, cudaStream_t s);
size_t scan_wide_smem_bytes();

// Kernel launchers (one translation unit each); return cudaGetLastError().
cudaError_t launch_chunk_map(const ChunkParams& p, cudaStream_t s);
// Forward kernels: prep (W, U, G, Atilde, B^T; M and Atilde^T when `save`), the scan,
// and the output kernel (O when p.o is set; E when `save`).  Stage events: ev0 before
// prep, ev0+1 before the scan, ev0+2 before the output, ev0+3 after it.
cudaError_t launch_fwd(const ChunkParams& p, bool is_bf16, bool save, cudaStream_t s, int ev0);
// Backward kernels given the saved factors: C^T, the reverse scan, local gradients and
// the head reduction.  Stage events: ev0 before C^T, ev0+1 before the scan, ev0+2 before
// the local gradients, ev0+3 before the reduction, ev0+4 after it.
cudaError_t launch_bwd(const ChunkParams& p, bool is_bf16, cudaStream_t s, int ev0);
// `groups`: several value heads per key head (the output kernel then double-buffers their tiles)
size_t fwd_smem_bytes(int kernel, bool is_bf16, int dk, int dv, bool pk = false, bool groups = false);
// tcgen05 kernels of the bf16 dk = dv = 128 path (chunk_tc.cu)
cudaError_t launch_prep_tc(const ChunkParams& p, cudaStream_t s);
cudaError_t launch_output_tc(const ChunkParams& p, cudaStream_t s);
size_t tc_smem_bytes(int kernel);
// tcgen05 prep and output kernels of the bf16 head-dim-256 path (value heads 64 wide; wide_tc.cu)
cudaError_t launch_prep_wide_tc(const ChunkParams& p, cudaStream_t s);
size_t prep_wide_tc_smem_bytes();
cudaError_t launch_output_wide_tc(const ChunkParams& p, cudaStream_t s);
size_t output_wide_tc_smem_bytes();
// tcgen05 local-gradient kernel of the same path (local_tc.cu)
cudaError_t launch_bwd_local_tc(const ChunkParams& p, cudaStream_t s);
size_t local_tc_smem_bytes();
// The tcgen05 kernels of chunk_tc.cu, local_tc.cu and scan.cu serve bf16 dk = dv = 128, with or
// without Comba-pk feedback vectors; bf16 dk = 256 runs the kernels of wide_tc.cu and
// scan_wide.cu with the mma.sync local-gradient kernel; every other case runs the mma.sync kernels.
inline bool use_tc_path(bool is_bf16, int dk, int dv) { return is_bf16 && dk == 128 && dv == 128; }
size_t bwd_smem_bytes(int kernel, bool is_bf16, int dk, int dv, bool pk = false);
// `p`: Comba-pk feedback vectors [Bd,H,dk] or null (p = k).
cudaError_t launch_recurrent_step(int Bd, int H, int dk, int dv, bool is_bf16, const void* q, const void* k,
                                  const void* v, const void* p, const float* alpha, const float* beta,
                                  const float* b, const float* d, float* state, void* o, bool iplr, cudaStream_t s);
// Value-head groups: sums over the vg value heads of each key head, in a fixed order, of the
// backward's per-value-head dq, dk [tokens, H, dk] (storage type), dalpha, dbeta [tokens, H] and,
// with Comba-pk feedback vectors, dp (dp_v and dp null otherwise).
cudaError_t launch_group_sum(const void* dq_v, const void* dk_v, const float* da_v, const float* db_v,
                             const void* dp_v, void* dq, void* dk, float* dalpha, float* dbeta, void* dp,
                             long long tokens, int H, int vg, int dk_, bool is_bf16, cudaStream_t s);
// Device address of the static scratch of comba_chunk_fwd_noalloc on the current device
// (noalloc.cu); its first 4 bytes are that entry point's status word.
cudaError_t static_scratch_address(void** out);
// Comba-pk correction applied before the chunk kernels: qt = q - d_h p over [rows = tokens*H, dk].
cudaError_t launch_pk_qtilde(const void* q, const void* p, const float* d, void* qt, long long rows, int H, int dk,
                             bool is_bf16, cudaStream_t s);

}  // namespace comba
