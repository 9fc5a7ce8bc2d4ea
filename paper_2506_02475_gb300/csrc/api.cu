// C ABI of the Comba library: argument validation, workspace carve-up and
// kernel sequencing.  Declarations and the contract live in include/comba.h.
#include <cuda_runtime.h>

#include "../../include/comba.h"
#include "params.cuh"

using comba::ChunkParams;

namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

struct Layout {
    size_t err, slot_info, seq_first, W, U, G, A, B, Us, Hs, E, M, AT, C, Z, dH, part;
    // gate and normalisation prologue (COMBA_GATED): its outputs, and the backward's gradients
    // w.r.t. them with the per-row contributions to da, dc
    size_t qh, kh, ga, gb, bg, dqh, dkh, dal, dbe, dbi, dar, dcr, dpa, dpc;
    // Comba-pk (COMBA_PK): the corrected queries q - d p and the zero d the chunk kernels then see
    size_t qt, dz;
    // value-head groups (vg > 1): the backward's per-value-head dq, dk, dalpha, dbeta (and dp)
    size_t gdq, gdk, gda, gdb, gdp;
    size_t total;
    int slots;
    int vg;      // value heads per key head; the kernels see H * vg heads of width dv / vg
};

// Value heads per key head: dv beyond 128 (a multiple of 128, dk = 128, bf16) runs as dv / 128
// value heads of width 128 that share the key head's q, k (p) and gates; at head dim dk = 256 the
// value heads are 64 wide (dv = 64 .. 256).
int value_groups(const comba_shape_t* s) {
    if (s->dk == 256) return s->dv >= 64 ? s->dv / 64 : 1;
    return s->dv > 128 ? s->dv / 128 : 1;
}

// Key widths with a chunk map Atilde (dk x dk) in the workspace; at dk = 256 the scan forms
// E = U - W H per chunk instead.
bool has_chunk_map(int dk) { return dk <= 128; }

// Validates the shape (not the pointers) and computes the workspace layout.
// The forward needs W, U, G, Atilde, B^T and the chunk states; saving for the
// backward (and the backward itself) adds E, M, Atilde^T, C^T, dH'^T and the
// per-chunk partial sums.
comba_status_t plan(const comba_shape_t* s, int backward, Layout* out) {
    if (!s) return COMBA_ERR_INVALID_ARG;
    if (s->B < 1 || s->T < 0 || s->H < 1 || s->num_seqs < 1) return COMBA_ERR_INVALID_ARG;
    if (s->dtype != COMBA_F32 && s->dtype != COMBA_BF16) return COMBA_ERR_INVALID_ARG;
    if (s->chunk != comba::kChunk) return COMBA_ERR_UNSUPPORTED;
    const int vg = value_groups(s);
    if (s->dk == 256) {
        // head dim 256 (bf16; plain, iplr, pk or gated form): value heads 64 wide, at most four per key head
        if (s->dtype != COMBA_BF16 || s->dv < 64 || s->dv % 64 != 0 || vg > 4) return COMBA_ERR_UNSUPPORTED;
    } else if (vg > 1) {
        // dv = 256, 384 or 512 as groups of 128-wide value heads on the tcgen05 path
        if (s->dv % 128 != 0 || vg > 4 || s->dk != 128 || s->dtype != COMBA_BF16) return COMBA_ERR_UNSUPPORTED;
    } else if ((s->dk != 64 && s->dk != 128) || (s->dv != 64 && s->dv != 128)) {
        return COMBA_ERR_UNSUPPORTED;
    }
    if ((long long)s->H * vg > 65535 || s->num_seqs > 2147483647 / 4) return COMBA_ERR_UNSUPPORTED;
    if (s->cu_seqlens) {
        if (s->B != 1) return COMBA_ERR_INVALID_ARG;
        if (!aligned16(s->cu_seqlens)) return COMBA_ERR_INVALID_ARG;
    } else if (s->num_seqs != s->B) {
        return COMBA_ERR_INVALID_ARG;
    }
    const long long ttot = (long long)s->B * s->T;
    if (ttot >= (1LL << 31)) return COMBA_ERR_UNSUPPORTED;
    if (backward && s->dtype == COMBA_F32 && (s->dk != 64 || s->dv != 64)) return COMBA_ERR_UNSUPPORTED;
    const long long slots = s->cu_seqlens ? ttot / comba::kChunk + s->num_seqs
                                          : (long long)s->B * ((s->T + comba::kChunk - 1) / comba::kChunk);
    const long long pairs_ll = slots * s->H * vg;   // (chunk slot, value head) units
    // the scan addresses chunk-state rows with 32-bit TMA coordinates
    if (slots >= (1LL << 30) || pairs_ll * 128 >= (1LL << 31)) return COMBA_ERR_UNSUPPORTED;
    const size_t es = s->dtype == COMBA_BF16 ? 2 : 4;
    const size_t pairs = (size_t)pairs_ll;
    const size_t dk = s->dk, dv = s->dv / vg;       // one value head's width
    Layout L{};
    L.vg = vg;
    size_t o = 0;
    auto take = [&](size_t bytes) { size_t at = o; o = align_up(o + bytes); return at; };
    L.err = take(sizeof(int));
    L.slot_info = take(sizeof(comba::SlotInfo) * (size_t)slots);
    L.seq_first = take(sizeof(int) * (size_t)(s->num_seqs + 1));
    L.W = take(pairs * 64 * dk * es);
    L.U = take(pairs * 64 * dv * es);
    L.G = take(pairs * 64 * sizeof(float));
    const bool tcp = comba::use_tc_path(s->dtype == COMBA_BF16, s->dk, s->dv / vg);
    if (has_chunk_map(s->dk)) {
        L.A = take(pairs * dk * dk * es);
        // the tcgen05 path keeps U_s^T (its forward scan forms B^T itself); the others B^T
        if (tcp)
            L.Us = take(pairs * dv * 64 * es);
        else
            L.B = take(pairs * dv * dk * es);
    }
    L.Hs = take(pairs * dv * dk * es);
    if (backward) {
        L.E = take(pairs * 64 * dv * es);
        L.M = take(pairs * 64 * 64 * es);
        // Atilde^T is only materialised off the tcgen05 path (that reverse scan reads Atilde directly)
        if (has_chunk_map(s->dk) && !comba::use_tc_path(s->dtype == COMBA_BF16, s->dk, s->dv))
            L.AT = take(pairs * dk * dk * es);
        // the tcgen05 path keeps Z^T, head dim 256 Z (their reverse scans form C themselves); the
        // others C^T
        if (tcp || s->dk == 256)
            L.Z = take(pairs * dk * 64 * es);
        else
            L.C = take(pairs * dv * dk * es);
        L.dH = take(pairs * dv * dk * es);
        L.part = take(pairs * 2 * sizeof(float));
    }
    if (s->flags & COMBA_GATED) {
        const size_t rows = (size_t)ttot * s->H;
        L.qh = take(rows * dk * es);
        L.kh = take(rows * dk * es);
        L.ga = take(rows * sizeof(float));
        L.gb = take(rows * sizeof(float));
        L.bg = take((size_t)s->H * sizeof(float));
        if (backward) {
            L.dqh = take(rows * dk * es);
            L.dkh = take(rows * dk * es);
            L.dal = take(rows * sizeof(float));
            L.dbe = take(rows * sizeof(float));
            L.dbi = take((size_t)s->H * sizeof(float));
            L.dar = take(rows * sizeof(float));
            L.dcr = take(rows * sizeof(float));
            const size_t parts = (size_t)((ttot + 63) / 64) * s->H;   // token blocks of the per-head sums
            L.dpa = take(parts * sizeof(float));
            L.dpc = take(parts * sizeof(float));
        }
    }
    if (s->flags & COMBA_PK) {
        L.qt = take((size_t)ttot * s->H * dk * es);
        L.dz = take((size_t)s->H * sizeof(float));
    }
    if (backward && vg > 1) {
        const size_t vrows = (size_t)ttot * s->H * vg;
        L.gdq = take(vrows * dk * es);
        L.gdk = take(vrows * dk * es);
        L.gda = take(vrows * sizeof(float));
        L.gdb = take(vrows * sizeof(float));
        if (s->flags & COMBA_PK) L.gdp = take(vrows * dk * es);
    }
    L.total = o;
    L.slots = (int)slots;
    *out = L;
    return COMBA_OK;
}

comba_status_t check_smem(const comba_shape_t* s, int backward) {
    int dev = 0, optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return COMBA_ERR_CUDA;
    if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return COMBA_ERR_CUDA;
    const bool bf = s->dtype == COMBA_BF16, pk = (s->flags & COMBA_PK) != 0;
    const int dv = s->dv / value_groups(s);
    for (int kern = 0; kern < 3; ++kern)
        if (comba::fwd_smem_bytes(kern, bf, s->dk, dv, pk, value_groups(s) > 1) > (size_t)optin)
            return COMBA_ERR_UNSUPPORTED;
    if (backward)
        for (int kern = 0; kern < 2; ++kern)
            if (comba::bwd_smem_bytes(kern, bf, s->dk, dv, pk) > (size_t)optin) return COMBA_ERR_UNSUPPORTED;
    return COMBA_OK;
}

void fill_common(ChunkParams& p, const comba_shape_t* s, const Layout& L, void* ws, bool backward_layout) {
    char* w = static_cast<char*>(ws);
    p.B = s->B; p.T = s->T; p.N = s->num_seqs;
    p.vg = L.vg;
    p.H = s->H * L.vg;                 // value heads
    p.dk = s->dk; p.dv = s->dv / L.vg;
    p.Ttot = (long long)s->B * s->T;
    p.cu = s->cu_seqlens;
    p.slots = L.slots;
    p.iplr = (s->flags & COMBA_IPLR) != 0;
    p.stall = (s->flags & COMBA_DIAG_STALL) != 0;
    p.ev = reinterpret_cast<cudaEvent_t*>(s->stage_events);
    p.nev = s->stage_events ? s->num_stage_events : 0;
    p.err = reinterpret_cast<int*>(w + L.err);
    const uint32_t lim = s->wait_limit_ns ? s->wait_limit_ns : comba::kDefaultWaitNs;
    p.wait_ns = lim < comba::kMaxWaitNs ? lim : comba::kMaxWaitNs;
    p.slot_info = reinterpret_cast<comba::SlotInfo*>(w + L.slot_info);
    p.seq_first = reinterpret_cast<int*>(w + L.seq_first);
    p.Wb = w + L.W;
    p.Ub = w + L.U;
    p.Gb = reinterpret_cast<float*>(w + L.G);
    // (offset 0 is the status word, so a zero offset marks a region that is not allocated)
    p.Ab = L.A ? w + L.A : nullptr;
    p.Bb = L.B ? w + L.B : nullptr;
    p.Usb = L.Us ? w + L.Us : nullptr;
    p.Hb = w + L.Hs;
    if (backward_layout) {
        p.Eb = w + L.E;
        p.Mb = w + L.M;
        p.ATb = L.AT ? w + L.AT : nullptr;
        p.Cb = L.C ? w + L.C : nullptr;
        p.Zb = L.Z ? w + L.Z : nullptr;
        p.dHb = w + L.dH;
        p.part = reinterpret_cast<float*>(w + L.part);
    }
}

#define COMBA_REQUIRE(ptr)                                   \
    do {                                                     \
        if (!(ptr) || !aligned16(ptr)) return COMBA_ERR_INVALID_ARG; \
    } while (0)
#define COMBA_OPTIONAL(ptr)                                  \
    do {                                                     \
        if ((ptr) && !aligned16(ptr)) return COMBA_ERR_INVALID_ARG; \
    } while (0)

}  // namespace

extern "C" {

const char* comba_status_string(comba_status_t status) {
    switch (status) {
        case COMBA_OK: return "ok";
        case COMBA_ERR_INVALID_ARG: return "invalid argument";
        case COMBA_ERR_UNSUPPORTED: return "unsupported configuration";
        case COMBA_ERR_WORKSPACE: return "workspace missing or too small";
        case COMBA_ERR_CUDA: return "CUDA error";
        case COMBA_ERR_TIMEOUT: return "device-side wait timed out";
    }
    return "unknown status";
}

size_t comba_workspace_size(const comba_shape_t* shape, int backward) {
    Layout L;
    if (plan(shape, backward, &L) != COMBA_OK) return 0;
    return L.total;
}

comba_status_t comba_workspace_status(const void* workspace, comba_stream_t stream) {
    const cudaStream_t s = stream;
    const void* word = workspace;   // the status word is the workspace's first 4 bytes (Layout::err = 0)
    if (!word) {
        void* scratch = nullptr;
        if (comba::static_scratch_address(&scratch) != cudaSuccess) return COMBA_ERR_CUDA;
        word = scratch;
    }
    int host = 0;
    if (cudaStreamSynchronize(s) != cudaSuccess) return COMBA_ERR_CUDA;
    if (cudaMemcpyAsync(&host, word, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return COMBA_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return COMBA_ERR_CUDA;
    return host ? COMBA_ERR_TIMEOUT : COMBA_OK;
}

}  // extern "C"

namespace {

// Comba-pk arguments of the chunk kernels: feedback vectors, the d of the correction applied
// to q beforehand, and dL/dp (backward).
struct PkArgs {
    const void* p = nullptr;
    const float* d = nullptr;
    void* dp = nullptr;
};

// Launch the forward on validated arguments (L from plan(); shape checks done).
comba_status_t forward_run(const comba_shape_t* shape, const Layout& L, void* workspace, const void* q, const void* k,
                           const void* v, const float* alpha, const float* beta, const float* b, const float* d,
                           const float* h0, void* o, float* hT, bool save, cudaStream_t s, PkArgs pk = {}) {
    comba_status_t st;
    if ((st = check_smem(shape, 0)) != COMBA_OK) return st;
    ChunkParams p{};
    fill_common(p, shape, L, workspace, save);
    p.q = q; p.k = k; p.v = v; p.alpha = alpha; p.beta = beta; p.b = b; p.d = d; p.h0 = h0;
    p.p = pk.p; p.d_fb = pk.d;
    p.o = o; p.hT = hT;
    comba::mark(p, 0, s);
    if (comba::launch_chunk_map(p, s) != cudaSuccess) return COMBA_ERR_CUDA;
    if (comba::launch_fwd(p, shape->dtype == COMBA_BF16, save, s, 1) != cudaSuccess) return COMBA_ERR_CUDA;
    return COMBA_OK;
}

comba_status_t backward_run(const comba_shape_t* shape, const Layout& L, void* workspace, const void* q,
                            const void* k, const void* v, const float* alpha, const float* beta, const float* b,
                            const float* d, const float* h0, const void* dO, const float* dhT, void* dq, void* dk,
                            void* dv, float* dalpha, float* dbeta, float* db, float* dd, float* dh0, bool reuse,
                            cudaStream_t s, PkArgs pk = {}) {
    comba_status_t st;
    if ((st = check_smem(shape, 1)) != COMBA_OK) return st;
    ChunkParams p{};
    fill_common(p, shape, L, workspace, true);
    p.q = q; p.k = k; p.v = v; p.alpha = alpha; p.beta = beta; p.b = b; p.d = d; p.h0 = h0;
    p.p = pk.p; p.d_fb = pk.d; p.dpp = pk.dp;
    p.dO = dO; p.dhT = dhT; p.dq = dq; p.dkk = dk; p.dvv = dv;
    p.dalpha = dalpha; p.dbeta = dbeta; p.db = db; p.dd = dd; p.dh0 = dh0;
    if (L.vg > 1) {
        // per-value-head key-side gradients into the workspace, summed per key head below
        char* w = static_cast<char*>(workspace);
        p.dq = w + L.gdq; p.dkk = w + L.gdk;
        p.dalpha = reinterpret_cast<float*>(w + L.gda);
        p.dbeta = reinterpret_cast<float*>(w + L.gdb);
        if (pk.dp) p.dpp = w + L.gdp;
    }
    const bool bf = shape->dtype == COMBA_BF16;
    comba::mark(p, 0, s);
    if (reuse) {
        for (int e = 1; e <= 4; ++e) comba::mark(p, e, s);
    } else {
        // recompute the forward factors and chunk states (no output, no final state)
        ChunkParams f = p;
        f.o = nullptr;
        f.hT = nullptr;
        if (comba::launch_chunk_map(f, s) != cudaSuccess) return COMBA_ERR_CUDA;
        if (comba::launch_fwd(f, bf, true, s, 1) != cudaSuccess) return COMBA_ERR_CUDA;
    }
    if (comba::launch_bwd(p, bf, s, 4) != cudaSuccess) return COMBA_ERR_CUDA;
    if (L.vg > 1 && comba::launch_group_sum(p.dq, p.dkk, p.dalpha, p.dbeta, pk.dp ? p.dpp : nullptr, dq, dk, dalpha,
                                            dbeta, pk.dp, p.Ttot, p.H, L.vg, p.dk, bf, s) != cudaSuccess)
        return COMBA_ERR_CUDA;
    return COMBA_OK;
}

// Decode head widths: dk in {64, 128, 256}; dv in {64, 128}, or 256 with dk >= 128.
bool step_dims_ok(int dk, int dv) {
    if (dk != 64 && dk != 128 && dk != 256) return false;
    return dv == 64 || dv == 128 || (dv == 256 && dk >= 128);
}

comba::GateParams gate_params(const comba_shape_t* shape, const Layout& L, void* workspace, const void* q,
                              const void* k, const float* g_alpha, const float* g_beta, const float* a,
                              const float* c, const float* b_raw) {
    char* w = static_cast<char*>(workspace);
    comba::GateParams g{};
    g.rows = (long long)shape->B * shape->T * shape->H;
    g.H = shape->H;
    g.eps = 1e-6f;
    g.q = q; g.k = k; g.g_alpha = g_alpha; g.g_beta = g_beta; g.a = a; g.c = c; g.b_raw = b_raw;
    g.qh = w + L.qh; g.kh = w + L.kh;
    g.alpha = reinterpret_cast<float*>(w + L.ga);
    g.beta = reinterpret_cast<float*>(w + L.gb);
    g.bgate = reinterpret_cast<float*>(w + L.bg);
    return g;
}

}  // namespace

extern "C" {

comba_status_t comba_chunk_fwd(const comba_shape_t* shape, const void* q, const void* k, const void* v,
                               const float* alpha, const float* beta, const float* b, const float* d,
                               const float* h0, void* o, float* hT, void* workspace, size_t workspace_bytes,
                               comba_stream_t stream) {
    Layout L;
    const bool save = shape && (shape->flags & COMBA_SAVE_FACTORS);
    comba_status_t st = plan(shape, save ? 1 : 0, &L);
    if (st != COMBA_OK) return st;
    if (shape->flags & ~(COMBA_SAVE_FACTORS | COMBA_IPLR | COMBA_DIAG_STALL)) return COMBA_ERR_INVALID_ARG;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(alpha); COMBA_REQUIRE(beta);
    COMBA_REQUIRE(d); COMBA_REQUIRE(o);
    COMBA_OPTIONAL(b); COMBA_OPTIONAL(h0); COMBA_OPTIONAL(hT);
    if (shape->stage_events && shape->num_stage_events < COMBA_FWD_EVENTS) return COMBA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < L.total) return COMBA_ERR_WORKSPACE;
    return forward_run(shape, L, workspace, q, k, v, alpha, beta, b, d, h0, o, hT, save,
                       stream);
}

comba_status_t comba_chunk_bwd(const comba_shape_t* shape, const void* q, const void* k, const void* v,
                               const float* alpha, const float* beta, const float* b, const float* d,
                               const float* h0, const void* dO, const float* dhT, void* dq, void* dk, void* dv,
                               float* dalpha, float* dbeta, float* db, float* dd, float* dh0, void* workspace,
                               size_t workspace_bytes, comba_stream_t stream) {
    Layout L;
    comba_status_t st = plan(shape, 1, &L);
    if (st != COMBA_OK) return st;
    if (shape->flags & ~(COMBA_REUSE_FACTORS | COMBA_IPLR | COMBA_DIAG_STALL)) return COMBA_ERR_INVALID_ARG;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(alpha); COMBA_REQUIRE(beta);
    COMBA_REQUIRE(d); COMBA_REQUIRE(dO);
    COMBA_REQUIRE(dq); COMBA_REQUIRE(dk); COMBA_REQUIRE(dv); COMBA_REQUIRE(dalpha); COMBA_REQUIRE(dbeta);
    COMBA_REQUIRE(dd);
    COMBA_OPTIONAL(b); COMBA_OPTIONAL(h0); COMBA_OPTIONAL(dhT); COMBA_OPTIONAL(db); COMBA_OPTIONAL(dh0);
    if (shape->stage_events && shape->num_stage_events < COMBA_BWD_EVENTS) return COMBA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < L.total) return COMBA_ERR_WORKSPACE;
    return backward_run(shape, L, workspace, q, k, v, alpha, beta, b, d, h0, dO, dhT, dq, dk, dv, dalpha, dbeta, db,
                        dd, dh0, (shape->flags & COMBA_REUSE_FACTORS) != 0, stream);
}

comba_status_t comba_chunk_fwd_gated(const comba_shape_t* shape, const void* q, const void* k, const void* v,
                                     const float* g_alpha, const float* g_beta, const float* a, const float* c,
                                     const float* b_raw, const float* d, const float* h0, void* o, float* hT,
                                     void* workspace, size_t workspace_bytes, comba_stream_t stream) {
    Layout L;
    const bool save = shape && (shape->flags & COMBA_SAVE_FACTORS);
    comba_status_t st = plan(shape, save ? 1 : 0, &L);
    if (st != COMBA_OK) return st;
    if (!(shape->flags & COMBA_GATED) || (shape->flags & ~(COMBA_GATED | COMBA_SAVE_FACTORS | COMBA_IPLR)))
        return COMBA_ERR_INVALID_ARG;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(g_alpha); COMBA_REQUIRE(g_beta);
    COMBA_REQUIRE(a); COMBA_REQUIRE(c); COMBA_REQUIRE(b_raw); COMBA_REQUIRE(d); COMBA_REQUIRE(o);
    COMBA_OPTIONAL(h0); COMBA_OPTIONAL(hT);
    if (shape->stage_events && shape->num_stage_events < COMBA_FWD_EVENTS) return COMBA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < L.total) return COMBA_ERR_WORKSPACE;
    const cudaStream_t s = stream;
    const comba::GateParams g = gate_params(shape, L, workspace, q, k, g_alpha, g_beta, a, c, b_raw);
    if (comba::launch_gate_prologue(g, shape->dtype == COMBA_BF16, shape->dk, s) != cudaSuccess) return COMBA_ERR_CUDA;
    return forward_run(shape, L, workspace, g.qh, g.kh, v, g.alpha, g.beta, g.bgate, d, h0, o, hT, save, s);
}

comba_status_t comba_chunk_bwd_gated(const comba_shape_t* shape, const void* q, const void* k, const void* v,
                                     const float* g_alpha, const float* g_beta, const float* a, const float* c,
                                     const float* b_raw, const float* d, const float* h0, const void* dO,
                                     const float* dhT, void* dq, void* dk, void* dv, float* dg_alpha, float* dg_beta,
                                     float* da, float* dc, float* db_raw, float* dd, float* dh0, void* workspace,
                                     size_t workspace_bytes, comba_stream_t stream) {
    Layout L;
    comba_status_t st = plan(shape, 1, &L);
    if (st != COMBA_OK) return st;
    if (!(shape->flags & COMBA_GATED) || (shape->flags & ~(COMBA_GATED | COMBA_REUSE_FACTORS | COMBA_IPLR)))
        return COMBA_ERR_INVALID_ARG;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(g_alpha); COMBA_REQUIRE(g_beta);
    COMBA_REQUIRE(a); COMBA_REQUIRE(c); COMBA_REQUIRE(b_raw); COMBA_REQUIRE(d); COMBA_REQUIRE(dO);
    COMBA_REQUIRE(dq); COMBA_REQUIRE(dk); COMBA_REQUIRE(dv); COMBA_REQUIRE(dg_alpha); COMBA_REQUIRE(dg_beta);
    COMBA_REQUIRE(da); COMBA_REQUIRE(dc); COMBA_REQUIRE(dd);
    COMBA_OPTIONAL(h0); COMBA_OPTIONAL(dhT); COMBA_OPTIONAL(db_raw); COMBA_OPTIONAL(dh0);
    if (shape->stage_events && shape->num_stage_events < COMBA_BWD_EVENTS) return COMBA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < L.total) return COMBA_ERR_WORKSPACE;
    const cudaStream_t s = stream;
    const bool reuse = (shape->flags & COMBA_REUSE_FACTORS) != 0;
    const bool bf = shape->dtype == COMBA_BF16;
    comba::GateParams g = gate_params(shape, L, workspace, q, k, g_alpha, g_beta, a, c, b_raw);
    // with reused factors the saving forward left the prologue's outputs in the workspace
    if (!reuse && comba::launch_gate_prologue(g, bf, shape->dk, s) != cudaSuccess) return COMBA_ERR_CUDA;
    char* w = static_cast<char*>(workspace);
    g.dqh = w + L.dqh; g.dkh = w + L.dkh;
    g.dalpha = reinterpret_cast<float*>(w + L.dal);
    g.dbeta = reinterpret_cast<float*>(w + L.dbe);
    g.db = reinterpret_cast<float*>(w + L.dbi);
    g.dq = dq; g.dk = dk; g.dg_alpha = dg_alpha; g.dg_beta = dg_beta; g.da = da; g.dc = dc; g.db_raw = db_raw;
    g.da_rows = reinterpret_cast<float*>(w + L.dar);
    g.dc_rows = reinterpret_cast<float*>(w + L.dcr);
    g.da_part = reinterpret_cast<float*>(w + L.dpa);
    g.dc_part = reinterpret_cast<float*>(w + L.dpc);
    st = backward_run(shape, L, workspace, g.qh, g.kh, v, g.alpha, g.beta, g.bgate, d, h0, dO, dhT,
                      const_cast<void*>(g.dqh), const_cast<void*>(g.dkh), dv, const_cast<float*>(g.dalpha),
                      const_cast<float*>(g.dbeta), const_cast<float*>(g.db), dd, dh0, reuse, s);
    if (st != COMBA_OK) return st;
    if (comba::launch_gate_epilogue(g, bf, shape->dk, s) != cudaSuccess) return COMBA_ERR_CUDA;
    return COMBA_OK;
}

// Comba-pk: q - d p into the workspace and a zeroed d for the chunk kernels.
// `reuse`: a backward reusing the saved factors of a forward on the same inputs and workspace,
// which already holds q - d p and the zero d.
static comba_status_t pk_prologue(const comba_shape_t* shape, const Layout& L, void* workspace, const void* q,
                                  const void* p, const float* d, cudaStream_t s, void** qt, float** dz,
                                  bool reuse = false) {
    char* w = static_cast<char*>(workspace);
    *qt = w + L.qt;
    *dz = reinterpret_cast<float*>(w + L.dz);
    if (reuse) return COMBA_OK;
    if (cudaMemsetAsync(*dz, 0, (size_t)shape->H * sizeof(float), s) != cudaSuccess) return COMBA_ERR_CUDA;
    if (comba::launch_pk_qtilde(q, p, d, *qt, (long long)shape->B * shape->T * shape->H, shape->H, shape->dk,
                                shape->dtype == COMBA_BF16, s) != cudaSuccess)
        return COMBA_ERR_CUDA;
    return COMBA_OK;
}

comba_status_t comba_chunk_fwd_pk(const comba_shape_t* shape, const void* q, const void* k, const void* v,
                                  const void* p, const float* alpha, const float* beta, const float* b,
                                  const float* d, const float* h0, void* o, float* hT, void* workspace,
                                  size_t workspace_bytes, comba_stream_t stream) {
    Layout L;
    const bool save = shape && (shape->flags & COMBA_SAVE_FACTORS);
    comba_status_t st = plan(shape, save ? 1 : 0, &L);
    if (st != COMBA_OK) return st;
    if (!(shape->flags & COMBA_PK) || (shape->flags & ~(COMBA_PK | COMBA_SAVE_FACTORS | COMBA_IPLR)))
        return COMBA_ERR_INVALID_ARG;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(p); COMBA_REQUIRE(alpha);
    COMBA_REQUIRE(beta); COMBA_REQUIRE(d); COMBA_REQUIRE(o);
    COMBA_OPTIONAL(b); COMBA_OPTIONAL(h0); COMBA_OPTIONAL(hT);
    if (shape->stage_events && shape->num_stage_events < COMBA_FWD_EVENTS) return COMBA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < L.total) return COMBA_ERR_WORKSPACE;
    const cudaStream_t s = stream;
    void* qt;
    float* dz;
    if ((st = pk_prologue(shape, L, workspace, q, p, d, s, &qt, &dz)) != COMBA_OK) return st;
    PkArgs pk;
    pk.p = p; pk.d = d;
    return forward_run(shape, L, workspace, qt, k, v, alpha, beta, b, dz, h0, o, hT, save, s, pk);
}

comba_status_t comba_chunk_bwd_pk(const comba_shape_t* shape, const void* q, const void* k, const void* v,
                                  const void* p, const float* alpha, const float* beta, const float* b,
                                  const float* d, const float* h0, const void* dO, const float* dhT, void* dq,
                                  void* dk, void* dv, void* dp, float* dalpha, float* dbeta, float* db, float* dd,
                                  float* dh0, void* workspace, size_t workspace_bytes, comba_stream_t stream) {
    Layout L;
    comba_status_t st = plan(shape, 1, &L);
    if (st != COMBA_OK) return st;
    if (!(shape->flags & COMBA_PK) || (shape->flags & ~(COMBA_PK | COMBA_REUSE_FACTORS | COMBA_IPLR)))
        return COMBA_ERR_INVALID_ARG;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(p); COMBA_REQUIRE(alpha);
    COMBA_REQUIRE(beta); COMBA_REQUIRE(d); COMBA_REQUIRE(dO);
    COMBA_REQUIRE(dq); COMBA_REQUIRE(dk); COMBA_REQUIRE(dv); COMBA_REQUIRE(dp); COMBA_REQUIRE(dalpha);
    COMBA_REQUIRE(dbeta); COMBA_REQUIRE(dd);
    COMBA_OPTIONAL(b); COMBA_OPTIONAL(h0); COMBA_OPTIONAL(dhT); COMBA_OPTIONAL(db); COMBA_OPTIONAL(dh0);
    if (shape->stage_events && shape->num_stage_events < COMBA_BWD_EVENTS) return COMBA_ERR_INVALID_ARG;
    if (!workspace || !aligned16(workspace) || workspace_bytes < L.total) return COMBA_ERR_WORKSPACE;
    const cudaStream_t s = stream;
    void* qt;
    float* dz;
    if ((st = pk_prologue(shape, L, workspace, q, p, d, s, &qt, &dz, (shape->flags & COMBA_REUSE_FACTORS) != 0)) !=
        COMBA_OK)
        return st;
    PkArgs pk;
    pk.p = p; pk.d = d; pk.dp = dp;
    return backward_run(shape, L, workspace, qt, k, v, alpha, beta, b, dz, h0, dO, dhT, dq, dk, dv, dalpha, dbeta, db,
                        dd, dh0, (shape->flags & COMBA_REUSE_FACTORS) != 0, s, pk);
}

comba_status_t comba_recurrent_step_pk(int Bd, int H, int dk, int dv, comba_dtype_t dtype, const void* q,
                                       const void* k, const void* v, const void* p, const float* alpha,
                                       const float* beta, const float* b, const float* d, float* state, void* o,
                                       int flags, comba_stream_t stream) {
    if (Bd < 1 || H < 1) return COMBA_ERR_INVALID_ARG;
    if (flags & ~COMBA_IPLR) return COMBA_ERR_INVALID_ARG;
    if (dtype != COMBA_F32 && dtype != COMBA_BF16) return COMBA_ERR_INVALID_ARG;
    if (!step_dims_ok(dk, dv)) return COMBA_ERR_UNSUPPORTED;
    if ((long long)Bd * H * (dv / 32) >= (1LL << 31)) return COMBA_ERR_UNSUPPORTED;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(p); COMBA_REQUIRE(alpha);
    COMBA_REQUIRE(beta); COMBA_REQUIRE(d); COMBA_REQUIRE(state); COMBA_REQUIRE(o);
    COMBA_OPTIONAL(b);
    if (comba::launch_recurrent_step(Bd, H, dk, dv, dtype == COMBA_BF16, q, k, v, p, alpha, beta, b, d, state, o,
                                     (flags & COMBA_IPLR) != 0, stream) != cudaSuccess)
        return COMBA_ERR_CUDA;
    return COMBA_OK;
}

comba_status_t comba_recurrent_step(int Bd, int H, int dk, int dv, comba_dtype_t dtype, const void* q,
                                    const void* k, const void* v, const float* alpha, const float* beta,
                                    const float* b, const float* d, float* state, void* o, int flags,
                                    comba_stream_t stream) {
    if (Bd < 1 || H < 1) return COMBA_ERR_INVALID_ARG;
    if (flags & ~COMBA_IPLR) return COMBA_ERR_INVALID_ARG;
    if (dtype != COMBA_F32 && dtype != COMBA_BF16) return COMBA_ERR_INVALID_ARG;
    if (!step_dims_ok(dk, dv)) return COMBA_ERR_UNSUPPORTED;
    if ((long long)Bd * H * (dv / 32) >= (1LL << 31)) return COMBA_ERR_UNSUPPORTED;
    COMBA_REQUIRE(q); COMBA_REQUIRE(k); COMBA_REQUIRE(v); COMBA_REQUIRE(alpha); COMBA_REQUIRE(beta);
    COMBA_REQUIRE(d); COMBA_REQUIRE(state); COMBA_REQUIRE(o);
    COMBA_OPTIONAL(b);
    if (comba::launch_recurrent_step(Bd, H, dk, dv, dtype == COMBA_BF16, q, k, v, nullptr, alpha, beta, b, d, state,
                                     o, (flags & COMBA_IPLR) != 0, stream) != cudaSuccess)
        return COMBA_ERR_CUDA;
    return COMBA_OK;
}

}  // extern "C"
