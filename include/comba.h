/*
 * comba.h -- C ABI of the GB300 (sm_103a) Comba chunk-parallel library.
 *
 * Comba ("Improving Bilinear RNNs with Closed-loop Control", arXiv 2506.02475)
 * is a bilinear RNN whose state S_t (dv x dk) follows, per sequence and head,
 *
 *     S_t = S_{t-1} (alpha_t I - btilde_t k_t k_t^T) + beta_t v_t k_t^T      (section 3, Eq. comba-S)
 *     o_t = S_t (q_t - d k_t)                                                (output correction, same Eq.)
 *     btilde_t = b * beta_t                                                  (section 3.1)
 *
 * This library stores the state transposed, H = S^T (dk x dv, row-major), as
 * the paper's recurrent listing does (appendix B.1).  Equivalently
 *     e_t = beta_t v_t - btilde_t H_{t-1}^T k_t,  H_t = alpha_t H_{t-1} + k_t e_t^T,
 *     o_t = H_t^T (q_t - d k_t).
 * There is no query scale.  Training uses the chunk-wise form of section 3.2
 * (WY representation with a single UT inverse per chunk, Eq. "prepare WY_M",
 * then the inter-chunk state and output equations); inference uses the
 * one-token recurrence.
 *
 * Conventions shared by every entry point
 *   - Every tensor argument is a DEVICE pointer owned by the caller.  The
 *     library allocates and frees nothing; scratch comes from the caller's
 *     workspace (size from comba_workspace_size).
 *   - Token tensors are row-major [B, T, H, D] (D contiguous).  For packed
 *     variable-length input pass B = 1, T = total tokens, num_seqs = N and
 *     cu_seqlens = device int32 [N+1] offsets (cu[0] = 0, non-decreasing,
 *     cu[N] = T); the state restarts at every sequence start and chunks never
 *     straddle a boundary.  With cu_seqlens == NULL, num_seqs must equal B.
 *   - q, k, v, o, dO, dq, dk, dv use the storage type `dtype` (fp32 or bf16).
 *     Gates alpha, beta and their gradients are fp32 [B, T, H]; the per-head
 *     scalars b, d and their gradients are fp32 [H].  States h0, hT, dhT, dh0
 *     are fp32 [num_seqs, H, dk, dv].  All arithmetic accumulates in fp32.
 *   - alpha must lie in (0, 1]: the chunk form takes logarithms of alpha.
 *   - All pointers must be 16-byte aligned.
 *   - Calls are asynchronous on `stream` (a cudaStream_t, as comba_stream_t; NULL =
 *     legacy default stream).  Outputs are overwritten, never accumulated into.
 *   - Validation is host-side only; invalid arguments return an error before
 *     anything is launched.  A failed launch returns COMBA_ERR_CUDA.
 *   - No global mutable state: calls on different streams may overlap as long
 *     as their workspaces and outputs are distinct.
 *   - Results are bitwise reproducible from run to run (fixed reduction order,
 *     no floating-point atomics).
 *
 * Head widths (chunk entry points; comba_workspace_size returns 0 for the rest)
 *   - dk, dv in {64, 128}, either storage type (the fp32 backward: dk = dv = 64).
 *   - dk = 128 with dv = 256, 384 or 512 (bf16, any of the four forms): each head
 *     runs as dv / 128 value heads of width 128 that share its q, k and gates
 *     (a state's columns evolve independently), and the key-side gradients are
 *     summed over them in a fixed order.
 *   - dk = 256 (the paper's head dim 256; bf16; plain, iplr, pk or gated form)
 *     with dv = 64, 128, 192 or 256: value heads 64 wide, the same way (with
 *     pk, dp is summed over a key head's value heads like dq and dk).
 */
#ifndef COMBA_H
#define COMBA_H

#include <stddef.h>
#include <stdint.h>

/* The CUDA runtime's stream handle: the same type as cudaStream_t, declared here so that this
 * header needs no CUDA include.  A cudaStream_t passes as it is; NULL is the legacy default
 * stream. */
struct CUstream_st;
typedef struct CUstream_st *comba_stream_t;

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    COMBA_OK = 0,
    COMBA_ERR_INVALID_ARG = 1,  /* NULL required pointer, bad shape, misalignment   */
    COMBA_ERR_UNSUPPORTED = 2,  /* valid but not implemented (head dim, chunk size) */
    COMBA_ERR_WORKSPACE = 3,    /* workspace NULL or smaller than required         */
    COMBA_ERR_CUDA = 4,         /* a CUDA launch or query failed                    */
    COMBA_ERR_TIMEOUT = 5       /* a device-side wait gave up (comba_workspace_status) */
} comba_status_t;

typedef enum { COMBA_F32 = 0, COMBA_BF16 = 1 } comba_dtype_t;

typedef struct {
    int B;                      /* batch; 1 when cu_seqlens != NULL               */
    int T;                      /* tokens per sequence, or total packed tokens    */
    int H;                      /* heads                                          */
    int dk;                     /* key/query head dim: 64, 128 or 256             */
    int dv;                     /* value head dim: 64 or 128; with dk = 128 also  */
                                /* 256, 384, 512; with dk = 256 64, 128, 192, 256 */
                                /* (wider dv and dk = 256: bf16; see "Head        */
                                /* widths" below)                                 */
    int num_seqs;               /* N: == B when cu_seqlens == NULL                */
    const int32_t *cu_seqlens;  /* device int32 [N+1] or NULL                     */
    comba_dtype_t dtype;        /* storage type of q, k, v, o and their grads     */
    int chunk;                  /* chunk length; must be 64                       */
    int flags;                  /* COMBA_SAVE_FACTORS / COMBA_REUSE_FACTORS, | COMBA_IPLR, COMBA_GATED, COMBA_PK */
    /* Optional instrumentation (NULL / 0 = off).  Caller-created cudaEvent_t
     * handles recorded on `stream` at kernel boundaries: comba_chunk_fwd
     * records COMBA_FWD_EVENTS of them (before chunk map, prep, state scan,
     * output, and after output); comba_chunk_bwd records COMBA_BWD_EVENTS
     * (before chunk map, prep, forward state scan, forward E, reverse-scan
     * term C, reverse state scan, local gradients, head reduction, and after
     * it).  Fewer handles than needed is COMBA_ERR_INVALID_ARG. */
    void **stage_events;
    int num_stage_events;
    /* Limit of each device-side wait of the call's kernels (tensor-core
     * completion, TMA arrival), in nanoseconds of the GPU's global timer;
     * 0 = the default of one second; values above 4e9 count as 4e9.  A wait
     * that runs past it gives up: the kernel lets its copies and products in
     * flight land, skips the rest of its work, marks the workspace's status
     * word and returns (see comba_workspace_status).  The outputs of such a
     * call are then incomplete. */
    unsigned int wait_limit_ns;
} comba_shape_t;

#define COMBA_FWD_EVENTS 5
#define COMBA_BWD_EVENTS 9

/*
 * Saved factors (training step without recomputation).
 *   comba_chunk_fwd with COMBA_SAVE_FACTORS also keeps everything the
 *   backward needs (chunk table, W, U, log-decays, the UT inverses M, the
 *   chunk-start states H_n, E = U - W H_n and, in bf16 at dk = dv = 128 and at
 *   dk = 256, the factor Z = Qhat - P W of the reverse scan's additive term) in
 *   its workspace, which must then
 *   hold comba_workspace_size(shape, 1) bytes (else COMBA_ERR_WORKSPACE).
 *   comba_chunk_bwd with COMBA_REUSE_FACTORS reads them from the workspace
 *   instead of recomputing the forward chunk factors and states.  The
 *   workspace must come unchanged from such a forward on the same shape and
 *   inputs; the library cannot check this.  Stage events of skipped kernels
 *   are recorded back to back.
 */
#define COMBA_SAVE_FACTORS 1
#define COMBA_REUSE_FACTORS 2

/*
 * Comba-iplr variant (table of state transitions for the Comba variants):
 * the transition alpha_t (I - 2 btilde_t k_t k_t^T) instead of
 * (alpha_t I - btilde_t k_t k_t^T), i.e. every formula above with the
 * feedback strength b beta_t replaced by 2 alpha_t b beta_t (gradients
 * included: dalpha gains the term through that factor).  A flag bit of
 * comba_chunk_fwd, comba_chunk_bwd (a backward that reuses saved factors must
 * use the variant of the forward that saved them) and comba_recurrent_step.
 */
#define COMBA_IPLR 4

/*
 * Gate and normalisation prologue (section 3.1 gates; L2-normalised q and k of
 * the neural-architecture section), for comba_chunk_fwd_gated and
 * comba_chunk_bwd_gated, which take raw q, k and gate pre-activations:
 *     q_hat = q / sqrt(|q|^2 + 1e-6)   (per token and head; likewise k)
 *     alpha = exp(-a_h softplus(g_alpha + c_h)),  beta = sigmoid(g_beta),
 *     b_h = sigmoid(b_raw_h)            (btilde = b beta)
 * and run the recurrence above on (q_hat, k_hat, v, alpha, beta, b, d).  The
 * shape passed to these calls and to comba_workspace_size must carry
 * COMBA_GATED (the workspace then also holds the prologue's outputs).
 */
#define COMBA_GATED 8

/*
 * The gated forward: as comba_chunk_fwd, with raw q, k [B,T,H,dk] (storage type),
 * gate pre-activations g_alpha, g_beta fp32 [B,T,H] and per-head fp32 a, c,
 * b_raw, d [H] (all required) instead of alpha, beta, b.  shape->flags must
 * contain COMBA_GATED and may add COMBA_SAVE_FACTORS (then the saved factors
 * include the prologue's outputs) and COMBA_IPLR.
 */
comba_status_t comba_chunk_fwd_gated(const comba_shape_t *shape,
                                     const void *q, const void *k, const void *v,
                                     const float *g_alpha, const float *g_beta,
                                     const float *a, const float *c, const float *b_raw, const float *d,
                                     const float *h0, void *o, float *hT,
                                     void *workspace, size_t workspace_bytes, comba_stream_t stream);

/*
 * The gated backward: gradients of L = <o,dO> + <hT,dhT> w.r.t. the raw inputs:
 * dq, dk (storage type), dv, dg_alpha, dg_beta fp32 [B,T,H], da, dc, dd fp32
 * [H], db_raw fp32 [H] or NULL, dh0 or NULL.  da, dc, db_raw and dd are sums over
 * all tokens in a fixed order.  shape->flags must contain COMBA_GATED and may
 * add COMBA_REUSE_FACTORS (after a gated forward with COMBA_SAVE_FACTORS on the
 * same workspace) and COMBA_IPLR.
 */
comba_status_t comba_chunk_bwd_gated(const comba_shape_t *shape,
                                     const void *q, const void *k, const void *v,
                                     const float *g_alpha, const float *g_beta,
                                     const float *a, const float *c, const float *b_raw, const float *d,
                                     const float *h0, const void *dO, const float *dhT,
                                     void *dq, void *dk, void *dv, float *dg_alpha, float *dg_beta,
                                     float *da, float *dc, float *db_raw, float *dd, float *dh0,
                                     void *workspace, size_t workspace_bytes, comba_stream_t stream);

/*
 * Comba-pk (appendix B.3, the "p" form of the recurrence): a per-token feedback
 * vector p_t, shaped like k_t, is read back from the state and corrects the query,
 * while k_t still writes the state:
 *     x_t = H_{t-1}^T p_t,  e_t = beta_t v_t - btilde_t x_t,
 *     H_t = alpha_t H_{t-1} + k_t e_t^T,  o_t = H_t^T (q_t - d p_t)
 * (transition alpha_t I - btilde_t p_t k_t^T on S = H^T; p = k is the form above,
 * p = b k with b = 1 the paper's way of folding b into p).  In the chunk form the
 * Gram inside the inverse becomes P K^T and W = M Diag(btilde gamma_{r-1}) P.  The
 * shape passed to the pk calls and to comba_workspace_size must carry COMBA_PK (the
 * workspace then also holds q - d p).  The pk calls run the same kernels as the
 * plain form at every head width (tcgen05 at bf16 dk = dv = 128; at head dim 256
 * the local gradients on the mma.sync kernel, as for the plain form).
 */
#define COMBA_PK 16

/*
 * Diagnostic flag of comba_chunk_fwd and comba_chunk_bwd (bf16, dk = dv = 128,
 * the tcgen05 kernels): the first tensor-core completion wait of every CTA of
 * the prep, output and local-gradient kernels waits on a barrier that nothing
 * arrives at, so it runs out after shape->wait_limit_ns.  The kernel then lets
 * its products land, skips its work and marks the workspace's status word, so
 * that a test can watch a device-side timeout reach the host
 * (comba_workspace_status) without faulting or hanging the GPU.  The call's
 * outputs are then meaningless.  Not for production use.
 */
#define COMBA_DIAG_STALL 32

/*
 * The pk forward: as comba_chunk_fwd plus p [B,T,H,dk] (storage type, required).
 * shape->flags must contain COMBA_PK and may add COMBA_SAVE_FACTORS and COMBA_IPLR.
 */
comba_status_t comba_chunk_fwd_pk(const comba_shape_t *shape,
                                  const void *q, const void *k, const void *v, const void *p,
                                  const float *alpha, const float *beta,
                                  const float *b, const float *d, const float *h0,
                                  void *o, float *hT,
                                  void *workspace, size_t workspace_bytes, comba_stream_t stream);

/*
 * The pk backward: as comba_chunk_bwd plus p and its gradient dp [B,T,H,dk]
 * (storage type, written).  dk then holds only the gradient through the state
 * write; dd = -sum_t p_t . dq_t.  shape->flags must contain COMBA_PK and may add
 * COMBA_REUSE_FACTORS (after a pk forward with COMBA_SAVE_FACTORS on the same
 * workspace and inputs; the backward then also reuses that forward's q - d p) and
 * COMBA_IPLR.
 */
comba_status_t comba_chunk_bwd_pk(const comba_shape_t *shape,
                                  const void *q, const void *k, const void *v, const void *p,
                                  const float *alpha, const float *beta,
                                  const float *b, const float *d, const float *h0,
                                  const void *dO, const float *dhT,
                                  void *dq, void *dk, void *dv, void *dp,
                                  float *dalpha, float *dbeta, float *db, float *dd, float *dh0,
                                  void *workspace, size_t workspace_bytes, comba_stream_t stream);

/*
 * Bytes of device workspace needed by comba_chunk_fwd (backward = 0) or
 * comba_chunk_bwd (backward = 1) for this shape.  Returns 0 for an invalid
 * shape.  The bound covers any cu_seqlens with the given T and num_seqs.
 */
size_t comba_workspace_size(const comba_shape_t *shape, int backward);

/*
 * Chunk-parallel forward (section 3.2).  Per chunk of 64 tokens: the
 * decay-masked, btilde-scaled Gram matrix, its unit-lower-triangular inverse
 * M = (I + strict_lower(Diag(btilde)(A^{(i-1)/j} * K K^T)))^{-1}, the WY/UT
 * factors W = M Diag(btilde*gamma_{r-1}) K and U = M Diag(beta) V
 * (Eq. "prepare WY_M"); then a sequential scan of the chunk states
 * H_{n+1} = gamma_C H_n + Kbar^T (U - W H_n); then the chunk outputs
 * O = Diag(gamma) Q~ H_n + Tril(Q~ K^T * A^{i/j}) (U - W H_n), Q~ = Q - d K.
 *
 *   q, k [B,T,H,dk]; v [B,T,H,dv]; alpha, beta fp32 [B,T,H];
 *   b fp32 [H] or NULL (b = 1); d fp32 [H];
 *   h0 fp32 [N,H,dk,dv] or NULL (zero state);
 *   o [B,T,H,dv] (written); hT fp32 [N,H,dk,dv] or NULL (final state, written).
 */
comba_status_t comba_chunk_fwd(const comba_shape_t *shape,
                               const void *q, const void *k, const void *v,
                               const float *alpha, const float *beta,
                               const float *b, const float *d, const float *h0,
                               void *o, float *hT,
                               void *workspace, size_t workspace_bytes, comba_stream_t stream);

/*
 * Chunk-parallel backward: exact gradients of
 *     L = <o, dO> + <hT, dhT>
 * through the forward above (the paper prints no backward; these are the
 * chain-rule derivatives of the chunk form).  The forward chunk factors and
 * chunk states are recomputed inside the call, or, with COMBA_REUSE_FACTORS,
 * read from a workspace that a forward with COMBA_SAVE_FACTORS filled.
 *
 *   inputs as comba_chunk_fwd, plus dO [B,T,H,dv] and dhT fp32 [N,H,dk,dv] or
 *   NULL (zero);
 *   dq, dk [B,T,H,dk], dv [B,T,H,dv] (storage type), dalpha, dbeta fp32
 *   [B,T,H], dd fp32 [H] (all written); db fp32 [H] or NULL (written when
 *   non-NULL; the gradient w.r.t. b, also when b == NULL meant b = 1);
 *   dh0 fp32 [N,H,dk,dv] or NULL (written when non-NULL).
 *   dalpha is d L / d alpha (not d L / d log alpha).
 *
 * The fp32 storage type supports dk, dv <= 64 in the backward.
 */
comba_status_t comba_chunk_bwd(const comba_shape_t *shape,
                               const void *q, const void *k, const void *v,
                               const float *alpha, const float *beta,
                               const float *b, const float *d, const float *h0,
                               const void *dO, const float *dhT,
                               void *dq, void *dk, void *dv,
                               float *dalpha, float *dbeta, float *db, float *dd, float *dh0,
                               void *workspace, size_t workspace_bytes, comba_stream_t stream);

/*
 * One decode token (appendix B.1, recurrent form) for Bd independent rows:
 *     x = H^T k, y = H^T (q - d k), e = beta v - b beta x,
 *     o = alpha y + e (k . (q - d k)),   H <- alpha H + k e^T
 * (o equals the new state applied to q - d k).  The state is read once and
 * written once, in place.
 *
 *   q, k [Bd,H,dk], v [Bd,H,dv], o [Bd,H,dv] (storage type `dtype`);
 *   alpha, beta fp32 [Bd,H]; b fp32 [H] or NULL; d fp32 [H];
 *   state fp32 [Bd,H,dk,dv], updated in place.
 *   dk in {64, 128, 256}; dv in {64, 128}, or 256 with dk >= 128 (either dtype);
 *   other widths are COMBA_ERR_UNSUPPORTED.
 *   flags: 0 or COMBA_IPLR (b beta replaced by 2 alpha b beta); other bits are
 *   COMBA_ERR_INVALID_ARG.
 */
comba_status_t comba_recurrent_step(int Bd, int H, int dk, int dv, comba_dtype_t dtype,
                                    const void *q, const void *k, const void *v,
                                    const float *alpha, const float *beta,
                                    const float *b, const float *d,
                                    float *state, void *o, int flags, comba_stream_t stream);

/*
 * One Comba-pk decode token: as comba_recurrent_step with the feedback vector
 * p [Bd,H,dk] (storage type, required) in place of k where the state is read
 * back and in the correction: x = H^T p, y = H^T (q - d p),
 * o = alpha y + e (k . (q - d p)), H <- alpha H + k e^T.
 */
comba_status_t comba_recurrent_step_pk(int Bd, int H, int dk, int dv, comba_dtype_t dtype,
                                       const void *q, const void *k, const void *v, const void *p,
                                       const float *alpha, const float *beta,
                                       const float *b, const float *d,
                                       float *state, void *o, int flags, comba_stream_t stream);

/*
 * Forward without a caller workspace, for callers that may not allocate
 * device memory (e.g. code running inside a framework's execute step that
 * forbids allocation, or a latency-critical loop that must not reach an
 * allocator).  The paper has no counterpart; this is a deployment variant of
 * comba_chunk_fwd with the same arguments minus the workspace, and bitwise
 * the same o and hT.  shape->flags may be 0 or COMBA_IPLR; any other flag
 * (saved factors, the gated or pk forms) returns COMBA_ERR_INVALID_ARG.
 *
 * Scratch comes from one file-scope device array of COMBA_STATIC_SCRATCH_BYTES
 * that every GPU loading this library holds until the process exits.  Shapes
 * whose comba_workspace_size(shape, 0) exceeds it return COMBA_ERR_WORKSPACE
 * without launching anything.  Each call looks up the array's device address
 * on the current device (cudaGetSymbolAddress); the first call on a device
 * also loads the library's device code there, so make it before any stream
 * capture.  All calls share the array: calls whose kernels may overlap on
 * the GPU race on it and must be serialised by the caller.  Nothing in it
 * needs to start zeroed.  No allocation is made.
 */
#define COMBA_STATIC_SCRATCH_BYTES (32u << 20)
comba_status_t comba_chunk_fwd_noalloc(const comba_shape_t *shape,
                                       const void *q, const void *k, const void *v,
                                       const float *alpha, const float *beta,
                                       const float *b, const float *d, const float *h0,
                                       void *o, float *hT, comba_stream_t stream);

/*
 * Status of the device-side waits of the calls that last used `workspace`.
 * Every kernel wait is bounded in time (comba_shape_t.wait_limit_ns); a wait
 * that gives up sets the status word in the workspace's first 4 bytes.  The
 * word is cleared by the first kernel of every forward call and of every
 * backward call that recomputes the forward's factors; a backward that reuses
 * saved factors adds to what its forward set.  This call waits for `stream`
 * (cudaStreamSynchronize), copies the word back with one cudaMemcpyAsync into
 * a host variable, and returns COMBA_ERR_TIMEOUT when it is set, COMBA_OK when
 * it is clear, COMBA_ERR_CUDA when the stream or the copy failed.  The word is
 * left as it is.  `workspace` NULL reads the word of the static scratch of
 * comba_chunk_fwd_noalloc on the current device.  Nothing is allocated.
 * (No counterpart in the paper: the hot-path boundary's error reporting.)
 */
comba_status_t comba_workspace_status(const void *workspace, comba_stream_t stream);

/* Static, human-readable name of a status code. */
const char *comba_status_string(comba_status_t status);

#ifdef __cplusplus
}
#endif

#endif /* COMBA_H */
