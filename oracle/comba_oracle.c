/*
 * Comba reference oracle -- fp64 token recurrence, plain C.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file; it exists so that tests, the smoke check and the CPU
 * baseline leg of the benchmark can compare the CUDA library against an
 * obviously-correct definition.  It shares no code, header or constant with
 * the CUDA sources.
 *
 * What it computes (paper section 3, Eq. "comba-S", with the feedback strength
 * of section 3.1 and the recurrent listing of appendix B.1), per sequence n
 * and head h, in the state orientation H = S^T (dk x dv):
 *
 *   x_t = H_{t-1}^T k_t                         (state feedback read, no decay)
 *   e_t = beta_t v_t - btilde_t x_t,  btilde_t = b_h * beta_t
 *   H_t = alpha_t H_{t-1} + k_t e_t^T           (S_t = S_{t-1}(alpha - btilde k k^T) + beta v k^T)
 *   o_t = H_t^T (q_t - d_h k_t)                 (output correction)
 *
 * H_0 = h0 (zero if absent); hT = H_T.  No query scale (the paper has none).
 *
 * Variant 1 is Comba-iplr (table of state transitions for the Comba variants):
 * the transition alpha_t (I - 2 btilde_t k_t k_t^T), i.e. the same recurrence
 * with the feedback strength btilde_t replaced by 2 alpha_t b_h beta_t.
 *
 * Comba-pk (appendix B.3, the "p" form of the recurrence): a per-token feedback
 * vector p_t replaces k_t where the state is read back and in the output
 * correction, while k_t still writes the state:
 *
 *   x_t = H_{t-1}^T p_t,   e_t = beta_t v_t - btilde_t x_t,
 *   H_t = alpha_t H_{t-1} + k_t e_t^T,   o_t = H_t^T (q_t - d_h p_t)
 *
 * (transition alpha_t I - btilde_t p_t k_t^T on S).  p = NULL means p_t = k_t,
 * which is the form above; p = b k with b = 1 in the pk form is the same model.
 *
 * The backward pass is exact back-propagation through time of that
 * recurrence (the paper prints no backward; these are the chain-rule
 * derivatives of the four lines above).  States are checkpointed every
 * SEG tokens and each segment is recomputed before it is differentiated.
 *
 * Layouts (all row-major, doubles, host memory):
 *   q, k, p   [Ttot, H, dk]      v, o, dO  [Ttot, H, dv]
 *   alpha,beta[Ttot, H]          b, d      [H]  (b may be NULL: b = 1)
 *   h0, hT    [N, H, dk, dv]     cu        int64 [N+1], token offsets
 * A dense batch [B, T, H, D] is the packed layout with cu = {0, T, 2T, ...}.
 *
 * Units (n, h) are independent; they are spread over `nthreads` pthreads.
 * Per-head sums (db, dd) are formed from per-unit partials in a fixed order.
 */
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define SEG 64

typedef struct {
    int N, H, dk, dv;
    const int64_t *cu;
    const double *q, *k, *v, *alpha, *beta, *b, *d, *h0;
    const double *p; /* [Ttot, H, dk] feedback vectors (Comba-pk), or NULL: p_t = k_t */
    double *o, *hT;
    const double *dO, *dhT;
    double *dq, *dk_, *dv_, *dp, *dalpha, *dbeta, *dh0;
    double *db_part, *dd_part; /* [N*H] */
    int nthreads, tid;
    int status;
    int variant; /* 0: SPLR (alpha - btilde k k^T); 1: iplr alpha (I - 2 btilde k k^T) */
} job_t;

/* Feedback strength of token t relative to b_h beta_t: 1, or 2 alpha_t for iplr. */
static double fb_scale(const job_t *J, double a) { return J->variant == 1 ? 2.0 * a : 1.0; }

/* The feedback vector of token t (row offset tk = (t * H + h) * dk): p_t, or k_t. */
static const double *fb_vec(const job_t *J, size_t tk) { return J->p ? J->p + tk : J->k + tk; }

/* ---------------------------------------------------------------- forward */

static void fwd_unit(const job_t *J, int n, int h, double *Hs, double *x, double *e, double *qn)
{
    const int Hh = J->H, dk = J->dk, dv = J->dv;
    const double bh = J->b ? J->b[h] : 1.0;
    const double dh = J->d[h];
    const size_t ssz = (size_t)dk * dv;
    if (J->h0)
        memcpy(Hs, J->h0 + ((size_t)n * Hh + h) * ssz, ssz * sizeof(double));
    else
        memset(Hs, 0, ssz * sizeof(double));

    for (int64_t t = J->cu[n]; t < J->cu[n + 1]; ++t) {
        const double *kt = J->k + ((size_t)t * Hh + h) * dk;
        const double *ft = fb_vec(J, ((size_t)t * Hh + h) * dk);
        const double *qt = J->q + ((size_t)t * Hh + h) * dk;
        const double *vt = J->v + ((size_t)t * Hh + h) * dv;
        const double a = J->alpha[(size_t)t * Hh + h];
        const double be = J->beta[(size_t)t * Hh + h];
        const double bt = bh * be * fb_scale(J, a);
        /* x = H^T p (p = k unless given), read from the state before this token's update */
        for (int j = 0; j < dv; ++j) x[j] = 0.0;
        for (int i = 0; i < dk; ++i) {
            const double fi = ft[i];
            const double *row = Hs + (size_t)i * dv;
            for (int j = 0; j < dv; ++j) x[j] += row[j] * fi;
        }
        for (int j = 0; j < dv; ++j) e[j] = be * vt[j] - bt * x[j];
        for (int i = 0; i < dk; ++i) {
            const double ki = kt[i];
            double *row = Hs + (size_t)i * dv;
            for (int j = 0; j < dv; ++j) row[j] = a * row[j] + ki * e[j];
        }
        for (int i = 0; i < dk; ++i) qn[i] = qt[i] - dh * ft[i];
        double *ot = J->o + ((size_t)t * Hh + h) * dv;
        for (int j = 0; j < dv; ++j) ot[j] = 0.0;
        for (int i = 0; i < dk; ++i) {
            const double qi = qn[i];
            const double *row = Hs + (size_t)i * dv;
            for (int j = 0; j < dv; ++j) ot[j] += row[j] * qi;
        }
    }
    if (J->hT) memcpy(J->hT + ((size_t)n * Hh + h) * ssz, Hs, ssz * sizeof(double));
}

static void *fwd_worker(void *arg)
{
    job_t *J = (job_t *)arg;
    const size_t ssz = (size_t)J->dk * J->dv;
    double *Hs = (double *)malloc(ssz * sizeof(double));
    double *x = (double *)malloc((size_t)J->dv * sizeof(double));
    double *e = (double *)malloc((size_t)J->dv * sizeof(double));
    double *qn = (double *)malloc((size_t)J->dk * sizeof(double));
    if (!Hs || !x || !e || !qn) {
        J->status = 1;
    } else {
        for (int u = J->tid; u < J->N * J->H; u += J->nthreads) fwd_unit(J, u / J->H, u % J->H, Hs, x, e, qn);
    }
    free(Hs); free(x); free(e); free(qn);
    return NULL;
}

/* --------------------------------------------------------------- backward */

/*
 * One unit.  G holds dL/dH_t while walking t downwards.  For token t, with
 * P = H_{t-1} and f_t the feedback vector (p_t, or k_t), the local derivatives are
 *   G      += qn_t dO_t^T                 (o_t = H_t^T qn_t)
 *   dqn_t   = H_t dO_t
 *   dalpha_t= <G, P>
 *   de_t    = G^T k_t
 *   dk_t    = G e_t                       (k writes the state)
 *   df_t    = -btilde_t P de_t - d_h dqn_t (f is read back and corrects q)
 *   dv_t    = beta_t de_t
 *   dbeta_t = v_t.de_t - b_h x_t.de_t     (direct + through btilde)
 *   db     -= beta_t x_t.de_t
 *   dd     -= f_t.dqn_t
 *   G       = alpha_t G - btilde_t f_t de_t^T
 * With f = k (no p) dk_t collects both lines.
 */
static void bwd_unit(job_t *J, int n, int h, double *ckpt, double *seg, double *G,
                     double *x, double *e, double *qn, double *de, double *dqn)
{
    const int Hh = J->H, dk = J->dk, dv = J->dv;
    const double bh = J->b ? J->b[h] : 1.0;
    const double dh = J->d[h];
    const size_t ssz = (size_t)dk * dv;
    const int64_t t0 = J->cu[n], t1 = J->cu[n + 1];
    const int64_t len = t1 - t0;
    const int64_t nseg = (len + SEG - 1) / SEG;
    double db_acc = 0.0, dd_acc = 0.0;

    /* forward pass storing the state at the start of every segment */
    if (J->h0)
        memcpy(ckpt, J->h0 + ((size_t)n * Hh + h) * ssz, ssz * sizeof(double));
    else
        memset(ckpt, 0, ssz * sizeof(double));
    for (int64_t s = 0; s < nseg; ++s) {
        double *Hs = ckpt + (size_t)s * ssz;
        double *Hn = ckpt + (size_t)(s + 1) * ssz;
        memcpy(Hn, Hs, ssz * sizeof(double));
        const int64_t ta = t0 + s * SEG, tb = (ta + SEG < t1) ? ta + SEG : t1;
        for (int64_t t = ta; t < tb; ++t) {
            const double *kt = J->k + ((size_t)t * Hh + h) * dk;
            const double *ft = fb_vec(J, ((size_t)t * Hh + h) * dk);
            const double *vt = J->v + ((size_t)t * Hh + h) * dv;
            const double a = J->alpha[(size_t)t * Hh + h];
            const double be = J->beta[(size_t)t * Hh + h];
            for (int j = 0; j < dv; ++j) x[j] = 0.0;
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j) x[j] += Hn[(size_t)i * dv + j] * ft[i];
            for (int j = 0; j < dv; ++j) e[j] = be * vt[j] - bh * be * fb_scale(J, a) * x[j];
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j) Hn[(size_t)i * dv + j] = a * Hn[(size_t)i * dv + j] + kt[i] * e[j];
        }
    }

    if (J->dhT)
        memcpy(G, J->dhT + ((size_t)n * Hh + h) * ssz, ssz * sizeof(double));
    else
        memset(G, 0, ssz * sizeof(double));

    for (int64_t s = nseg - 1; s >= 0; --s) {
        const int64_t ta = t0 + s * SEG, tb = (ta + SEG < t1) ? ta + SEG : t1;
        const int m = (int)(tb - ta);
        /* recompute H_{ta-1+r} for r = 0..m into seg[r] */
        memcpy(seg, ckpt + (size_t)s * ssz, ssz * sizeof(double));
        for (int r = 0; r < m; ++r) {
            const int64_t t = ta + r;
            const double *kt = J->k + ((size_t)t * Hh + h) * dk;
            const double *ft = fb_vec(J, ((size_t)t * Hh + h) * dk);
            const double *vt = J->v + ((size_t)t * Hh + h) * dv;
            const double a = J->alpha[(size_t)t * Hh + h];
            const double be = J->beta[(size_t)t * Hh + h];
            const double *P = seg + (size_t)r * ssz;
            double *Q = seg + (size_t)(r + 1) * ssz;
            for (int j = 0; j < dv; ++j) x[j] = 0.0;
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j) x[j] += P[(size_t)i * dv + j] * ft[i];
            for (int j = 0; j < dv; ++j) e[j] = be * vt[j] - bh * be * fb_scale(J, a) * x[j];
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j) Q[(size_t)i * dv + j] = a * P[(size_t)i * dv + j] + kt[i] * e[j];
        }
        for (int r = m - 1; r >= 0; --r) {
            const int64_t t = ta + r;
            const size_t tk = ((size_t)t * Hh + h) * dk, tv = ((size_t)t * Hh + h) * dv;
            const double *kt = J->k + tk, *qt = J->q + tk, *vt = J->v + tv, *dOt = J->dO + tv;
            const double *ft = fb_vec(J, tk);
            const double a = J->alpha[(size_t)t * Hh + h];
            const double be = J->beta[(size_t)t * Hh + h];
            const double f = fb_scale(J, a);
            const double bt = bh * be * f;
            const double *P = seg + (size_t)r * ssz;       /* H_{t-1} */
            const double *Hc = seg + (size_t)(r + 1) * ssz; /* H_t     */
            /* recompute x_t, e_t */
            for (int j = 0; j < dv; ++j) x[j] = 0.0;
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j) x[j] += P[(size_t)i * dv + j] * ft[i];
            for (int j = 0; j < dv; ++j) e[j] = be * vt[j] - bt * x[j];
            for (int i = 0; i < dk; ++i) qn[i] = qt[i] - dh * ft[i];

            /* output: G += qn dO^T ; dqn = H_t dO */
            for (int i = 0; i < dk; ++i) {
                double acc = 0.0;
                for (int j = 0; j < dv; ++j) {
                    G[(size_t)i * dv + j] += qn[i] * dOt[j];
                    acc += Hc[(size_t)i * dv + j] * dOt[j];
                }
                dqn[i] = acc;
            }
            /* dalpha = <G, H_{t-1}> ; de = G^T k */
            double da = 0.0;
            for (int j = 0; j < dv; ++j) de[j] = 0.0;
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j) {
                    da += G[(size_t)i * dv + j] * P[(size_t)i * dv + j];
                    de[j] += G[(size_t)i * dv + j] * kt[i];
                }
            J->dalpha[(size_t)t * Hh + h] = da;
            /* dk = G e ; df = -btilde P de - d dqn (into dk when f = k) ; dq = dqn */
            double *dkt = J->dk_ + tk, *dqt = J->dq + tk, *dvt = J->dv_ + tv;
            double fdq = 0.0;
            for (int i = 0; i < dk; ++i) {
                double ge = 0.0, pde = 0.0;
                for (int j = 0; j < dv; ++j) {
                    ge += G[(size_t)i * dv + j] * e[j];
                    pde += P[(size_t)i * dv + j] * de[j];
                }
                const double df = -bt * pde - dh * dqn[i];
                if (J->p) {
                    dkt[i] = ge;
                    J->dp[tk + i] = df;
                } else {
                    dkt[i] = ge + df;
                }
                dqt[i] = dqn[i];
                fdq += ft[i] * dqn[i];
            }
            double vde = 0.0, xde = 0.0;
            for (int j = 0; j < dv; ++j) {
                dvt[j] = be * de[j];
                vde += vt[j] * de[j];
                xde += x[j] * de[j];
            }
            /* dbtilde = -x.de, through btilde = b beta f (f = 1, or 2 alpha for iplr) */
            J->dbeta[(size_t)t * Hh + h] = vde - bh * f * xde;
            db_acc -= be * f * xde;
            if (J->variant == 1) J->dalpha[(size_t)t * Hh + h] -= 2.0 * bh * be * xde;
            dd_acc -= fdq;
            /* carry to H_{t-1} */
            for (int i = 0; i < dk; ++i)
                for (int j = 0; j < dv; ++j)
                    G[(size_t)i * dv + j] = a * G[(size_t)i * dv + j] - bt * ft[i] * de[j];
        }
    }
    if (J->dh0) memcpy(J->dh0 + ((size_t)n * Hh + h) * ssz, G, ssz * sizeof(double));
    J->db_part[(size_t)n * Hh + h] = db_acc;
    J->dd_part[(size_t)n * Hh + h] = dd_acc;
}

static void *bwd_worker(void *arg)
{
    job_t *J = (job_t *)arg;
    const size_t ssz = (size_t)J->dk * J->dv;
    int64_t maxlen = 0;
    for (int n = 0; n < J->N; ++n)
        if (J->cu[n + 1] - J->cu[n] > maxlen) maxlen = J->cu[n + 1] - J->cu[n];
    const int64_t nseg = (maxlen + SEG - 1) / SEG;
    double *ckpt = (double *)malloc((size_t)(nseg + 1) * ssz * sizeof(double));
    double *seg = (double *)malloc((size_t)(SEG + 1) * ssz * sizeof(double));
    double *G = (double *)malloc(ssz * sizeof(double));
    double *x = (double *)malloc((size_t)J->dv * sizeof(double));
    double *e = (double *)malloc((size_t)J->dv * sizeof(double));
    double *de = (double *)malloc((size_t)J->dv * sizeof(double));
    double *qn = (double *)malloc((size_t)J->dk * sizeof(double));
    double *dqn = (double *)malloc((size_t)J->dk * sizeof(double));
    if (!ckpt || !seg || !G || !x || !e || !de || !qn || !dqn) {
        J->status = 1;
    } else {
        for (int u = J->tid; u < J->N * J->H; u += J->nthreads)
            bwd_unit(J, u / J->H, u % J->H, ckpt, seg, G, x, e, qn, de, dqn);
    }
    free(ckpt); free(seg); free(G); free(x); free(e); free(de); free(qn); free(dqn);
    return NULL;
}

/* ------------------------------------------------------------ thread pool */

static int run_pool(job_t *proto, void *(*fn)(void *))
{
    int nt = proto->nthreads < 1 ? 1 : proto->nthreads;
    const int units = proto->N * proto->H;
    if (nt > units) nt = units < 1 ? 1 : units;
    job_t *jobs = (job_t *)calloc((size_t)nt, sizeof(job_t));
    pthread_t *th = (pthread_t *)calloc((size_t)nt, sizeof(pthread_t));
    if (!jobs || !th) { free(jobs); free(th); return 1; }
    for (int i = 0; i < nt; ++i) {
        jobs[i] = *proto;
        jobs[i].nthreads = nt;
        jobs[i].tid = i;
        jobs[i].status = 0;
    }
    int started = 0, rc = 0;
    for (int i = 1; i < nt; ++i) {
        if (pthread_create(&th[i], NULL, fn, &jobs[i]) != 0) { rc = 1; break; }
        started = i;
    }
    if (rc) {
        for (int i = 1; i <= started; ++i) pthread_join(th[i], NULL);
        free(jobs); free(th);
        return 1;
    }
    fn(&jobs[0]);
    for (int i = 1; i < nt; ++i) pthread_join(th[i], NULL);
    for (int i = 0; i < nt; ++i) rc |= jobs[i].status;
    free(jobs); free(th);
    return rc;
}

/* --------------------------------------------------------------- exports */

int comba_oracle_fwd(int N, const int64_t *cu, int H, int dk, int dv,
                     const double *q, const double *k, const double *v, const double *p,
                     const double *alpha, const double *beta, const double *b, const double *d,
                     const double *h0, double *o, double *hT, int nthreads, int variant)
{
    job_t J;
    memset(&J, 0, sizeof(J));
    J.variant = variant;
    J.N = N; J.H = H; J.dk = dk; J.dv = dv; J.cu = cu;
    J.q = q; J.k = k; J.v = v; J.p = p; J.alpha = alpha; J.beta = beta; J.b = b; J.d = d; J.h0 = h0;
    J.o = o; J.hT = hT; J.nthreads = nthreads;
    return run_pool(&J, fwd_worker);
}

int comba_oracle_bwd(int N, const int64_t *cu, int H, int dk, int dv,
                     const double *q, const double *k, const double *v, const double *p,
                     const double *alpha, const double *beta, const double *b, const double *d,
                     const double *h0, const double *dO, const double *dhT,
                     double *dq, double *dk_, double *dv_, double *dp, double *dalpha, double *dbeta,
                     double *db, double *dd, double *dh0, int nthreads, int variant)
{
    job_t J;
    memset(&J, 0, sizeof(J));
    J.variant = variant;
    J.N = N; J.H = H; J.dk = dk; J.dv = dv; J.cu = cu;
    J.q = q; J.k = k; J.v = v; J.p = p; J.alpha = alpha; J.beta = beta; J.b = b; J.d = d; J.h0 = h0;
    J.dO = dO; J.dhT = dhT;
    J.dq = dq; J.dk_ = dk_; J.dv_ = dv_; J.dp = dp; J.dalpha = dalpha; J.dbeta = dbeta; J.dh0 = dh0;
    if (p && !dp) return 1;
    J.nthreads = nthreads;
    J.db_part = (double *)calloc((size_t)N * H, sizeof(double));
    J.dd_part = (double *)calloc((size_t)N * H, sizeof(double));
    if (!J.db_part || !J.dd_part) { free(J.db_part); free(J.dd_part); return 1; }
    int rc = run_pool(&J, bwd_worker);
    for (int h = 0; h < H; ++h) {
        double sb = 0.0, sd = 0.0;
        for (int n = 0; n < N; ++n) { sb += J.db_part[(size_t)n * H + h]; sd += J.dd_part[(size_t)n * H + h]; }
        if (db) db[h] = sb;
        dd[h] = sd;
    }
    free(J.db_part); free(J.dd_part);
    return rc;
}

/*
 * One decode token for Bd independent (row, head) states, updated in place:
 * the same four lines as the forward, applied once.  q,k,p [Bd,H,dk], v,o
 * [Bd,H,dv], alpha,beta [Bd,H], state [Bd,H,dk,dv].  Rows are the N of the
 * thread pool; the state is indexed by (row, head) like h0.
 */
static void *step_worker(void *arg)
{
    job_t *J = (job_t *)arg;
    const int Hh = J->H, dk = J->dk, dv = J->dv;
    double *x = (double *)malloc((size_t)dv * sizeof(double));
    double *e = (double *)malloc((size_t)dv * sizeof(double));
    double *qn = (double *)malloc((size_t)dk * sizeof(double));
    if (!x || !e || !qn) {
        J->status = 1;
    } else {
        for (int u = J->tid; u < J->N * Hh; u += J->nthreads) {
            const int h = u % Hh;
            const double *kt = J->k + (size_t)u * dk, *qt = J->q + (size_t)u * dk, *vt = J->v + (size_t)u * dv;
            const double *ft = fb_vec(J, (size_t)u * dk);
            double *Hs = J->hT + (size_t)u * dk * dv;
            const double a = J->alpha[u], be = J->beta[u];
            const double bt = (J->b ? J->b[h] : 1.0) * be * fb_scale(J, a);
            for (int j = 0; j < dv; ++j) x[j] = 0.0;
            for (int r = 0; r < dk; ++r)
                for (int j = 0; j < dv; ++j) x[j] += Hs[(size_t)r * dv + j] * ft[r];
            for (int j = 0; j < dv; ++j) e[j] = be * vt[j] - bt * x[j];
            for (int r = 0; r < dk; ++r)
                for (int j = 0; j < dv; ++j) Hs[(size_t)r * dv + j] = a * Hs[(size_t)r * dv + j] + kt[r] * e[j];
            for (int r = 0; r < dk; ++r) qn[r] = qt[r] - J->d[h] * ft[r];
            double *ot = J->o + (size_t)u * dv;
            for (int j = 0; j < dv; ++j) ot[j] = 0.0;
            for (int r = 0; r < dk; ++r)
                for (int j = 0; j < dv; ++j) ot[j] += Hs[(size_t)r * dv + j] * qn[r];
        }
    }
    free(x); free(e); free(qn);
    return NULL;
}

int comba_oracle_step(int Bd, int H, int dk, int dv,
                      const double *q, const double *k, const double *v, const double *p,
                      const double *alpha, const double *beta, const double *b, const double *d,
                      double *state, double *o, int nthreads, int variant)
{
    job_t J;
    memset(&J, 0, sizeof(J));
    J.variant = variant;
    J.N = Bd; J.H = H; J.dk = dk; J.dv = dv;
    J.q = q; J.k = k; J.v = v; J.p = p; J.alpha = alpha; J.beta = beta; J.b = b; J.d = d;
    J.hT = state; J.o = o; J.nthreads = nthreads;
    return run_pool(&J, step_worker);
}
