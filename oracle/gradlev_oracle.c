/*
 * gradlev_oracle.c -- the parity oracle for the GradLev token scans.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is a plain, slow, sequential CPU
 * restatement of what the scans compute, in fp64.  Only the test suite, the
 * package's smoke check and the bench's CPU-baseline leg may load it; the
 * CUDA library never links, includes or calls it, and it shares no code with
 * the CUDA path.
 *
 * What it computes (GradLev, Sec. 3, "Observation" and steps 2-3):
 *   The online learner with centered weight decay (Eq. 2),
 *       W_{t+1} = W_0 + alpha_t (W_t - W_0) - eta_t g_t x_t^T,   W at t=0 is W_0,
 *   driven by supplied costate proposals g_t := ghat_t (step 2, Eq. 3), and read
 *   at every token BEFORE that token's write:
 *       forward read   y_t      = W_t x_t                          (Eq. 3)
 *       costate read   gin_t    = W_t^T gout_t                     (Eq. 4)
 *   The reverse holds the incoming weights fixed (Sec. 3 step 3), so the costate
 *   read at token t needs only W_t: walking tokens in order and reading before
 *   writing is exactly "backpropagate through the stored per-token W_t".
 *
 * The two-layer MLP variant follows Appendix A (Eqs. online-forward,
 * online-reverse, online-update, scan1-scan2, reconstructed-reverse): both
 * matrices are read with pre-update weights, then written simultaneously.
 *
 * Everything is fp64; inputs arrive already upcast from the tensors the GPU
 * sees.  There is no blocking, chunking or reordering: one token at a time,
 * one dot product at a time.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Activation codes (same numbering as the public header's enum; restated here
 * so that the oracle includes nothing from the CUDA side). */
enum { OR_ACT_NONE = 0, OR_ACT_GELU_TANH = 1, OR_ACT_GELU_ERF = 2, OR_ACT_TANH = 3 };

/* sigma and sigma' (Sec. 3 step 3 uses sigma'(z) (.) g; App. E names the
 * tanh-approximate GELU).  Written from the formulas, using libm. */
static double act_f(int act, double z) {
    const double k0 = 0.7978845608028654; /* sqrt(2/pi) */
    switch (act) {
    case OR_ACT_GELU_TANH: return 0.5 * z * (1.0 + tanh(k0 * (z + 0.044715 * z * z * z)));
    case OR_ACT_GELU_ERF:  return 0.5 * z * (1.0 + erf(z / sqrt(2.0)));
    case OR_ACT_TANH:      return tanh(z);
    default:               return z;
    }
}

static double act_df(int act, double z) {
    const double k0 = 0.7978845608028654;
    switch (act) {
    case OR_ACT_GELU_TANH: {
        double u = k0 * (z + 0.044715 * z * z * z);
        double th = tanh(u);
        double du = k0 * (1.0 + 3.0 * 0.044715 * z * z);
        return 0.5 * (1.0 + th) + 0.5 * z * (1.0 - th * th) * du;
    }
    case OR_ACT_GELU_ERF: {
        double cdf = 0.5 * (1.0 + erf(z / sqrt(2.0)));
        double pdf = exp(-0.5 * z * z) * 0.3989422804014327; /* 1/sqrt(2 pi) */
        return cdf + z * pdf;
    }
    case OR_ACT_TANH: { double th = tanh(z); return 1.0 - th * th; }
    default: return 1.0;
    }
}

double oracle_act(int act, double z) { return act_f(act, z); }
double oracle_act_deriv(int act, double z) { return act_df(act, z); }

/* One write of Eq. 2: W <- W0 + alpha (W - W0) - eta g x^T. */
static void write_update(int m, int d, double* W, const double* W0, double alpha, double eta,
                         const double* g, const double* x) {
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < d; ++j) {
            double w = W[(size_t)i * d + j];
            if (alpha != 1.0) w = W0[(size_t)i * d + j] + alpha * (w - W0[(size_t)i * d + j]);
            W[(size_t)i * d + j] = w - eta * g[i] * x[j];
        }
}

/*
 * oracle_linear -- one adapted linear map y_t = W_t x_t over T tokens.
 *   x     [T][d]   layer inputs x_t
 *   ghat  [T][m]   costate proposals ghat_t (the writes)
 *   W0    [m][d]   slow initialisation
 *   eta   [T]      step size per token (Eq. 2 eta_t)
 *   alpha [T]      retention per token, or NULL for alpha_t = 1
 *   gout  [T][m]   incoming costates for the costate read, or NULL
 *   y     [T][m]   out: forward read W_t x_t, or NULL
 *   gin   [T][d]   out: costate read W_t^T gout_t, or NULL
 *   Wscr  [m][d]   scratch holding the running W_t
 * Reads precede the write at every token (Sec. 3 step 2: "read before each
 * write"), so y_0 = W_0 x_0 and gin_0 = W_0^T gout_0.
 */
void oracle_linear(int T, int d, int m, const double* x, const double* ghat, const double* W0,
                   const double* eta, const double* alpha, const double* gout, double* y,
                   double* gin, double* Wscr) {
    memcpy(Wscr, W0, sizeof(double) * (size_t)m * d);
    for (int t = 0; t < T; ++t) {
        const double* xt = x + (size_t)t * d;
        if (y) {
            for (int i = 0; i < m; ++i) {
                double s = 0.0;
                for (int j = 0; j < d; ++j) s += Wscr[(size_t)i * d + j] * xt[j];
                y[(size_t)t * m + i] = s;
            }
        }
        if (gin) {
            const double* gt = gout + (size_t)t * m;
            for (int j = 0; j < d; ++j) {
                double s = 0.0;
                for (int i = 0; i < m; ++i) s += Wscr[(size_t)i * d + j] * gt[i];
                gin[(size_t)t * d + j] = s;
            }
        }
        write_update(m, d, Wscr, W0, alpha ? alpha[t] : 1.0, eta[t], ghat + (size_t)t * m, xt);
    }
}

/*
 * oracle_linear_batch -- oracle_linear over U independent units (each its own
 * W0), in parallel over units.  Arrays are [U][...] contiguous; eta/alpha are
 * shared by all units ([T]).  nthreads <= 0 uses the OpenMP default.
 * Returns 0, or -1 if scratch could not be allocated.
 */
int oracle_linear_batch(int U, int T, int d, int m, const double* x, const double* ghat,
                        const double* W0, const double* eta, const double* alpha,
                        const double* gout, double* y, double* gin, int nthreads) {
    int err = 0;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel
    {
        double* W = (double*)malloc(sizeof(double) * (size_t)m * d);
        if (!W) {
#pragma omp atomic write
            err = -1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int u = 0; u < U; ++u) {
                oracle_linear(T, d, m, x + (size_t)u * T * d, ghat + (size_t)u * T * m,
                              W0 + (size_t)u * m * d, eta, alpha,
                              gout ? gout + (size_t)u * T * m : NULL,
                              y ? y + (size_t)u * T * m : NULL,
                              gin ? gin + (size_t)u * T * d : NULL, W);
            }
            free(W);
        }
    }
    return err;
}

/*
 * oracle_mlp -- the online two-layer MLP of Appendix A, token by token.
 *   z_t = W1_t x_t,  h_t = sigma(z_t),  y_t = W2_t h_t                 (online-forward)
 *   costate chain for an incoming gout_t (Sec. 3 step 3 applied twice):
 *     gh_t = W2_t^T gout_t,  gz_t = sigma'(z_t) (.) gh_t,  gx_t = W1_t^T gz_t
 *   writes (online-update, with the proposals as the written costates):
 *     W1 <- W10 + alpha (W1 - W10) - eta1_t ghz_t x_t^T
 *     W2 <- W20 + alpha (W2 - W20) - eta2_t ghy_t h_t^T
 * Deployment (Sec. 3, training objective paragraph; Appendix A: once a target is
 * scored, the maps are written with actual costates, not proposals): with ghz
 * NULL layer 1 writes its reconstructed gz_t, and with ghy NULL layer 2 writes
 * gout_t.  Either needs gout.
 * Widths: input d, hidden m, output k (Appendix A has k = d; Sec. 4.1 uses 4->7->3).
 * Shapes: x [T][d], ghz [T][m], ghy [T][k], W10 [m][d], W20 [k][m], gout [T][k].
 * Outputs (each nullable): z, h [T][m]; y [T][k]; gh, gz [T][m]; gx [T][d].
 * W1s [m][d], W2s [k][m], tmp [3m] are scratch.
 */
void oracle_mlp(int T, int d, int m, int k, int act, const double* x, const double* ghz,
                const double* ghy, const double* W10, const double* W20, const double* eta1,
                const double* eta2, const double* alpha, const double* gout, double* z, double* h,
                double* y, double* gh, double* gz, double* gx, double* W1s, double* W2s,
                double* tmp) {
    memcpy(W1s, W10, sizeof(double) * (size_t)m * d);
    memcpy(W2s, W20, sizeof(double) * (size_t)k * m);
    double* zt = tmp;          /* [m] */
    double* ht = tmp + m;      /* [m] */
    double* ght = tmp + 2 * m; /* [m] */
    for (int t = 0; t < T; ++t) {
        const double* xt = x + (size_t)t * d;
        for (int i = 0; i < m; ++i) {
            double s = 0.0;
            for (int j = 0; j < d; ++j) s += W1s[(size_t)i * d + j] * xt[j];
            zt[i] = s;
            ht[i] = act_f(act, s);
        }
        if (z) memcpy(z + (size_t)t * m, zt, sizeof(double) * m);
        if (h) memcpy(h + (size_t)t * m, ht, sizeof(double) * m);
        if (y) {
            for (int o = 0; o < k; ++o) {
                double s = 0.0;
                for (int i = 0; i < m; ++i) s += W2s[(size_t)o * m + i] * ht[i];
                y[(size_t)t * k + o] = s;
            }
        }
        if (gout) {
            const double* go = gout + (size_t)t * k;
            for (int i = 0; i < m; ++i) {
                double s = 0.0;
                for (int o = 0; o < k; ++o) s += W2s[(size_t)o * m + i] * go[o];
                ght[i] = s;
            }
            if (gh) memcpy(gh + (size_t)t * m, ght, sizeof(double) * m);
            for (int i = 0; i < m; ++i) ght[i] *= act_df(act, zt[i]);
            if (gz) memcpy(gz + (size_t)t * m, ght, sizeof(double) * m);
            if (gx) {
                for (int j = 0; j < d; ++j) {
                    double s = 0.0;
                    for (int i = 0; i < m; ++i) s += W1s[(size_t)i * d + j] * ght[i];
                    gx[(size_t)t * d + j] = s;
                }
            }
        }
        double a = alpha ? alpha[t] : 1.0;
        /* in deployment gz_t is still in ght: it is written before being overwritten */
        write_update(m, d, W1s, W10, a, eta1[t], ghz ? ghz + (size_t)t * m : ght, xt);
        write_update(k, m, W2s, W20, a, eta2[t], ghy ? ghy + (size_t)t * k : gout + (size_t)t * k,
                     ht);
    }
}

/* oracle_mlp over U independent sequences ([U][...] contiguous, shared W10/W20
 * and step arrays), in parallel over sequences.  Returns 0 or -1. */
int oracle_mlp_batch(int U, int T, int d, int m, int k, int act, const double* x,
                     const double* ghz, const double* ghy, const double* W10, const double* W20,
                     const double* eta1, const double* eta2, const double* alpha,
                     const double* gout, double* z, double* h, double* y, double* gh, double* gz,
                     double* gx, int nthreads) {
    int err = 0;
    if ((!ghz || !ghy) && !gout) return -2;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel
    {
        double* W1s = (double*)malloc(sizeof(double) * (size_t)m * d);
        double* W2s = (double*)malloc(sizeof(double) * (size_t)k * m);
        double* tmp = (double*)malloc(sizeof(double) * 3 * (size_t)m);
        if (!W1s || !W2s || !tmp) {
#pragma omp atomic write
            err = -1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int u = 0; u < U; ++u) {
                size_t tm = (size_t)u * T * m, td = (size_t)u * T * d, tk = (size_t)u * T * k;
                oracle_mlp(T, d, m, k, act, x + td, ghz ? ghz + tm : NULL, ghy ? ghy + tk : NULL,
                           W10, W20, eta1, eta2,
                           alpha, gout ? gout + tk : NULL, z ? z + tm : NULL, h ? h + tm : NULL,
                           y ? y + tk : NULL, gh ? gh + tm : NULL, gz ? gz + tm : NULL,
                           gx ? gx + td : NULL, W1s, W2s, tmp);
            }
        }
        free(W1s);
        free(W2s);
        free(tmp);
    }
    return err;
}

/*
 * oracle_suffix -- the anti-causal read of the writes, for outer gradients
 * through the reads (Sec. 3, practical architecture and training: the gates
 * are learned and their derivatives kept, the writes are detached):
 *     r_s = sum_{t > s} (k_t . q_s) v_t
 * walked backwards in time with R = sum_{t > s} v_t k_t^T (dv x dq), read before
 * its own write, the mirror image of the forward learner.
 *   q, k [T][dq], v [T][dv], r [T][dv]; R [dv][dq] is scratch.
 * For the forward read y_t = W_t x_t with per-token step sizes, the derivative
 * of sum_t u_t . y_t with respect to eta_s is -ghat_s . r_s (q = k = x, v = u).
 */
void oracle_suffix(int T, int dq, int dv, const double* q, const double* k, const double* v,
                   double* r, double* R) {
    memset(R, 0, sizeof(double) * (size_t)dv * dq);
    for (int s = T - 1; s >= 0; --s) {
        const double* qs = q + (size_t)s * dq;
        for (int i = 0; i < dv; ++i) {
            double acc = 0.0;
            for (int j = 0; j < dq; ++j) acc += R[(size_t)i * dq + j] * qs[j];
            r[(size_t)s * dv + i] = acc;
        }
        const double* ks = k + (size_t)s * dq;
        const double* vs = v + (size_t)s * dv;
        for (int i = 0; i < dv; ++i)
            for (int j = 0; j < dq; ++j) R[(size_t)i * dq + j] += vs[i] * ks[j];
    }
}

/* oracle_suffix over U independent units ([U][...] contiguous), in parallel. */
int oracle_suffix_batch(int U, int T, int dq, int dv, const double* q, const double* k,
                        const double* v, double* r, int nthreads) {
    int err = 0;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel
    {
        double* R = (double*)malloc(sizeof(double) * (size_t)dv * dq);
        if (!R) {
#pragma omp atomic write
            err = -1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int u = 0; u < U; ++u)
                oracle_suffix(T, dq, dv, q + (size_t)u * T * dq, k + (size_t)u * T * dq,
                              v + (size_t)u * T * dv, r + (size_t)u * T * dv, R);
            free(R);
        }
    }
    return err;
}

/*
 * oracle_gate_grads -- derivatives of an outer objective with respect to the gates
 * of one unit (Sec. 3, practical architecture and training: the gates are learned
 * and their derivatives kept, the writes detached).  The fast weights minus W0,
 * D_t = W_t - W0, follow Eq. 2:  D_0 = 0,  D_{t+1} = alpha_t D_t - eta_t ghat_t x_t^T.
 * Each read of W_t adds a_t^T W_t b_t to the objective: for the forward read
 * y_t = W_t x_t with outer gradient u_t, a = u and b = x; for the costate read
 * gin_t = W_t^T gout_t with outer gradient w_t, a = gout and b = w.  With
 *     R_j = sum_{s>j} (prod_{j<r<s} alpha_r) a_s b_s^T               (m x d)
 * the derivatives are
 *     dL/dalpha_j = <D_j, R_j>  (Frobenius),     dL/deta_j = -ghat_j^T R_j x_j,
 * and the function returns alpha_j dL/dalpha_j (the derivative in log alpha_j) in
 * g_alpha and dL/deta_j in g_eta.  W0 does not enter.
 * R is walked backwards (R_{T-1} = 0, R_{j-1} = alpha_j R_j + a_j b_j^T) and kept at
 * the last token of every block of GG_BLK tokens; inside a block it is recomputed
 * backwards from that copy while D_j is walked forwards.
 *   x [T][d], ghat [T][m], eta, alpha [T], a [T][m], b [T][d]; scratch holds
 *   (ceil(T / GG_BLK) + GG_BLK + 1) m d doubles.
 */
#define GG_BLK 64
void oracle_gate_grads(int T, int d, int m, const double* x, const double* ghat, const double* eta,
                       const double* alpha, const double* a, const double* b, double* g_alpha,
                       double* g_eta, double* scratch) {
    const size_t md = (size_t)m * d;
    const int nb = (T + GG_BLK - 1) / GG_BLK;
    double* ck = scratch;                   /* [nb][m][d] R at each block's last token */
    double* blk = ck + (size_t)nb * md;     /* [GG_BLK][m][d] R inside one block */
    double* D = blk + (size_t)GG_BLK * md;  /* [m][d] */
    /* backward: R_j for j = T-1 .. 0 in D (as scratch), copied at block ends */
    memset(D, 0, sizeof(double) * md);
    for (int j = T - 1; j >= 0; --j) {
        if (j == T - 1 || (j + 1) % GG_BLK == 0) memcpy(ck + (size_t)(j / GG_BLK) * md, D, sizeof(double) * md);
        if (j > 0) {
            const double* aj = a + (size_t)j * m;
            const double* bj = b + (size_t)j * d;
            for (int i = 0; i < m; ++i)
                for (int k = 0; k < d; ++k) D[(size_t)i * d + k] = alpha[j] * D[(size_t)i * d + k] + aj[i] * bj[k];
        }
    }
    /* forward: D_j, with R_j of the block recomputed backwards from its last token */
    memset(D, 0, sizeof(double) * md);
    for (int q = 0; q < nb; ++q) {
        const int j0 = q * GG_BLK;
        const int e = (j0 + GG_BLK < T ? j0 + GG_BLK : T) - 1;
        memcpy(blk + (size_t)(e - j0) * md, ck + (size_t)q * md, sizeof(double) * md);
        for (int j = e; j > j0; --j) {
            const double* Rj = blk + (size_t)(j - j0) * md;
            double* Rp = blk + (size_t)(j - 1 - j0) * md;
            const double* aj = a + (size_t)j * m;
            const double* bj = b + (size_t)j * d;
            for (int i = 0; i < m; ++i)
                for (int k = 0; k < d; ++k) Rp[(size_t)i * d + k] = alpha[j] * Rj[(size_t)i * d + k] + aj[i] * bj[k];
        }
        for (int j = j0; j <= e; ++j) {
            const double* Rj = blk + (size_t)(j - j0) * md;
            const double* xj = x + (size_t)j * d;
            const double* gj = ghat + (size_t)j * m;
            double f = 0.0, ge = 0.0;
            for (int i = 0; i < m; ++i) {
                double rx = 0.0;
                for (int k = 0; k < d; ++k) {
                    f += D[(size_t)i * d + k] * Rj[(size_t)i * d + k];
                    rx += Rj[(size_t)i * d + k] * xj[k];
                }
                ge += gj[i] * rx;
            }
            g_alpha[j] = alpha[j] * f;
            g_eta[j] = -ge;
            for (int i = 0; i < m; ++i)
                for (int k = 0; k < d; ++k)
                    D[(size_t)i * d + k] = alpha[j] * D[(size_t)i * d + k] - eta[j] * gj[i] * xj[k];
        }
    }
}

/* oracle_gate_grads over U independent units ([U][...] contiguous, gates [U][T]). */
int oracle_gate_grads_batch(int U, int T, int d, int m, const double* x, const double* ghat,
                            const double* eta, const double* alpha, const double* a, const double* b,
                            double* g_alpha, double* g_eta, int nthreads) {
    int err = 0;
    const size_t md = (size_t)m * d;
    const size_t ns = ((size_t)(T + GG_BLK - 1) / GG_BLK + GG_BLK + 1) * md;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel
    {
        double* scratch = (double*)malloc(sizeof(double) * ns);
        if (!scratch) {
#pragma omp atomic write
            err = -1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int u = 0; u < U; ++u)
                oracle_gate_grads(T, d, m, x + (size_t)u * T * d, ghat + (size_t)u * T * m,
                                  eta + (size_t)u * T, alpha + (size_t)u * T, a + (size_t)u * T * m,
                                  b + (size_t)u * T * d, g_alpha + (size_t)u * T, g_eta + (size_t)u * T,
                                  scratch);
            free(scratch);
        }
    }
    return err;
}

/* Threads the OpenMP runtime would use (for reporting the CPU baseline). */
int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
