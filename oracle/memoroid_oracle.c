/*
 * memoroid_oracle.c -- plain fp64 CPU oracle for the resettable memoroid scans.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path links, loads or calls
 * this file: only the test suite, the smoke check and the benchmark's CPU
 * baseline use it.  It shares no code, header or constant with the CUDA path.
 *
 * Every routine is a direct, unblocked transcription of a definition from
 * "Recurrent Reinforcement Learning with Memoroids" (arXiv 2402.09900):
 *
 *   - the memoroid state sequence h_t = e_I . f(P_0) . ... . f(P_t)
 *     (Definition 3.1, the equation giving h_t and s_t);
 *   - the resettable monoid transform (A,b) o (A',b') =
 *     ((A (1-b') + e_I b') . A', b or b') with identity (e_I, 0) (Theorem 3.2),
 *     read as a select: when b' = 1 the left operand is replaced by e_I;
 *   - the S5 / LRU monoid (X,x) . (X',x') = (X'X, X'x + x') with e_I = (I, 0),
 *     here with diagonal X (Appendix "Simplified State Space Models" and
 *     "Linear Recurrent Unit");
 *   - the Linear Transformer sum monoid (X + X') (Appendix "Linear
 *     Transformer"), generalised with a per-step decay gamma_t that multiplies
 *     the carried state, read out as y_t = S_t^T q_t;
 *   - the discounted-return and GAE memoroids (a, r) . (a', r') =
 *     (a a', a r' + r), f = (gamma, r) resp. (gamma lambda, delta) (Appendix
 *     "The Discounted Return as a Memoroid" and "The Generalized Advantage
 *     Estimate as a Memoroid"), evaluated for every step of every episode.
 *
 * Conventions (readings of the paper, listed in the design notes):
 *   - b_t = 1 on the first step of an episode (Section 2.1).
 *   - Diagonal scan: within an episode h_t = lambda_t * h_{t-1} + u_t and the
 *     head step keeps its own f(P): h_s = u_s.  A tape whose row begins with
 *     b_0 = 0 continues an earlier episode from h0 (h0 = NULL means e_I = 0).
 *   - Backward passes use PyTorch's complex-gradient convention
 *     (grad = dL/dRe + i dL/dIm), for which the holomorphic chain rule of
 *     z = a*w reads grad_w = conj(a) * grad_z.
 *
 * All routines return 0 on success and a negative value on a bad argument.
 * Arrays are row-major; complex arrays are interleaved (re, im) doubles,
 * i.e. C99 double complex.
 */
#include <complex.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef double complex cplx;

/* Thread count used by the parallel loops over independent channels, heads
 * and tapes (1 when built without OpenMP). */
void oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* The resettable S5/LRU monoid for one diagonal channel (Theorem 3.2 applied
 * to the diagonal S5/LRU monoid).  An element is ((a, x), b): a is the
 * product of the lambdas, x the state, b the begin flag.                    */
/* ------------------------------------------------------------------------ */

void oracle_diag_combine(const double *left, int b_left, const double *right, int b_right,
                         double *out, int *b_out)
{
    /* left, right, out: [a_re, a_im, x_re, x_im] */
    cplx a = left[0] + I * left[1], x = left[2] + I * left[3];
    cplx a2 = right[0] + I * right[1], x2 = right[2] + I * right[3];
    cplx ra, rx;
    if (b_right) {
        /* (A,b) o (A',1) = (e_I . A', 1) = A'  (first row of the b'=1 cases) */
        ra = a2;
        rx = x2;
    } else {
        /* (A,b) o (A',0) = (A . A', b);  (a,x).(a',x') = (a' a, a' x + x') */
        ra = a2 * a;
        rx = a2 * x + x2;
    }
    out[0] = creal(ra); out[1] = cimag(ra);
    out[2] = creal(rx); out[3] = cimag(rx);
    *b_out = (b_left || b_right) ? 1 : 0;
}

/* lambda for tape b, step t, channel d */
static inline cplx lam_at(const cplx *lambda, int per_step, int64_t b, int64_t t, int64_t L,
                          int64_t D, int64_t d)
{
    return per_step ? lambda[(b * L + t) * D + d] : lambda[d];
}

/*
 * Diagonal scan, forward: the definition, episode by episode.
 * lambda: [D] or [B,L,D]; u, h: [B,L,D]; start: [B,L]; h0, h_last: [B,D] or NULL.
 */
int oracle_diag_fwd(int64_t B, int64_t L, int64_t D, const cplx *lambda, int lambda_per_step,
                    const cplx *u, const uint8_t *start, const cplx *h0, cplx *h, cplx *h_last)
{
    if (B < 0 || L < 0 || D < 0) return -1;
    if (L > 0 && (!lambda || !u || !start || !h)) return -1;
#pragma omp parallel for collapse(2) schedule(static)
    for (int64_t b = 0; b < B; ++b) {
        for (int64_t d = 0; d < D; ++d) {
            int64_t s = 0;
            while (s < L) {
                /* episode [s, e): next begin flag after s, or the tape end */
                int64_t e = s + 1;
                while (e < L && !start[b * L + e]) ++e;
                cplx prev;
                if (start[b * L + s]) {
                    prev = 0.0; /* e_I; unused: the head keeps its own f(P) */
                } else {
                    /* only possible at s = 0: a row that continues an episode */
                    prev = h0 ? h0[b * D + d] : 0.0;
                }
                for (int64_t t = s; t < e; ++t) {
                    cplx ut = u[(b * L + t) * D + d];
                    cplx ht = (t == s && start[b * L + s])
                                  ? ut
                                  : lam_at(lambda, lambda_per_step, b, t, L, D, d) * prev + ut;
                    h[(b * L + t) * D + d] = ht;
                    prev = ht;
                }
                s = e;
            }
            if (h_last) {
                h_last[b * D + d] = (L > 0) ? h[(b * L + L - 1) * D + d] : (h0 ? h0[b * D + d] : 0.0);
            }
        }
    }
    return 0;
}

/*
 * Diagonal scan, forward, by folding the resettable combine from the identity
 * g_I = (e_I, 0) (Definition 3.1 with Theorem 3.2).  The element lifted from
 * step t is ((lambda_t, u_t), b_t).  A row that starts with b_0 = 0 folds from
 * ((1, h0), 0) instead of g_I.
 */
int oracle_diag_fold(int64_t B, int64_t L, int64_t D, const cplx *lambda, int lambda_per_step,
                     const cplx *u, const uint8_t *start, const cplx *h0, cplx *h)
{
    if (B < 0 || L < 0 || D < 0) return -1;
    for (int64_t b = 0; b < B; ++b) {
        for (int64_t d = 0; d < D; ++d) {
            double acc[4] = {1.0, 0.0, h0 ? creal(h0[b * D + d]) : 0.0, h0 ? cimag(h0[b * D + d]) : 0.0};
            int acc_b = 0;
            for (int64_t t = 0; t < L; ++t) {
                cplx l = lam_at(lambda, lambda_per_step, b, t, L, D, d);
                cplx x = u[(b * L + t) * D + d];
                double el[4] = {creal(l), cimag(l), creal(x), cimag(x)};
                double out[4];
                int ob;
                oracle_diag_combine(acc, acc_b, el, start[b * L + t], out, &ob);
                memcpy(acc, out, sizeof(acc));
                acc_b = ob;
                h[(b * L + t) * D + d] = acc[2] + I * acc[3];
            }
        }
    }
    return 0;
}

/*
 * Diagonal scan, backward (reverse-mode of the forward definition).
 * Inputs: the forward's h [B,L,D], upstream g = dL/dh [B,L,D], g_last =
 * dL/dh_last [B,D] or NULL.  The adjoint of h_t is
 *     delta_t = g_t + [b_{t+1} = 0] conj(lambda_{t+1}) delta_{t+1},
 *     delta_{L-1} = g_{L-1} + g_last,
 * and grad_u_t = delta_t, grad_lambda_t = [b_t = 0] delta_t conj(h_{t-1})
 * (h_{-1} = h0, or 0 when h0 is NULL), grad_h0 = [b_0 = 0] conj(lambda_0) delta_0.
 * grad_lambda is [D] (summed over B and L) for a per-channel lambda and
 * [B,L,D] for a per-step lambda.  Any output may be NULL to skip it.
 */
int oracle_diag_bwd(int64_t B, int64_t L, int64_t D, const cplx *lambda, int lambda_per_step,
                    const uint8_t *start, const cplx *h0, const cplx *h, const cplx *g,
                    const cplx *g_last, cplx *grad_u, cplx *grad_lambda, cplx *grad_h0)
{
    if (B < 0 || L < 0 || D < 0) return -1;
    if (grad_lambda && !lambda_per_step) {
        for (int64_t d = 0; d < D; ++d) grad_lambda[d] = 0.0;
    }
#pragma omp parallel for schedule(static)
    for (int64_t d = 0; d < D; ++d) {
        cplx lam_sum = 0.0;
        for (int64_t b = 0; b < B; ++b) {
            cplx delta_next = 0.0; /* delta_{t+1} */
            for (int64_t t = L - 1; t >= 0; --t) {
                cplx delta = g[(b * L + t) * D + d];
                if (t == L - 1) {
                    if (g_last) delta += g_last[b * D + d];
                } else if (!start[b * L + t + 1]) {
                    delta += conj(lam_at(lambda, lambda_per_step, b, t + 1, L, D, d)) * delta_next;
                }
                if (grad_u) grad_u[(b * L + t) * D + d] = delta;
                if (grad_lambda) {
                    cplx gl = 0.0;
                    if (!start[b * L + t]) {
                        cplx hprev = (t > 0) ? h[(b * L + t - 1) * D + d] : (h0 ? h0[b * D + d] : 0.0);
                        gl = delta * conj(hprev);
                    }
                    if (lambda_per_step) grad_lambda[(b * L + t) * D + d] = gl;
                    else lam_sum += gl;
                }
                delta_next = delta;
            }
            if (grad_h0) {
                grad_h0[b * D + d] = (L > 0 && !start[b * L])
                                         ? conj(lam_at(lambda, lambda_per_step, b, 0, L, D, d)) * delta_next
                                         : (L == 0 && g_last ? g_last[b * D + d] : 0.0);
            }
        }
        if (grad_lambda && !lambda_per_step) grad_lambda[d] = lam_sum;
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Decayed linear-attention memoroid.                                        */
/*   S_t = [b_t = 0] gamma_t S_{t-1} + k_t v_t^T,   y_t = S_t^T q_t           */
/* (sum monoid of the Linear Transformer with a multiplicative decay on the  */
/* carried state; the head step of an episode starts from e_I = 0).          */
/* ------------------------------------------------------------------------ */

static inline double gam_at(const double *gamma, int per_step, int64_t b, int64_t t, int64_t L,
                            int64_t H, int64_t hh)
{
    return per_step ? gamma[(b * L + t) * H + hh] : gamma[hh];
}

/*
 * q, k: [B,L,H,dk]; v: [B,L,H,dv]; gamma: [H] or [B,L,H]; start: [B,L];
 * S0, S_last: [B,H,dk,dv] or NULL; y: [B,L,H,dv].
 */
int oracle_linattn_fwd(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, const double *q,
                       const double *k, const double *v, const double *gamma, int gamma_per_step,
                       const uint8_t *start, const double *S0, double *y, double *S_last)
{
    if (B < 0 || L < 0 || H < 0 || dk <= 0 || dv <= 0) return -1;
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int64_t b = 0; b < B; ++b) {
        for (int64_t hh = 0; hh < H; ++hh) {
            double *S = (double *)calloc((size_t)(dk * dv), sizeof(double));
            if (S0) memcpy(S, S0 + (b * H + hh) * dk * dv, sizeof(double) * dk * dv);
            for (int64_t t = 0; t < L; ++t) {
                const double *kt = k + ((b * L + t) * H + hh) * dk;
                const double *vt = v + ((b * L + t) * H + hh) * dv;
                const double *qt = q + ((b * L + t) * H + hh) * dk;
                double gt = start[b * L + t] ? 0.0 : gam_at(gamma, gamma_per_step, b, t, L, H, hh);
                for (int64_t i = 0; i < dk; ++i)
                    for (int64_t j = 0; j < dv; ++j)
                        S[i * dv + j] = (start[b * L + t] ? 0.0 : gt * S[i * dv + j]) + kt[i] * vt[j];
                double *yt = y + ((b * L + t) * H + hh) * dv;
                for (int64_t j = 0; j < dv; ++j) {
                    double acc = 0.0;
                    for (int64_t i = 0; i < dk; ++i) acc += S[i * dv + j] * qt[i];
                    yt[j] = acc;
                }
            }
            if (S_last) memcpy(S_last + (b * H + hh) * dk * dv, S, sizeof(double) * dk * dv);
            free(S);
        }
    }
    return 0;
}

/*
 * Backward of oracle_linattn_fwd, by the transposed recurrence:
 *   dS_t = q_t dy_t^T + [b_{t+1} = 0] gamma_{t+1} dS_{t+1}   (dS_{L-1} += dS_last)
 *   dq_t = S_t dy_t,  dk_t = dS_t v_t,  dv_t = dS_t^T k_t,
 *   dgamma_t = [b_t = 0] <dS_t, S_{t-1}>_F,  dS0 = [b_0 = 0] gamma_0 dS_0.
 * The forward states of each episode are recomputed and kept for the reverse
 * sweep.  dgamma is [H] (summed over B, L) or [B,L,H] for a per-step gamma.
 * Any output may be NULL.
 */
int oracle_linattn_bwd(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, const double *q,
                       const double *k, const double *v, const double *gamma, int gamma_per_step,
                       const uint8_t *start, const double *S0, const double *dy,
                       const double *dS_last, double *dq, double *dkk, double *dvv, double *dgamma,
                       double *dS0)
{
    if (B < 0 || L < 0 || H < 0 || dk <= 0 || dv <= 0) return -1;
    const int64_t M = dk * dv;
    double *gsum = NULL;
    if (dgamma && !gamma_per_step) {
        gsum = (double *)calloc((size_t)(B * H > 0 ? B * H : 1), sizeof(double));
    }
    int bad = 0;
#pragma omp parallel for collapse(2) schedule(dynamic)
    for (int64_t b = 0; b < B; ++b) {
        for (int64_t hh = 0; hh < H; ++hh) {
            double *dS = (double *)calloc((size_t)M, sizeof(double));
            double gacc = 0.0;
            /* episodes in reverse order; [s, e) */
            int64_t e = L;
            while (e > 0) {
                int64_t s = e - 1;
                while (s > 0 && !start[b * L + s]) --s;
                const int64_t n = e - s;
                /* states S_{s-1} .. S_{e-1}: slot 0 holds the incoming state */
                double *St = (double *)calloc((size_t)((n + 1) * M), sizeof(double));
                if (!St) { bad = 1; break; }
                if (!start[b * L + s] && S0) memcpy(St, S0 + (b * H + hh) * M, sizeof(double) * M);
                for (int64_t t = s; t < e; ++t) {
                    const double *kt = k + ((b * L + t) * H + hh) * dk;
                    const double *vt = v + ((b * L + t) * H + hh) * dv;
                    double gt = start[b * L + t] ? 0.0 : gam_at(gamma, gamma_per_step, b, t, L, H, hh);
                    double *prev = St + (t - s) * M, *cur = St + (t - s + 1) * M;
                    for (int64_t i = 0; i < dk; ++i)
                        for (int64_t j = 0; j < dv; ++j)
                            cur[i * dv + j] = (start[b * L + t] ? 0.0 : gt * prev[i * dv + j]) + kt[i] * vt[j];
                }
                /* reverse sweep */
                for (int64_t t = e - 1; t >= s; --t) {
                    const double *kt = k + ((b * L + t) * H + hh) * dk;
                    const double *vt = v + ((b * L + t) * H + hh) * dv;
                    const double *qt = q + ((b * L + t) * H + hh) * dk;
                    const double *dyt = dy + ((b * L + t) * H + hh) * dv;
                    if (t == e - 1) {
                        /* the step after e-1 starts a new episode (or is past the tape) */
                        for (int64_t x = 0; x < M; ++x) dS[x] = 0.0;
                        if (e == L && dS_last) memcpy(dS, dS_last + (b * H + hh) * M, sizeof(double) * M);
                    } else {
                        double gn = gam_at(gamma, gamma_per_step, b, t + 1, L, H, hh);
                        for (int64_t x = 0; x < M; ++x) dS[x] *= gn;
                    }
                    for (int64_t i = 0; i < dk; ++i)
                        for (int64_t j = 0; j < dv; ++j) dS[i * dv + j] += qt[i] * dyt[j];
                    const double *Scur = St + (t - s + 1) * M, *Sprev = St + (t - s) * M;
                    if (dq) {
                        double *o = dq + ((b * L + t) * H + hh) * dk;
                        for (int64_t i = 0; i < dk; ++i) {
                            double acc = 0.0;
                            for (int64_t j = 0; j < dv; ++j) acc += Scur[i * dv + j] * dyt[j];
                            o[i] = acc;
                        }
                    }
                    if (dkk) {
                        double *o = dkk + ((b * L + t) * H + hh) * dk;
                        for (int64_t i = 0; i < dk; ++i) {
                            double acc = 0.0;
                            for (int64_t j = 0; j < dv; ++j) acc += dS[i * dv + j] * vt[j];
                            o[i] = acc;
                        }
                    }
                    if (dvv) {
                        double *o = dvv + ((b * L + t) * H + hh) * dv;
                        for (int64_t j = 0; j < dv; ++j) {
                            double acc = 0.0;
                            for (int64_t i = 0; i < dk; ++i) acc += dS[i * dv + j] * kt[i];
                            o[j] = acc;
                        }
                    }
                    double dg = 0.0;
                    if (!start[b * L + t]) {
                        for (int64_t x = 0; x < M; ++x) dg += dS[x] * Sprev[x];
                    }
                    if (dgamma) {
                        if (gamma_per_step) dgamma[(b * L + t) * H + hh] = dg;
                        else gacc += dg;
                    }
                }
                if (s == 0 && dS0) {
                    double *o = dS0 + (b * H + hh) * M;
                    double g0 = gam_at(gamma, gamma_per_step, b, 0, L, H, hh);
                    for (int64_t x = 0; x < M; ++x) o[x] = start[b * L] ? 0.0 : g0 * dS[x];
                }
                free(St);
                e = s;
            }
            if (L == 0 && dS0) {
                double *o = dS0 + (b * H + hh) * M;
                for (int64_t x = 0; x < M; ++x) o[x] = dS_last ? dS_last[(b * H + hh) * M + x] : 0.0;
            }
            if (gsum) gsum[b * H + hh] = gacc;
            free(dS);
        }
    }
    if (gsum) {
        for (int64_t hh = 0; hh < H; ++hh) {
            double acc = 0.0;
            for (int64_t b = 0; b < B; ++b) acc += gsum[b * H + hh];
            dgamma[hh] = acc;
        }
        free(gsum);
    }
    return bad ? -2 : 0;
}

/* ------------------------------------------------------------------------ */
/* Episode index list I <-> begin flags (Algorithm 1: I = where(b)).         */
/* ------------------------------------------------------------------------ */

int oracle_starts_from_offsets(const int64_t *offsets, int64_t E, int64_t L, uint8_t *start)
{
    if (E < 0 || L < 0) return -1;
    for (int64_t t = 0; t < L; ++t) start[t] = 0;
    for (int64_t i = 0; i < E; ++i) {
        if (offsets[i] >= 0 && offsets[i] < L) start[offsets[i]] = 1;
    }
    return 0;
}

int64_t oracle_offsets_from_starts(const uint8_t *start, int64_t L, int64_t *offsets)
{
    int64_t n = 0;
    for (int64_t t = 0; t < L; ++t) {
        if (start[t]) offsets[n++] = t;
    }
    return n;
}


/* ------------------------------------------------------------------------ */
/* Discounted return and GAE per step, reset at episode boundaries           */
/* ------------------------------------------------------------------------ */
/*
 * The return memoroid folds (1,0) . (gamma, r_t) . (gamma, r_{t+1}) . ... and
 * its second element is sum_l gamma^l r_{t+l}; evaluated for every step t of
 * an episode it is the suffix sum
 *     G_t = sum_{l = 0}^{e - 1 - t} gamma^l r_{t+l}        (episode [s, e))
 * i.e. G_t = r_t + gamma G_{t+1} inside the episode and G_{e-1} = r_{e-1}.
 * The tape's last episode may be cut: if boot is given, G_{L-1} = r_{L-1} +
 * gamma boot[b] (the value of the state after the tape).
 * r, G: [B, L]; start: [B, L] (1 on the first step of an episode); boot: [B] or NULL.
 */
int oracle_discounted_return(int64_t B, int64_t L, const double *r, const uint8_t *start, double gamma,
                             const double *boot, double *G)
{
    if (B < 0 || L < 0) return -1;
    for (int64_t b = 0; b < B; ++b) {
        /* episodes in reverse: e is one past the last step */
        int64_t e = L;
        while (e > 0) {
            int64_t s = e - 1;
            while (s > 0 && !start[b * L + s]) --s;
            double next = (e == L && boot) ? boot[b] : 0.0;
            for (int64_t t = e - 1; t >= s; --t) {
                const double g = r[b * L + t] + gamma * next;
                G[b * L + t] = g;
                next = g;
            }
            e = s;
        }
    }
    return 0;
}

/*
 * GAE per step: A_t = sum_{l = 0}^{e - 1 - t} (gamma lambda)^l delta_{t+l} with
 *     delta_t = r_t + gamma V_{t+1} - V_t,
 * where V_{t+1} is the value of the next step of the same episode, 0 after an
 * episode's last step (the episode ended), and v_boot[b] after the tape's last
 * step when given (the cut episode continues).
 * r, v, A: [B, L]; v_boot: [B] or NULL.
 */
int oracle_gae(int64_t B, int64_t L, const double *r, const double *v, const uint8_t *start, double gamma,
               double lambda, const double *v_boot, double *A)
{
    if (B < 0 || L < 0) return -1;
    for (int64_t b = 0; b < B; ++b) {
        int64_t e = L;
        while (e > 0) {
            int64_t s = e - 1;
            while (s > 0 && !start[b * L + s]) --s;
            double next_v = (e == L && v_boot) ? v_boot[b] : 0.0;
            double next_a = 0.0;
            for (int64_t t = e - 1; t >= s; --t) {
                const double delta = r[b * L + t] + gamma * next_v - v[b * L + t];
                const double a = delta + gamma * lambda * next_a;
                A[b * L + t] = a;
                next_a = a;
                next_v = v[b * L + t];
            }
            e = s;
        }
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Fast and Forgetful Memory as a memoroid (Appendix "Fast and Forgetful     */
/* Memory"):                                                                */
/*   H = {(X, t)}, X complex m x c, t integer;  e_I = (0, 0);               */
/*   (X, t) . (X', t') = (X (.) exp(t' (-|alpha| (+) i omega)) + X', t + t')  */
/*   f(o, b) = (the m-vector x~ repeated over the c columns, 1).             */
/* (+) is the outer sum: entry (i, j) of the exponent is t'(-|alpha_i| +    */
/* i omega_j).  The cell's readout takes Re(X) || Im(X), each flattened     */
/* row-major (i * c + j).  Made resettable by Theorem 3.2 (a begin flag     */
/* replaces the left operand by e_I).                                        */
/* ------------------------------------------------------------------------ */

/* (X, t) . (X', t') for one entry (i, j) of the state */
static void ffm_combine(cplx X, int64_t t, cplx Xp, int64_t tp, double alpha_i, double omega_j,
                        cplx *out, int64_t *t_out)
{
    *out = X * cexp((double)tp * (-fabs(alpha_i) + I * omega_j)) + Xp;
    *t_out = t + tp;
}

/*
 * Forward: the state after every step, by folding the resettable combine
 * from e_I over the lifted steps f(o_t, b_t) = (x~_t repeated, 1).
 * xt: [B, L, m]; start: [B, L]; S0: [B, m*c] complex or NULL (the state
 * before step 0 of a row that continues an episode); z: [B, L, 2*m*c] =
 * Re(X_t) || Im(X_t); S_last: [B, m*c] complex or NULL.
 */
int oracle_ffm_fwd(int64_t B, int64_t L, int64_t m, int64_t c, const double *alpha, const double *omega,
                   const double *xt, const uint8_t *start, const cplx *S0, double *z, cplx *S_last)
{
    if (B < 0 || L < 0 || m < 0 || c < 0) return -1;
    const int64_t D = m * c;
    int bad = 0;
#pragma omp parallel for schedule(static) reduction(| : bad)
    for (int64_t b = 0; b < B; ++b) {
        /* the state (X, t) of every entry, advanced step by step */
        cplx *X = (cplx *)malloc(sizeof(cplx) * (size_t)(D > 0 ? D : 1));
        int64_t *tc = (int64_t *)malloc(sizeof(int64_t) * (size_t)(D > 0 ? D : 1));
        if (!X || !tc) {
            free(X);
            free(tc);
            bad = 1;
            continue;
        }
        for (int64_t ij = 0; ij < D; ++ij) {
            X[ij] = S0 ? S0[b * D + ij] : 0.0; /* e_I unless the row continues an episode */
            tc[ij] = 0;
        }
        for (int64_t t = 0; t < L; ++t) {
            for (int64_t ij = 0; ij < D; ++ij) {
                const int64_t i = ij / c, j = ij % c;
                const cplx Xp = xt[(b * L + t) * m + i];
                if (start[b * L + t]) { /* Theorem 3.2: the left operand becomes e_I = (0, 0) */
                    X[ij] = 0.0;
                    tc[ij] = 0;
                }
                cplx nx;
                int64_t nt;
                ffm_combine(X[ij], tc[ij], Xp, 1, alpha[i], omega[j], &nx, &nt);
                X[ij] = nx;
                tc[ij] = nt;
                z[(b * L + t) * 2 * D + ij] = creal(nx);
                z[(b * L + t) * 2 * D + D + ij] = cimag(nx);
            }
        }
        if (S_last)
            for (int64_t ij = 0; ij < D; ++ij) S_last[b * D + ij] = X[ij];
        free(X);
        free(tc);
    }
    return bad ? -2 : 0;
}

/*
 * Backward (reverse-mode of the forward above).  With lambda_ij =
 * exp(-|alpha_i| + i omega_j) and the upstream G_t = dL/dRe X_t + i dL/dIm X_t
 * (read from grad_z's two halves), the adjoint of X_t is
 *     delta_t = G_t + [b_{t+1} = 0] conj(lambda) delta_{t+1},
 *     delta_{L-1} = G_{L-1} + grad_S_last,
 * and
 *     grad_xt[t, i]  = sum_j Re(delta_t[i, j])          (x~ enters every column)
 *     grad_lambda_ij = sum_{t: b_t = 0} delta_t conj(X_{t-1})  (X_{-1} = S0 or 0)
 *     grad_alpha_i   = sum_j Re(conj(grad_lambda_ij) * (-sign(alpha_i)) lambda_ij)
 *     grad_omega_j   = sum_i Re(conj(grad_lambda_ij) * i lambda_ij)
 *     grad_S0        = [b_0 = 0] conj(lambda) delta_0.
 * z is the forward's output (X_t as Re || Im).  Outputs may be NULL.
 */
int oracle_ffm_bwd(int64_t B, int64_t L, int64_t m, int64_t c, const double *alpha, const double *omega,
                   const uint8_t *start, const cplx *S0, const double *z, const double *grad_z,
                   const cplx *grad_S_last, double *grad_xt, double *grad_alpha, double *grad_omega,
                   cplx *grad_S0)
{
    if (B < 0 || L < 0 || m < 0 || c < 0) return -1;
    const int64_t D = m * c;
    const size_t nD = (size_t)(D > 0 ? D : 1);
    /* per tape: the running grad_lambda sum of every entry (summed over tapes in order below) */
    cplx *glam_b = (cplx *)calloc(nD * (size_t)(B > 0 ? B : 1), sizeof(cplx));
    cplx *glam = (cplx *)calloc(nD, sizeof(cplx));
    cplx *lam = (cplx *)malloc(sizeof(cplx) * nD);
    if (!glam_b || !glam || !lam) {
        free(glam_b);
        free(glam);
        free(lam);
        return -2;
    }
    for (int64_t ij = 0; ij < D; ++ij) lam[ij] = cexp(-fabs(alpha[ij / c]) + I * omega[ij % c]);
    int bad = 0;
#pragma omp parallel for schedule(static) reduction(| : bad)
    for (int64_t b = 0; b < B; ++b) {
        cplx *dn = (cplx *)malloc(sizeof(cplx) * nD); /* delta_{t+1} of every entry */
        if (!dn) {
            bad = 1;
            continue;
        }
        cplx *gl = glam_b + b * D;
        for (int64_t t = L - 1; t >= 0; --t) {
            const double *gz = grad_z + (b * L + t) * 2 * D;
            for (int64_t i = 0; i < m; ++i) {
                double gx = 0.0;
                for (int64_t j = 0; j < c; ++j) {
                    const int64_t ij = i * c + j;
                    cplx d = gz[ij] + I * gz[D + ij];
                    if (t == L - 1) {
                        if (grad_S_last) d += grad_S_last[b * D + ij];
                    } else if (!start[b * L + t + 1]) {
                        d += conj(lam[ij]) * dn[ij];
                    }
                    gx += creal(d);
                    if (!start[b * L + t]) {
                        cplx prev;
                        if (t > 0) {
                            const double *zp = z + (b * L + t - 1) * 2 * D;
                            prev = zp[ij] + I * zp[D + ij];
                        } else {
                            prev = S0 ? S0[b * D + ij] : 0.0;
                        }
                        gl[ij] += d * conj(prev);
                    }
                    dn[ij] = d;
                }
                if (grad_xt) grad_xt[(b * L + t) * m + i] = gx;
            }
        }
        if (grad_S0) {
            for (int64_t ij = 0; ij < D; ++ij)
                grad_S0[b * D + ij] = (L > 0 && !start[b * L]) ? conj(lam[ij]) * dn[ij]
                                                               : (L == 0 && grad_S_last ? grad_S_last[b * D + ij] : 0.0);
        }
        free(dn);
    }
    for (int64_t b = 0; b < B; ++b)
        for (int64_t ij = 0; ij < D; ++ij) glam[ij] += glam_b[b * D + ij];
    free(glam_b);
    if (bad) {
        free(glam);
        free(lam);
        return -2;
    }
    if (grad_alpha) {
        for (int64_t i = 0; i < m; ++i) {
            const double sg = alpha[i] > 0 ? 1.0 : (alpha[i] < 0 ? -1.0 : 0.0);
            double acc = 0.0;
            for (int64_t j = 0; j < c; ++j) acc += creal(conj(glam[i * c + j]) * (-sg) * lam[i * c + j]);
            grad_alpha[i] = acc;
        }
    }
    if (grad_omega) {
        for (int64_t j = 0; j < c; ++j) {
            double acc = 0.0;
            for (int64_t i = 0; i < m; ++i) acc += creal(conj(glam[i * c + j]) * I * lam[i * c + j]);
            grad_omega[j] = acc;
        }
    }
    free(glam);
    free(lam);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Tape-based batching, sampling (Algorithm 2): starting from an empty       */
/* batch, append the episode D[I[i] : I[i+1]] of a randomly drawn index i    */
/* while the batch is shorter than B, then cut the batch to B transitions.  */
/* The draws are an input here: ep[0..K) are the successive indices i, and  */
/* begin[0..E) is the index list I.  The episode of the last index runs to  */
/* the end of D (I[E] reads as N).                                          */
/* ------------------------------------------------------------------------ */

/*
 * Outputs, for the B steps of the batch: src[t] = the index in D of the
 * transition at step t; start[t] = 1 where an appended episode begins.
 * Returns the number of draws used (>= 0), -1 on a bad argument, -2 if an
 * index is out of range, -3 if the K draws do not fill B steps.
 */
int64_t oracle_tbb_sample(const int64_t *begin, int64_t E, int64_t N, const int64_t *ep, int64_t K, int64_t B,
                          uint8_t *start, int64_t *src)
{
    if (E < 0 || N < 0 || K < 0 || B < 0) return -1;
    int64_t len = 0; /* len(batch) */
    int64_t k = 0;
    while (len < B) {
        if (k >= K) return -3;
        const int64_t i = ep[k++];
        if (i < 0 || i >= E) return -2;
        const int64_t lo = begin[i], hi = (i + 1 < E) ? begin[i + 1] : N;
        /* batch <- concat(batch, D[lo:hi]); the cut to B happens on the fly */
        for (int64_t s = lo; s < hi && len < B; ++s) {
            start[len] = (s == lo);
            src[len] = s;
            ++len;
        }
    }
    return k;
}

/* ------------------------------------------------------------------------ */
/* The Linear Transformer memoroid with its feature map and normalizer      */
/* (Appendix "Linear Transformer"):                                         */
/*   (X, x) . (X', x') = (X + X', x + x'),                                   */
/*   f(o, b) = (phi(k) v^T, phi(k)),  g = X^T phi(q) / (x^T phi(q)),         */
/*   phi(z) = 1 + ELU(z) (= 1 + z for z > 0, exp(z) otherwise),              */
/* with the same multiplicative decay gamma_t on the carried pair as the     */
/* decayed memoroid above (gamma = 1 is the paper's model) and the reset of  */
/* Theorem 3.2.  The readout X^T phi(q) follows the reading y = S^T q.      */
/* ------------------------------------------------------------------------ */

static inline double phi1(double z) { return z > 0.0 ? 1.0 + z : exp(z); }
static inline double dphi1(double z) { return z > 0.0 ? 1.0 : exp(z); }

/*
 * q, k: [B,L,H,dk]; v: [B,L,H,dv]; gamma: [H] or [B,L,H]; start: [B,L];
 * S0, S_last: [B,H,dk,dv] or NULL; z0, z_last: [B,H,dk] or NULL (the
 * normalizer state x); y: [B,L,H,dv]; den: [B,L,H] or NULL (x^T phi(q)).
 */
int oracle_linattn_norm_fwd(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, const double *q,
                            const double *k, const double *v, const double *gamma, int gamma_per_step,
                            const uint8_t *start, const double *S0, const double *z0, double *y, double *den,
                            double *S_last, double *z_last)
{
    if (B < 0 || L < 0 || H < 0 || dk <= 0 || dv <= 0) return -1;
    int bad = 0;
#pragma omp parallel for collapse(2) schedule(dynamic) reduction(| : bad)
    for (int64_t b = 0; b < B; ++b) {
        for (int64_t hh = 0; hh < H; ++hh) {
            double *X = (double *)calloc((size_t)(dk * dv), sizeof(double));
            double *x = (double *)calloc((size_t)dk, sizeof(double));
            double *pk = (double *)malloc(sizeof(double) * (size_t)dk);
            double *pq = (double *)malloc(sizeof(double) * (size_t)dk);
            if (!X || !x || !pk || !pq) {
                free(X); free(x); free(pk); free(pq);
                bad = 1;
                continue;
            }
            if (S0) memcpy(X, S0 + (b * H + hh) * dk * dv, sizeof(double) * dk * dv);
            if (z0) memcpy(x, z0 + (b * H + hh) * dk, sizeof(double) * dk);
            for (int64_t t = 0; t < L; ++t) {
                const int64_t r = (b * L + t) * H + hh;
                const int reset = start[b * L + t] != 0;
                const double gt = reset ? 0.0 : gam_at(gamma, gamma_per_step, b, t, L, H, hh);
                for (int64_t i = 0; i < dk; ++i) {
                    pk[i] = phi1(k[r * dk + i]);
                    pq[i] = phi1(q[r * dk + i]);
                }
                /* (X, x) <- gamma (X, x) . f(o_t), or f(o_t) at a begin flag */
                for (int64_t i = 0; i < dk; ++i) {
                    for (int64_t j = 0; j < dv; ++j)
                        X[i * dv + j] = (reset ? 0.0 : gt * X[i * dv + j]) + pk[i] * v[r * dv + j];
                    x[i] = (reset ? 0.0 : gt * x[i]) + pk[i];
                }
                double d = 0.0;
                for (int64_t i = 0; i < dk; ++i) d += x[i] * pq[i];
                for (int64_t j = 0; j < dv; ++j) {
                    double n = 0.0;
                    for (int64_t i = 0; i < dk; ++i) n += X[i * dv + j] * pq[i];
                    y[r * dv + j] = n / d;
                }
                if (den) den[r] = d;
            }
            if (S_last) memcpy(S_last + (b * H + hh) * dk * dv, X, sizeof(double) * dk * dv);
            if (z_last) memcpy(z_last + (b * H + hh) * dk, x, sizeof(double) * dk);
            free(X); free(x); free(pk); free(pq);
        }
    }
    return bad ? -2 : 0;
}

/*
 * Backward of oracle_linattn_norm_fwd (reverse mode).  With n_t = X_t^T phi(q_t),
 * d_t = x_t^T phi(q_t), y_t = n_t / d_t:
 *   dn_t = dy_t / d_t,  dd_t = -(dy_t . y_t) / d_t,
 *   dX_t = phi(q_t) dn_t^T + [b_{t+1} = 0] gamma_{t+1} dX_{t+1}   (+ dS_last at L-1)
 *   dx_t = phi(q_t) dd_t   + [b_{t+1} = 0] gamma_{t+1} dx_{t+1}   (+ dz_last at L-1)
 *   dq_t = (X_t dn_t + x_t dd_t) (.) phi'(q_t),  dk_t = (dX_t v_t + dx_t) (.) phi'(k_t),
 *   dv_t = dX_t^T phi(k_t),  dgamma_t = [b_t = 0] (<dX_t, X_{t-1}> + dx_t . x_{t-1}),
 *   dS0 = [b_0 = 0] gamma_0 dX_0,  dz0 = [b_0 = 0] gamma_0 dx_0.
 * dgamma is [H] (summed over B, L) or [B,L,H].  Any output may be NULL.
 */
int oracle_linattn_norm_bwd(int64_t B, int64_t L, int64_t H, int64_t dk, int64_t dv, const double *q,
                            const double *k, const double *v, const double *gamma, int gamma_per_step,
                            const uint8_t *start, const double *S0, const double *z0, const double *dy,
                            const double *dS_last, const double *dz_last, double *dq, double *dkk, double *dvv,
                            double *dgamma, double *dS0, double *dz0)
{
    if (B < 0 || L < 0 || H < 0 || dk <= 0 || dv <= 0) return -1;
    const int64_t M = dk * dv, W = M + dk; /* one state: X (M values) then x (dk values) */
    double *gsum = (dgamma && !gamma_per_step) ? (double *)calloc((size_t)(B * H > 0 ? B * H : 1), sizeof(double)) : NULL;
    int bad = 0;
#pragma omp parallel for collapse(2) schedule(dynamic) reduction(| : bad)
    for (int64_t b = 0; b < B; ++b) {
        for (int64_t hh = 0; hh < H; ++hh) {
            /* all states of the row: slot t + 1 holds (X_t, x_t), slot 0 the state before step 0 */
            double *St = (double *)calloc((size_t)((L + 1) * W), sizeof(double));
            double *G = (double *)calloc((size_t)W, sizeof(double)); /* (dX, dx) */
            double *pq = (double *)malloc(sizeof(double) * (size_t)dk);
            double *pk = (double *)malloc(sizeof(double) * (size_t)dk);
            double *dn = (double *)malloc(sizeof(double) * (size_t)dv);
            if (!St || !G || !pq || !pk || !dn) {
                free(St); free(G); free(pq); free(pk); free(dn);
                bad = 1;
                continue;
            }
            if (S0) memcpy(St, S0 + (b * H + hh) * M, sizeof(double) * M);
            if (z0) memcpy(St + M, z0 + (b * H + hh) * dk, sizeof(double) * dk);
            for (int64_t t = 0; t < L; ++t) {
                const int64_t r = (b * L + t) * H + hh;
                const int reset = start[b * L + t] != 0;
                const double gt = reset ? 0.0 : gam_at(gamma, gamma_per_step, b, t, L, H, hh);
                const double *P = St + t * W;
                double *C = St + (t + 1) * W;
                for (int64_t i = 0; i < dk; ++i) {
                    const double f = phi1(k[r * dk + i]);
                    for (int64_t j = 0; j < dv; ++j) C[i * dv + j] = (reset ? 0.0 : gt * P[i * dv + j]) + f * v[r * dv + j];
                    C[M + i] = (reset ? 0.0 : gt * P[M + i]) + f;
                }
            }
            double gacc = 0.0;
            for (int64_t t = L - 1; t >= 0; --t) {
                const int64_t r = (b * L + t) * H + hh;
                const double *C = St + (t + 1) * W, *P = St + t * W;
                if (t == L - 1) {
                    for (int64_t w = 0; w < W; ++w) G[w] = 0.0;
                    if (dS_last) memcpy(G, dS_last + (b * H + hh) * M, sizeof(double) * M);
                    if (dz_last) memcpy(G + M, dz_last + (b * H + hh) * dk, sizeof(double) * dk);
                } else {
                    const double gn = start[b * L + t + 1] ? 0.0 : gam_at(gamma, gamma_per_step, b, t + 1, L, H, hh);
                    for (int64_t w = 0; w < W; ++w) G[w] *= gn;
                }
                for (int64_t i = 0; i < dk; ++i) {
                    pq[i] = phi1(q[r * dk + i]);
                    pk[i] = phi1(k[r * dk + i]);
                }
                double d = 0.0;
                for (int64_t i = 0; i < dk; ++i) d += C[M + i] * pq[i];
                double dyy = 0.0;
                for (int64_t j = 0; j < dv; ++j) {
                    double n = 0.0;
                    for (int64_t i = 0; i < dk; ++i) n += C[i * dv + j] * pq[i];
                    dyy += dy[r * dv + j] * (n / d);
                    dn[j] = dy[r * dv + j] / d;
                }
                const double dd = -dyy / d;
                for (int64_t i = 0; i < dk; ++i) {
                    for (int64_t j = 0; j < dv; ++j) G[i * dv + j] += pq[i] * dn[j];
                    G[M + i] += pq[i] * dd;
                }
                for (int64_t i = 0; i < dk; ++i) {
                    double a = C[M + i] * dd, c = G[M + i];
                    for (int64_t j = 0; j < dv; ++j) {
                        a += C[i * dv + j] * dn[j];
                        c += G[i * dv + j] * v[r * dv + j];
                    }
                    if (dq) dq[r * dk + i] = a * dphi1(q[r * dk + i]);
                    if (dkk) dkk[r * dk + i] = c * dphi1(k[r * dk + i]);
                }
                if (dvv) {
                    for (int64_t j = 0; j < dv; ++j) {
                        double a = 0.0;
                        for (int64_t i = 0; i < dk; ++i) a += G[i * dv + j] * pk[i];
                        dvv[r * dv + j] = a;
                    }
                }
                double dg = 0.0;
                if (!start[b * L + t])
                    for (int64_t w = 0; w < W; ++w) dg += G[w] * P[w];
                if (dgamma) {
                    if (gamma_per_step) dgamma[r] = dg;
                    else gacc += dg;
                }
            }
            if (dS0 || dz0) {
                double g0 = (L > 0 && !start[b * L]) ? gam_at(gamma, gamma_per_step, b, 0, L, H, hh) : 0.0;
                if (L == 0) { /* nothing between the states: the gradient passes through */
                    for (int64_t w = 0; w < W; ++w) G[w] = 0.0;
                    if (dS_last) memcpy(G, dS_last + (b * H + hh) * M, sizeof(double) * M);
                    if (dz_last) memcpy(G + M, dz_last + (b * H + hh) * dk, sizeof(double) * dk);
                    g0 = 1.0;
                }
                if (dS0) for (int64_t w = 0; w < M; ++w) dS0[(b * H + hh) * M + w] = g0 * G[w];
                if (dz0) for (int64_t i = 0; i < dk; ++i) dz0[(b * H + hh) * dk + i] = g0 * G[M + i];
            }
            if (gsum) gsum[b * H + hh] = gacc;
            free(St); free(G); free(pq); free(pk); free(dn);
        }
    }
    if (gsum) {
        for (int64_t hh = 0; hh < H; ++hh) {
            double acc = 0.0;
            for (int64_t b = 0; b < B; ++b) acc += gsum[b * H + hh];
            dgamma[hh] = acc;
        }
        free(gsum);
    }
    return bad ? -2 : 0;
}
