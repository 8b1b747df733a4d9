/*
 * gracekv_oracle.c -- plain CPU oracle of the GraceKV compression pass.
 *
 * TEST INFRASTRUCTURE ONLY (see gracekv_oracle.h): single-threaded fp64,
 * plain loops, each block citing the paper passage it follows.  Nothing in
 * the CUDA library includes or links this file.
 */
#include "gracekv_oracle.h"

#include <float.h>
#include <math.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_EINVAL 1
#define ORC_EBUDGET 2
#define ORC_ENOMEM 3
#define ORC_ECAP 4

static double sqr(double x) { return x * x; }

/* ------------------------------------------------------------------------ */
/* Budget.  App. A.1 Eq. (app_total_budget) gives B_total = floor(L G N_ctx/x)  */
/* (computed by the caller, who knows x); the recent window r = 32 is kept     */
/* and counted in the budget, shortened (minimum 4) only when L G r does not   */
/* fit; B_free = B_total - L G r (Eq. app_free_budget with B_floor = 0).       */
/* ------------------------------------------------------------------------ */
int orc_budget(const orc_params *p, int64_t B_total, int32_t *r_eff, int64_t *B_free)
{
    int64_t LG = (int64_t)p->L * p->G;
    int64_t r = p->recent;
    if (LG * r > B_total) {
        r = B_total / LG;
        if (r < 4) return ORC_EBUDGET;
    }
    int64_t n_ctx = (int64_t)p->ctx_end - p->ctx_start;
    if (n_ctx - r < 1) return ORC_EBUDGET;
    *r_eff = (int32_t)r;
    *B_free = B_total - LG * r;
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* RoPE (reading R11): rotate pair (x_i, x_{i+d/2}) by angle t * theta_i,     */
/* theta_i = base^(-2i/d).  RoPE^-1(x, t) = RoPE(x, -t).  App. A.3             */
/* Eq. (app_rope_prototype) uses both directions.                              */
/* ------------------------------------------------------------------------ */
static void rope(const double *x, double t, int d, double base, double *out)
{
    int half = d / 2;
    if (base == 0.0) {
        for (int i = 0; i < d; i++) out[i] = x[i];
        return;
    }
    for (int i = 0; i < half; i++) {
        double theta = pow(base, -2.0 * (double)i / (double)d);
        double ang = t * theta;
        double c = cos(ang), s = sin(ang);
        double a = x[i], b = x[i + half];
        out[i] = a * c - b * s;
        out[i + half] = a * s + b * c;
    }
}

/* ------------------------------------------------------------------------ */
/* Segmentation layers L_seg = Unique{min(floor(rho L), L-1)}, App. B.2        */
/* Eq. (app_seg_layers); the caller may pass an explicit list instead.         */
/* ------------------------------------------------------------------------ */
static int seg_layers(const orc_params *p, int32_t *out)
{
    if (p->n_seg_layers > 0) {
        for (int i = 0; i < p->n_seg_layers; i++) out[i] = p->seg_layers[i];
        return p->n_seg_layers;
    }
    static const double rho[3] = {0.33, 0.50, 0.67};
    int n = 0;
    for (int k = 0; k < 3; k++) {
        int l = (int)floor(rho[k] * p->L);
        if (l > p->L - 1) l = p->L - 1;
        int dup = 0;
        for (int j = 0; j < n; j++) dup |= (out[j] == l);
        if (!dup) out[n++] = l;
    }
    return n;
}

/* Normalised trajectory hbar^(l)_t, App. B.2 Eq. (app_hidden_normalization).
 * Reading R1: h^(l)_t = concat_g v^(l,g)_t (D = G d) unless hidden states
 * [n_seg, T, Dh] are given.  out: [T][D]. */
static void trajectory(const orc_params *p, const double *V, const double *hidden, int Dh,
                       int li, int l, double *out, int D)
{
    int T = p->T, d = p->d, G = p->G;
    for (int t = 0; t < T; t++) {
        double *h = out + (size_t)t * D;
        if (hidden) {
            for (int c = 0; c < D; c++) h[c] = hidden[((size_t)li * T + t) * Dh + c];
        } else {
            for (int g = 0; g < G; g++)
                for (int c = 0; c < d; c++)
                    h[g * d + c] = V[(((size_t)l * G + g) * T + t) * d + c];
        }
        double nrm = 0.0;
        for (int c = 0; c < D; c++) nrm += h[c] * h[c];
        nrm = sqrt(nrm);
        double den = nrm > 1e-6 ? nrm : 1e-6;
        for (int c = 0; c < D; c++) h[c] /= den;
    }
}

/* ------------------------------------------------------------------------ */
/* Multi-layer, multi-scale curvature, App. B.2:                               */
/*   mu_-, mu_+          Eq. (app_local_means)                                 */
/*   delta_-, delta_+    Eq. (app_local_directions)                            */
/*   u_-, u_+            Eqs. (app_incoming_direction), (app_outgoing_direction)*/
/*   kappa^(l,w)_i       Eq. (app_local_curvature), zero unless w <= i < T-w   */
/*   kappa_i = Mean - lambda_stab PopStd     Eq. (app_stabilized_curvature)    */
/* kappa_lw_out (nullable): [T][n_seg * n_windows], layer-major.               */
/* ------------------------------------------------------------------------ */
int orc_curvature(const orc_params *p, const double *V, const double *hidden, int32_t Dh,
                  double *kappa_out, double *kappa_lw_out)
{
    int32_t layers[8];
    int nl = seg_layers(p, layers);
    int T = p->T;
    int D = hidden ? Dh : p->G * p->d;
    int nw = p->n_windows;
    int nk = nl * nw;
    double *hb = (double *)malloc(sizeof(double) * (size_t)T * D);
    double *kl = (double *)calloc((size_t)T * nk, sizeof(double));
    double *mm = (double *)malloc(sizeof(double) * D);
    double *mp = (double *)malloc(sizeof(double) * D);
    if (!hb || !kl || !mm || !mp) { free(hb); free(kl); free(mm); free(mp); return ORC_ENOMEM; }
    for (int li = 0; li < nl; li++) {
        trajectory(p, V, hidden, Dh, li, layers[li], hb, D);
        for (int wi = 0; wi < nw; wi++) {
            int w = p->windows[wi];
            for (int i = w; i < T - w; i++) {
                for (int c = 0; c < D; c++) { mm[c] = 0.0; mp[c] = 0.0; }
                for (int tau = 0; tau <= w - 1; tau++)
                    for (int c = 0; c < D; c++) mm[c] += hb[(size_t)(i - tau) * D + c];
                for (int tau = 1; tau <= w; tau++)
                    for (int c = 0; c < D; c++) mp[c] += hb[(size_t)(i + tau) * D + c];
                double nm = 0, np_ = 0, dot = 0;
                for (int c = 0; c < D; c++) {
                    double hi = hb[(size_t)i * D + c];
                    double dm = hi - mm[c] / w;       /* delta_- = hbar_i - mu_- */
                    double dp = mp[c] / w - hi;       /* delta_+ = mu_+ - hbar_i */
                    nm += dm * dm;
                    np_ += dp * dp;
                    dot += dm * dp;
                }
                double a = sqrt(nm), b = sqrt(np_);
                double den = (a > 1e-6 ? a : 1e-6) * (b > 1e-6 ? b : 1e-6);
                kl[(size_t)i * nk + li * nw + wi] = 1.0 - dot / den;
            }
        }
    }
    for (int i = 0; i < T; i++) {
        double mean = 0.0;
        for (int k = 0; k < nk; k++) mean += kl[(size_t)i * nk + k];
        mean /= nk;
        double var = 0.0;
        for (int k = 0; k < nk; k++) var += sqr(kl[(size_t)i * nk + k] - mean);
        var /= nk;                                    /* population std */
        kappa_out[i] = mean - p->lambda_stab * sqrt(var);
    }
    if (kappa_lw_out) memcpy(kappa_lw_out, kl, sizeof(double) * (size_t)T * nk);
    free(hb); free(kl); free(mm); free(mp);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Robust z, App. B.2 Eqs. (app_robust_z), (app_mad): (a - median) /          */
/* (1.4826 MAD + 1e-6) over the complete sequence, no clipping.  Reading R4:  */
/* lower median (rank floor((n-1)/2) of the sorted values).                    */
/* ------------------------------------------------------------------------ */
static int cmp_double(const void *x, const void *y)
{
    double a = *(const double *)x, b = *(const double *)y;
    return (a > b) - (a < b);
}

static double lower_median(const double *a, int n, double *scratch)
{
    memcpy(scratch, a, sizeof(double) * n);
    qsort(scratch, n, sizeof(double), cmp_double);
    return scratch[(n - 1) / 2];
}

int orc_robust_z(const double *a, int32_t n, double *z)
{
    double *s = (double *)malloc(sizeof(double) * n);
    double *dev = (double *)malloc(sizeof(double) * n);
    if (!s || !dev) { free(s); free(dev); return ORC_ENOMEM; }
    double med = lower_median(a, n, s);
    for (int i = 0; i < n; i++) dev[i] = fabs(a[i] - med);
    double mad = lower_median(dev, n, s);
    for (int i = 0; i < n; i++) z[i] = (a[i] - med) / (1.4826 * mad + 1e-6);
    free(s); free(dev);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Within-slot dispersion, App. B.3.  Relative coordinates over the           */
/* compressible region [c_s, c_s + N).  d_t = hbar_{c_s+t+1} - hbar_{c_s+t}    */
/* (Eq. app_adjacent_difference).  Mode 0 is the sample-variance definition   */
/* (Eqs. app_mean_difference, app_layer_dispersion); mode 1 is the paper's     */
/* equivalent form Eq. (app_prefix_dispersion), with sum ||d_t||^2 by a prefix */
/* sum and sum d_t = hbar_{e-1} - hbar_a (the differences telescope).          */
/* ------------------------------------------------------------------------ */
typedef struct {
    int nl, D, cs, N;
    double *hb;      /* [nl][T][D] */
    double *pref2;   /* [nl][N]: pref2[t] = sum_{s<t} ||d_s||^2 (mode 1) */
    double *tmp;     /* [D] */
    int T;
    int mode;
} disp_ctx;

static double disp_layer(const disp_ctx *c, int li, int a, int e)
{
    int nS = e - a - 1;
    if (nS < 2) return 0.0;
    int D = c->D;
    const double *hb = c->hb + (size_t)li * c->T * D;
    if (c->mode == 0) {
        double *mean = c->tmp;
        for (int k = 0; k < D; k++) mean[k] = 0.0;
        for (int t = a; t <= e - 2; t++) {
            const double *h1 = hb + (size_t)(c->cs + t + 1) * D, *h0 = hb + (size_t)(c->cs + t) * D;
            for (int k = 0; k < D; k++) mean[k] += h1[k] - h0[k];
        }
        for (int k = 0; k < D; k++) mean[k] /= nS;
        double acc = 0.0;
        for (int t = a; t <= e - 2; t++) {
            const double *h1 = hb + (size_t)(c->cs + t + 1) * D, *h0 = hb + (size_t)(c->cs + t) * D;
            for (int k = 0; k < D; k++) acc += sqr(h1[k] - h0[k] - mean[k]);
        }
        return acc / (nS - 1);
    }
    const double *pr = c->pref2 + (size_t)li * c->N;
    double s2 = pr[e - 1] - pr[a];            /* sum_{t=a}^{e-2} ||d_t||^2 */
    const double *he = hb + (size_t)(c->cs + e - 1) * D, *ha = hb + (size_t)(c->cs + a) * D;
    double sd = 0.0;
    for (int k = 0; k < D; k++) sd += sqr(he[k] - ha[k]);
    return (s2 - sd / nS) / (nS - 1 > 1 ? nS - 1 : 1);
}

static double disp(const disp_ctx *c, int a, int e)
{
    double s = 0.0;
    for (int li = 0; li < c->nl; li++) s += disp_layer(c, li, a, e);
    return s / c->nl;                          /* Eq. (app_slot_dispersion) */
}

/* ------------------------------------------------------------------------ */
/* Curvature-guided segmentation, App. B.2-B.3:                               */
/*   b_i = z(kappa)_i + lambda_s z(surp)_i      Eq. (app_boundary_score)       */
/*   Gamma(a) = b_{c_s+a-1} - c_cut (a > 0)     Eq. (app_boundary_reward)      */
/*   F[i] = max_{a in A(i)} F[a] + Gamma(a) - lambda_d Disp([a,i))             */
/*                           - lambda_n ((i-a-n0)/n0)^2    Eq. (app_dp_recurrence) */
/*   A(i) = {n_min <= i-a <= n_max}             Eq. (app_predecessor_set)      */
/*   terminal relaxation 1 <= N-a <= n_max      Eq. (app_terminal_predecessor) */
/* Reading R5: ties -> first maximum in ascending a; unreachable F = -inf.     */
/* Slot starts are absolute positions; slot_starts[J] = c_s + N.              */
/* dp_best / dp_second (nullable, [N+1]): best and second-best candidate       */
/* values per endpoint (for near-tie classification).                          */
/* ------------------------------------------------------------------------ */
int orc_segment(const orc_params *p, const double *V, const double *hidden, int32_t Dh,
                const double *surprisal, double *kappa_out, double *b_out,
                int32_t *slot_starts, int32_t cap, int32_t *n_slots,
                double *dp_best, double *dp_second)
{
    int T = p->T;
    int cs = p->ctx_start;
    int N = p->ctx_end - p->recent - cs;
    if (N < 1) return ORC_EINVAL;
    int rc = orc_curvature(p, V, hidden, Dh, kappa_out, NULL);
    if (rc) return rc;
    double *zk = (double *)malloc(sizeof(double) * T);
    double *zs = (double *)calloc(T, sizeof(double));
    double *zero = (double *)calloc(T, sizeof(double));
    if (!zk || !zs || !zero) { free(zk); free(zs); free(zero); return ORC_ENOMEM; }
    orc_robust_z(kappa_out, T, zk);
    orc_robust_z(surprisal ? surprisal : zero, T, zs);
    for (int i = 0; i < T; i++) b_out[i] = zk[i] + p->lambda_s * zs[i];
    free(zk); free(zs); free(zero);

    int32_t layers[8];
    int nl = seg_layers(p, layers);
    int D = hidden ? Dh : p->G * p->d;
    disp_ctx c;
    c.nl = nl; c.D = D; c.cs = cs; c.N = N; c.T = T; c.mode = p->disp_mode;
    c.hb = (double *)malloc(sizeof(double) * (size_t)nl * T * D);
    c.pref2 = (double *)calloc((size_t)nl * N, sizeof(double));
    c.tmp = (double *)malloc(sizeof(double) * D);
    double *F = (double *)malloc(sizeof(double) * (N + 1));
    int32_t *P = (int32_t *)malloc(sizeof(int32_t) * (N + 1));
    if (!c.hb || !c.pref2 || !c.tmp || !F || !P) {
        free(c.hb); free(c.pref2); free(c.tmp); free(F); free(P);
        return ORC_ENOMEM;
    }
    for (int li = 0; li < nl; li++) {
        double *hb = c.hb + (size_t)li * T * D;
        trajectory(p, V, hidden, Dh, li, layers[li], hb, D);
        double *pr = c.pref2 + (size_t)li * N;
        pr[0] = 0.0;
        for (int t = 1; t < N; t++) {
            double s = 0.0;
            for (int k = 0; k < D; k++)
                s += sqr(hb[(size_t)(cs + t) * D + k] - hb[(size_t)(cs + t - 1) * D + k]);
            pr[t] = pr[t - 1] + s;
        }
    }
    F[0] = 0.0;
    P[0] = -1;
    for (int i = 1; i <= N; i++) {
        double best = -INFINITY, second = -INFINITY;
        int arg = -1;
        for (int pass = 0; pass < 2 && arg < 0; pass++) {
            /* pass 0: standard predecessor set; pass 1: terminal relaxation (i = N) */
            if (pass == 1 && i != N) break;
            int lo_len = pass == 0 ? p->n_min : 1;
            for (int a = 0; a < i; a++) {
                int len = i - a;
                if (len < lo_len || len > p->n_max) continue;
                if (F[a] == -INFINITY) continue;
                double gamma = a == 0 ? 0.0 : b_out[cs + a - 1] - p->c_cut;
                double v = F[a] + gamma - p->lambda_d * disp(&c, a, i)
                           - p->lambda_n * sqr((double)(len - p->n0) / p->n0);
                if (v > best) { second = best; best = v; arg = a; }
                else if (v > second) second = v;
            }
        }
        F[i] = best;
        P[i] = arg;
        if (dp_best) dp_best[i] = best;
        if (dp_second) dp_second[i] = second;
    }
    /* backtrack (App. B.3: follow P from N) */
    int J = 0;
    for (int i = N; i > 0; i = P[i]) {
        if (P[i] < 0) { J = -1; break; }
        J++;
    }
    int ok = J > 0 && J + 1 <= cap;
    if (ok) {
        int k = J;
        slot_starts[k] = cs + N;
        for (int i = N; i > 0; i = P[i]) slot_starts[--k] = cs + P[i];
        *n_slots = J;
    }
    free(c.hb); free(c.pref2); free(c.tmp); free(F); free(P);
    return ok ? ORC_OK : (J > 0 ? ORC_ECAP : ORC_EINVAL);
}

/* ------------------------------------------------------------------------ */
/* DP edge weights w(a, i) = Gamma(a) - lambda_d Disp([a, i)) - lambda_n      */
/* ((i - a - n0) / n0)^2 of Eq. (app_dp_recurrence), for given pairs of       */
/* region-relative positions 0 <= a < i <= N, with the boundary score b given */
/* (b[cs + a - 1] enters Gamma(a), a > 0).  Same Disp as orc_segment.  Used   */
/* to check the optimality of a partition locally at sizes where the full DP  */
/* is too slow.                                                               */
/* ------------------------------------------------------------------------ */
/* "w/o CS" ablation, App. B.4 (last paragraph): the curvature-guided
 * segmentation is replaced by uniform slots of target length n0 (64) over the
 * compressible context [c_s, c_e - r) (reading R13). */
int orc_uniform_slots(const orc_params *p, int32_t *slot_starts, int32_t cap, int32_t *n_slots)
{
    int cs = p->ctx_start;
    int N = p->ctx_end - p->recent - cs;
    if (N < 1 || p->n0 < 1) return ORC_EINVAL;
    int J = (N + p->n0 / 2) / p->n0;
    if (J < 1) J = 1;
    *n_slots = J;
    if (J > cap) return ORC_ECAP;
    for (int j = 0; j <= J; j++) slot_starts[j] = cs + (int32_t)(((int64_t)j * N) / J);
    return ORC_OK;
}

int orc_dp_weights(const orc_params *p, const double *V, const double *hidden, int32_t Dh,
                   const double *b, int32_t n, const int32_t *a_rel, const int32_t *i_rel,
                   double *w_out)
{
    int T = p->T;
    int cs = p->ctx_start;
    int N = p->ctx_end - p->recent - cs;
    if (N < 1) return ORC_EINVAL;
    for (int k = 0; k < n; k++)
        if (a_rel[k] < 0 || i_rel[k] <= a_rel[k] || i_rel[k] > N) return ORC_EINVAL;
    int32_t layers[8];
    int nl = seg_layers(p, layers);
    int D = hidden ? Dh : p->G * p->d;
    disp_ctx c;
    c.nl = nl; c.D = D; c.cs = cs; c.N = N; c.T = T; c.mode = p->disp_mode;
    c.hb = (double *)malloc(sizeof(double) * (size_t)nl * T * D);
    c.pref2 = (double *)calloc((size_t)nl * N, sizeof(double));
    c.tmp = (double *)malloc(sizeof(double) * D);
    if (!c.hb || !c.pref2 || !c.tmp) {
        free(c.hb); free(c.pref2); free(c.tmp);
        return ORC_ENOMEM;
    }
    for (int li = 0; li < nl; li++) {
        double *hb = c.hb + (size_t)li * T * D;
        trajectory(p, V, hidden, Dh, li, layers[li], hb, D);
        double *pr = c.pref2 + (size_t)li * N;
        pr[0] = 0.0;
        for (int t = 1; t < N; t++) {
            double s = 0.0;
            for (int k = 0; k < D; k++)
                s += sqr(hb[(size_t)(cs + t) * D + k] - hb[(size_t)(cs + t - 1) * D + k]);
            pr[t] = pr[t - 1] + s;
        }
    }
    for (int k = 0; k < n; k++) {
        int a = a_rel[k], i = i_rel[k];
        double gamma = a == 0 ? 0.0 : b[cs + a - 1] - p->c_cut;
        w_out[k] = gamma - p->lambda_d * disp(&c, a, i)
                   - p->lambda_n * sqr((double)(i - a - p->n0) / p->n0);
    }
    free(c.hb); free(c.pref2); free(c.tmp);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Row statistics.  For every probe row (l, h, u) and key t in the visible    */
/* range [0, T) (reading R2): x = q . k_t / sqrt(d); m = max_t x (the          */
/* max-logit shift of App. A.3 "Prototype distortion"); Z = sum exp(x - m)    */
/* (softmax denominator of Eq. app_attention_probability); Z^C = the same sum */
/* restricted to the compressible context C = [c_s, c_e - r).                  */
/* Output layout [L][Hq][W].                                                   */
/* ------------------------------------------------------------------------ */
static double logit(const double *q, const double *k, int d)
{
    double s = 0.0;
    for (int i = 0; i < d; i++) s += q[i] * k[i];
    return s / sqrt((double)d);
}

int orc_row_stats(const orc_params *p, const double *Q, const double *K,
                  double *m, double *Z, double *ZC)
{
    int L = p->L, G = p->G, Hq = p->Hq, W = p->W, T = p->T, d = p->d;
    int gq = Hq / G;
    int c0 = p->ctx_start, c1 = p->ctx_end - p->recent;
    double *x = (double *)malloc(sizeof(double) * T);
    if (!x) return ORC_ENOMEM;
    for (int l = 0; l < L; l++)
        for (int h = 0; h < Hq; h++)
            for (int u = 0; u < W; u++) {
                int g = h / gq;
                const double *q = Q + (((size_t)l * Hq + h) * W + u) * d;
                double mx = -INFINITY;
                for (int t = 0; t < T; t++) {
                    x[t] = logit(q, K + (((size_t)l * G + g) * T + t) * d, d);
                    if (x[t] > mx) mx = x[t];
                }
                double z = 0.0, zc = 0.0;
                for (int t = 0; t < T; t++) {
                    double e = exp(x[t] - mx);
                    z += e;
                    if (t >= c0 && t < c1) zc += e;
                }
                size_t r = ((size_t)l * Hq + h) * W + u;
                m[r] = mx; Z[r] = z; ZC[r] = zc;
            }
    free(x);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Token values, App. A.4:                                                     */
/*   s_{l,g,t} = sum_u sum_{h in H(g)} pi_{u,t}   Eq. (app_direct_relevance)   */
/*   shat = s / (sum_{tau in C} s_tau + eps)                                   */
/*   R_tok = (1 - lambda_graph) shat + lambda_graph dhat, lambda_graph = 0     */
/*   (reading R1)                                 Eq. (app_bottom_up_value)    */
/* Output [L][G][N_c], position c_s + i at index i.                            */
/* ------------------------------------------------------------------------ */
int orc_token_values(const orc_params *p, const double *Q, const double *K,
                     const double *m, const double *Z, double *rtok)
{
    int L = p->L, G = p->G, Hq = p->Hq, W = p->W, T = p->T, d = p->d;
    int gq = Hq / G;
    int c0 = p->ctx_start, Nc = p->ctx_end - p->recent - c0;
    double *s = (double *)malloc(sizeof(double) * Nc);
    if (!s) return ORC_ENOMEM;
    for (int l = 0; l < L; l++)
        for (int g = 0; g < G; g++) {
            for (int i = 0; i < Nc; i++) {
                const double *k = K + (((size_t)l * G + g) * T + c0 + i) * d;
                double acc = 0.0;
                for (int hh = 0; hh < gq; hh++)
                    for (int u = 0; u < W; u++) {
                        int h = g * gq + hh;
                        size_t r = ((size_t)l * Hq + h) * W + u;
                        double xx = logit(Q + r * d, k, d);
                        acc += exp(xx - m[r]) / Z[r];
                    }
                s[i] = acc;
            }
            double tot = 0.0;
            for (int i = 0; i < Nc; i++) tot += s[i];
            for (int i = 0; i < Nc; i++)
                rtok[((size_t)l * G + g) * Nc + i] = s[i] / (tot + p->eps);
        }
    free(s);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Prototype of interval [a, b) of (l, g), App. A.3:                           */
/*   k_circ_t = RoPE^-1(k_t, t); p = round(mean t) (reading R9, half-even);    */
/*   ktil = RoPE(mean k_circ, p)                   Eq. (app_rope_prototype)    */
/*   beta = 0.1 Mean R_tok; w = R_tok + beta;                                  */
/*   vtil = sum w v / (sum w + eps)                Eq. (app_value_prototype)   */
/*   coh = ||mean k_circ|| / (mean ||k_circ|| + eps);                          */
/*   m_eff = clamp(n coh^2, 1, n)                  Eq. (app_effective_multiplicity) */
/* Single-token intervals keep the original K/V, p = t, m = 1 (reading R10).   */
/* ------------------------------------------------------------------------ */
typedef struct {
    int n, pos;
    double meff;
    double *ktil, *vtil;   /* [d] */
} proto_t;

static int round_half_even_mid(int a, int b)
{
    int s = a + b - 1;                       /* 2 * mean position */
    if (s % 2 == 0) return s / 2;
    int lo = (s - 1) / 2, hi = lo + 1;
    return (lo % 2 == 0) ? lo : hi;
}

static void prototype(const orc_params *p, const double *K, const double *V,
                      const double *rtok, int l, int g, int a, int b, proto_t *pr,
                      double *tmp_kc, double *tmp_mu)
{
    int d = p->d, T = p->T, G = p->G;
    int c0 = p->ctx_start, Nc = p->ctx_end - p->recent - c0;
    const double *Kl = K + ((size_t)l * G + g) * T * d;
    const double *Vl = V + ((size_t)l * G + g) * T * d;
    const double *R = rtok + ((size_t)l * G + g) * Nc;
    int n = b - a;
    pr->n = n;
    if (n == 1) {
        for (int i = 0; i < d; i++) { pr->ktil[i] = Kl[(size_t)a * d + i]; pr->vtil[i] = Vl[(size_t)a * d + i]; }
        pr->pos = a;
        pr->meff = 1.0;
        return;
    }
    for (int i = 0; i < d; i++) tmp_mu[i] = 0.0;
    double mean_norm = 0.0;
    for (int t = a; t < b; t++) {
        rope(Kl + (size_t)t * d, -(double)t, d, p->rope_base, tmp_kc);
        double nn = 0.0;
        for (int i = 0; i < d; i++) { tmp_mu[i] += tmp_kc[i]; nn += tmp_kc[i] * tmp_kc[i]; }
        mean_norm += sqrt(nn);
    }
    for (int i = 0; i < d; i++) tmp_mu[i] /= n;
    mean_norm /= n;
    pr->pos = round_half_even_mid(a, b);
    rope(tmp_mu, (double)pr->pos, d, p->rope_base, pr->ktil);
    double mu_norm = 0.0;
    for (int i = 0; i < d; i++) mu_norm += tmp_mu[i] * tmp_mu[i];
    mu_norm = sqrt(mu_norm);
    double coh = mu_norm / (mean_norm + p->eps);
    double me = n * coh * coh;
    pr->meff = me < 1.0 ? 1.0 : (me > n ? (double)n : me);
    double rsum = 0.0;
    for (int t = a; t < b; t++) rsum += R[t - c0];
    double beta = p->base_frac * (rsum / n);
    double wsum = 0.0;
    for (int i = 0; i < d; i++) pr->vtil[i] = 0.0;
    for (int t = a; t < b; t++) {
        double w = R[t - c0] + beta;
        wsum += w;
        for (int i = 0; i < d; i++) pr->vtil[i] += w * Vl[(size_t)t * d + i];
    }
    for (int i = 0; i < d; i++) pr->vtil[i] /= (wsum + p->eps);
}

/* ------------------------------------------------------------------------ */
/* Distortion of interval [a, b), App. A.3:                                    */
/*   Z_q, M_q                        Eq. (app_original_attention_stats)        */
/*   Ztil = m_eff exp(q.ktil/sqrt d), Mtil = Ztil vtil                         */
/*                                   Eq. (app_prototype_attention_stats)       */
/*   D_q = lambda_Z (Z-Ztil)^2/(Z^2+eps) + lambda_M ||M-Mtil||^2/(||M||^2+eps) */
/*                                   Eq. (app_probe_distortion)                */
/*   D = Mean_q [Z_q/Ztot_q D_q], Ddrop = Mean_q Z_q/Ztot_q                    */
/*                                   Eq. (app_node_and_drop_distortion)        */
/* All logits carry the probe's max-logit shift m (App. A.3, text after        */
/* Eq. app_original_attention_stats); Ztot_q is the probe's full partition     */
/* with that shift (reading R7).  Probe u of KV head g uses query head         */
/* H(g)[u mod |H(g)|] (App. A.3, GQA round robin).  D = 0 for one token (R10). */
/* ------------------------------------------------------------------------ */
typedef struct {
    const orc_params *p;
    const double *K, *V, *Q, *m, *Z, *rtok;
    double *kc, *mu, *Mu;      /* scratch [d] each */
    proto_t pr;
} eval_ctx;

static void interval_distortion(eval_ctx *c, int l, int g, int a, int b, double *D, double *Ddrop)
{
    const orc_params *p = c->p;
    int d = p->d, T = p->T, G = p->G, Hq = p->Hq, W = p->W;
    int gq = Hq / G;
    const double *Kl = c->K + ((size_t)l * G + g) * T * d;
    const double *Vl = c->V + ((size_t)l * G + g) * T * d;
    int n = b - a;
    int need_proto = n >= 2;
    if (need_proto) prototype(p, c->K, c->V, c->rtok, l, g, a, b, &c->pr, c->kc, c->mu);
    double Dsum = 0.0, Psum = 0.0;
    for (int u = 0; u < W; u++) {
        int h = g * gq + (u % gq);
        size_t r = ((size_t)l * Hq + h) * W + u;
        const double *q = c->Q + r * d;
        double mr = c->m[r];
        double z = 0.0;
        for (int i = 0; i < d; i++) c->Mu[i] = 0.0;
        for (int t = a; t < b; t++) {
            double e = exp(logit(q, Kl + (size_t)t * d, d) - mr);
            z += e;
            for (int i = 0; i < d; i++) c->Mu[i] += e * Vl[(size_t)t * d + i];
        }
        double pi = z / c->Z[r];
        Psum += pi;
        if (!need_proto) continue;
        double zt = c->pr.meff * exp(logit(q, c->pr.ktil, d) - mr);
        double num = 0.0, den = 0.0;
        for (int i = 0; i < d; i++) {
            num += sqr(c->Mu[i] - zt * c->pr.vtil[i]);
            den += sqr(c->Mu[i]);
        }
        double Dq = p->lambda_Z * sqr(z - zt) / (z * z + p->eps) + p->lambda_M * num / (den + p->eps);
        Dsum += pi * Dq;
    }
    *D = need_proto ? Dsum / W : 0.0;
    *Ddrop = Psum / W;
}

int orc_eval_interval(const orc_params *p, const double *K, const double *V,
                      const double *Q, const double *m, const double *Z,
                      const double *rtok, int32_t l, int32_t g, int32_t a, int32_t b,
                      double *D, double *Ddrop, double *ktil, double *vtil,
                      int32_t *pos, double *logm)
{
    int d = p->d;
    eval_ctx c = {p, K, V, Q, m, Z, rtok, NULL, NULL, NULL, {0}};
    c.kc = (double *)malloc(sizeof(double) * d * 5);
    if (!c.kc) return ORC_ENOMEM;
    c.mu = c.kc + d; c.Mu = c.kc + 2 * d; c.pr.ktil = c.kc + 3 * d; c.pr.vtil = c.kc + 4 * d;
    interval_distortion(&c, l, g, a, b, D, Ddrop);
    prototype(p, K, V, rtok, l, g, a, b, &c.pr, c.kc, c.mu);
    if (ktil) memcpy(ktil, c.pr.ktil, sizeof(double) * d);
    if (vtil) memcpy(vtil, c.pr.vtil, sizeof(double) * d);
    if (pos) *pos = c.pr.pos;
    if (logm) *logm = log(c.pr.meff);
    free(c.kc);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Tree construction, App. A.3 "Recursive refinement rule" and App. B.4:       */
/*   X_v = TopK16(kappa) U {midpoint}            Eq. (app_tree_split_candidates) */
/*   G_bin(xi) = D(I) - D([a,xi)) - D([xi,b)) + lambda_kappa kappahat          */
/*                                               Eq. (app_binary_split)        */
/*   G_ext(p) = D(I) - sum D(children), c_ext = |children| - 1                 */
/*                                               Eq. (app_extract_split)       */
/*   rho_bin = max G_bin, rho_ext = G_ext / c_ext; pick the larger              */
/*                                               Eq. (app_split_choice)        */
/* recursing to single-token leaves (reading R6 fixes candidates and ties).    */
/* Gains, App. A.5 Eq. (app_operation_gains), clamped at 0 (reading R12):      */
/*   Delta_add = omega R(root) (Ddrop - D), Delta_split = omega R(v) (D(v) -   */
/*   sum D(child)); c_add = 1, c_split = |child| - 1; U = Delta / c.           */
/* Node value R(v) = sum R_tok over I_v (Eq. app_bottom_up_value).             */
/* kappa / kscale: bottleneck key of each Split op (min of U along the path    */
/* from the Add) and the magnitude scale of the op that sets it; they are      */
/* outputs for the tests' near-tie classification, not used by the heap.      */
/* ------------------------------------------------------------------------ */
static double rel_gap(double x, double y, double scale)
{
    double s = fmax(fmax(fabs(x), fabs(y)), fabs(scale));
    if (s == 0.0) return 0.0;
    return fabs(x - y) / s;
}

typedef struct { double v; int t; } kv_t;

static int cmp_kv_desc(const void *x, const void *y)
{
    const kv_t *a = (const kv_t *)x, *b = (const kv_t *)y;
    if (a->v > b->v) return -1;
    if (a->v < b->v) return 1;
    return (a->t > b->t) - (a->t < b->t);
}

/* ------------------------------------------------------------------------ */
/* Stage I singleton floor, App. A.5 (Eqs. app_floor_score, app_floor_gate,   */
/* app_floor_cap) and App. C.4 (candidates, path charging, the cap), in the   */
/* reading R15 of the header.                                                  */
/* ------------------------------------------------------------------------ */
static int slot_of(const int32_t *slot_starts, int32_t n_slots, int t)
{
    int lo = 0, hi = n_slots;            /* the last j with slot_starts[j] <= t */
    while (hi - lo > 1) {
        int mid = (lo + hi) / 2;
        if (slot_starts[mid] <= t) lo = mid; else hi = mid;
    }
    return lo;
}

int orc_floor(const orc_params *p, const double *rtok, const int32_t *slot_starts, int32_t n_slots,
              int64_t B_base, double *f, uint8_t *accepted, int64_t *B_floor, int64_t *n_cand)
{
    int LG = p->L * p->G, c0 = p->ctx_start, Nc = p->ctx_end - p->recent - c0;
    int h = p->floor_half;
    memset(accepted, 0, (size_t)LG * Nc);
    *B_floor = 0;
    *n_cand = 0;
    double *Rbar = (double *)calloc((size_t)Nc, sizeof(double));
    double *mix = (double *)malloc(sizeof(double) * (size_t)Nc);
    kv_t *ord = (kv_t *)malloc(sizeof(kv_t) * (size_t)Nc);
    int32_t *cand = (int32_t *)malloc(sizeof(int32_t) * (size_t)LG * Nc);
    int32_t *ncand = (int32_t *)calloc((size_t)LG, sizeof(int32_t));
    uint8_t *inS = (uint8_t *)malloc((size_t)Nc);
    uint8_t *covered = (uint8_t *)malloc((size_t)n_slots);
    if (!Rbar || !mix || !ord || !cand || !ncand || !inS || !covered) {
        free(Rbar); free(mix); free(ord); free(cand); free(ncand); free(inS); free(covered);
        return ORC_ENOMEM;
    }
    /* consensus value and floor score (Eq. app_floor_score) */
    for (int lg = 0; lg < LG; lg++)
        for (int t = 0; t < Nc; t++) Rbar[t] += rtok[(size_t)lg * Nc + t];
    for (int t = 0; t < Nc; t++) Rbar[t] /= LG;
    for (int lg = 0; lg < LG; lg++) {
        const double *R = rtok + (size_t)lg * Nc;
        double *fl = f + (size_t)lg * Nc;
        for (int t = 0; t < Nc; t++) mix[t] = (1.0 - p->floor_c) * R[t] + p->floor_c * Rbar[t];
        for (int t = 0; t < Nc; t++) {
            double mx = -INFINITY;
            for (int u = t - h; u <= t + h; u++)
                if (u >= 0 && u < Nc && mix[u] > mx) mx = mix[u];
            fl[t] = mx;
        }
        /* candidates: f descending, the gate (Eq. app_floor_gate), the value mass eta */
        for (int t = 0; t < Nc; t++) { ord[t].v = fl[t]; ord[t].t = t; }
        qsort(ord, (size_t)Nc, sizeof(kv_t), cmp_kv_desc);
        double cum = 0.0;
        int n = 0;
        for (int k = 0; k < Nc; k++) {
            if (ord[k].v < p->floor_gamma / Nc) break;
            if (cum + R[ord[k].t] > p->floor_eta) break;
            cum += R[ord[k].t];
            cand[(size_t)lg * Nc + n++] = ord[k].t;
        }
        ncand[lg] = n;
        *n_cand += n;
    }
    /* joint cost of all candidates: per slot |S| + maximal runs outside S */
    int64_t C0 = 0;
    for (int lg = 0; lg < LG; lg++) {
        if (!ncand[lg]) continue;
        memset(inS, 0, (size_t)Nc);
        for (int k = 0; k < ncand[lg]; k++) inS[cand[(size_t)lg * Nc + k]] = 1;
        for (int j = 0; j < n_slots; j++) {
            int a = slot_starts[j] - c0, b = slot_starts[j + 1] - c0, k = 0, runs = 0;
            for (int t = a; t < b; t++) {
                k += inS[t];
                if (!inS[t] && (t == a || inS[t - 1])) runs++;
            }
            if (k) C0 += k + runs;
        }
    }
    int64_t cap = (int64_t)floor(p->alpha_floor * (double)B_base);
    int64_t nkept = 0;
    for (int lg = 0; lg < LG; lg++) {
        if (ncand[lg] && C0 > cap) {
            int64_t keep = (int64_t)ncand[lg] * cap / C0;        /* exact integer floor */
            ncand[lg] = (int32_t)(keep < 1 ? 1 : keep);
        }
        nkept += ncand[lg];
    }
    /* acceptance with path charging: every kept candidate, in order, whose
       complete path fits the head's share; one that does not fit is skipped */
    int64_t used = 0;
    for (int lg = 0; lg < LG; lg++) {
        if (!ncand[lg]) continue;
        int64_t cap_h = cap * ncand[lg] / nkept;               /* exact integer floor */
        uint8_t *acc = accepted + (size_t)lg * Nc;
        memset(covered, 0, (size_t)n_slots);
        int64_t used_h = 0;
        for (int k = 0; k < ncand[lg]; k++) {
            int t = cand[(size_t)lg * Nc + k];
            int j = slot_of(slot_starts, n_slots, t + c0);
            int a = slot_starts[j] - c0, b = slot_starts[j + 1] - c0;
            int lo = t, hi = t;                  /* frontier interval [lo, hi] holding t */
            while (lo > a && !acc[lo - 1]) lo--;
            while (hi < b - 1 && !acc[hi + 1]) hi++;
            int64_t cost = (covered[j] ? 0 : 1) + (lo < t) + (t < hi);
            if (used_h + cost > cap_h) continue;
            acc[t] = 1;
            covered[j] = 1;
            used += cost;
            used_h += cost;
        }
    }
    *B_floor = used;
    free(Rbar); free(mix); free(ord); free(cand); free(ncand); free(inS); free(covered);
    return ORC_OK;
}

int orc_build_trees(const orc_params *p, const double *K, const double *V, const double *Q,
                    const double *omega, const double *kappa, const int32_t *slot_starts,
                    int32_t n_slots, const double *m, const double *Z, const double *rtok,
                    const uint8_t *floor_acc, const double *floor_f,
                    orc_nodes *nd, double *unit_Uadd, int64_t *unit_root)
{
    int L = p->L, G = p->G, d = p->d;
    int c0 = p->ctx_start, Nc = p->ctx_end - p->recent - c0;
    eval_ctx c = {p, K, V, Q, m, Z, rtok, NULL, NULL, NULL, {0}};
    c.kc = (double *)malloc(sizeof(double) * d * 5);
    kv_t *kv = (kv_t *)malloc(sizeof(kv_t) * (Nc + 1));
    int *cand = (int *)malloc(sizeof(int) * (Nc + 2));
    if (!c.kc || !kv || !cand) { free(c.kc); free(kv); free(cand); return ORC_ENOMEM; }
    c.mu = c.kc + d; c.Mu = c.kc + 2 * d; c.pr.ktil = c.kc + 3 * d; c.pr.vtil = c.kc + 4 * d;
    int64_t cnt = 0;
    int rc = ORC_OK;
    for (int l = 0; l < L && rc == ORC_OK; l++)
        for (int g = 0; g < G && rc == ORC_OK; g++) {
            int lg = l * G + g;
            const double *R = rtok + (size_t)lg * Nc;
            double om = omega ? omega[lg] : 1.0;
            for (int j = 0; j < n_slots && rc == ORC_OK; j++) {
                int sa = slot_starts[j], sb = slot_starts[j + 1];
                if (cnt + 2 * (sb - sa) > nd->cap) { rc = ORC_ECAP; break; }
                int64_t root = cnt++;
                unit_root[(size_t)lg * n_slots + j] = root;
                double Dr, Ddr;
                interval_distortion(&c, l, g, sa, sb, &Dr, &Ddr);
                double Rr = 0.0;
                for (int t = sa; t < sb; t++) Rr += R[t - c0];
                nd->lg[root] = lg; nd->slot[root] = j; nd->a[root] = sa; nd->b[root] = sb;
                nd->parent[root] = -1; nd->D[root] = Dr; nd->Ddrop[root] = Ddr; nd->R[root] = Rr;
                double dadd = om * Rr * (Ddr - Dr);
                if (dadd < 0.0) dadd = 0.0;
                unit_Uadd[(size_t)lg * n_slots + j] = dadd;
                double add_scale = fabs(om * Rr) * fmax(fabs(Ddr), fabs(Dr));
                /* a slot holding an accepted floor position: its Add is a floor op,
                   executed before the auction (it sets no bound on its children) */
                int unit_fl = 0;
                if (floor_acc)
                    for (int t = sa; t < sb; t++) unit_fl |= floor_acc[(size_t)lg * Nc + (t - c0)];
                /* breadth-first expansion of the unit's tree */
                for (int64_t v = root; v < cnt; v++) {
                    int a = nd->a[v], b = nd->b[v], n = b - a;
                    nd->m_cut[v] = INFINITY; nd->m_form[v] = INFINITY;
                    nd->m_topk[v] = INFINITY; nd->m_ext[v] = INFINITY;
                    nd->floor_op[v] = 0;
                    if (n == 1) {
                        nd->child0[v] = -1; nd->nchild[v] = 0; nd->form[v] = -1; nd->cost[v] = 0;
                        nd->U[v] = 0.0; nd->kappa[v] = 0.0; nd->kscale[v] = 0.0;
                        continue;
                    }
                    double DI = nd->D[v];
                    /* forced extraction at the accepted floor position of largest f */
                    int fp = -1;
                    if (floor_acc) {
                        double fb = -INFINITY;
                        for (int t = a; t < b; t++) {
                            size_t q = (size_t)lg * Nc + (t - c0);
                            if (floor_acc[q] && floor_f[q] > fb) { fb = floor_f[q]; fp = t; }
                        }
                    }
                    double best = -INFINITY, second = -INFINITY;
                    int bxi = -1;
                    double bDL = 0, bDR = 0;
                    if (fp < 0) {
                    /* binary candidates: top-K positions in [a, b-2] by kappa, + midpoint */
                    int np = n - 1;
                    for (int t = a; t <= b - 2; t++) { kv[t - a].v = kappa[t]; kv[t - a].t = t; }
                    qsort(kv, np, sizeof(kv_t), cmp_kv_desc);
                    int K_ = p->k_cand < np ? p->k_cand : np;
                    if (K_ > 0 && np > K_) nd->m_topk[v] = rel_gap(kv[K_ - 1].v, kv[K_].v, 0.0);
                    int nc = 0;
                    for (int k = 0; k < K_; k++) cand[nc++] = kv[k].t + 1;
                    int mid = a + n / 2;
                    int have = 0;
                    for (int k = 0; k < nc; k++) have |= (cand[k] == mid);
                    if (!have) cand[nc++] = mid;
                    /* kappa-hat: min-max of kappa over [a, b-2] */
                    double kmin = INFINITY, kmax = -INFINITY;
                    for (int t = a; t <= b - 2; t++) { kmin = fmin(kmin, kappa[t]); kmax = fmax(kmax, kappa[t]); }
                    /* candidates in ascending xi so that ties keep the smallest xi */
                    for (int x1 = 0; x1 < nc; x1++)
                        for (int x2 = x1 + 1; x2 < nc; x2++)
                            if (cand[x2] < cand[x1]) { int tt = cand[x1]; cand[x1] = cand[x2]; cand[x2] = tt; }
                    for (int k = 0; k < nc; k++) {
                        int xi = cand[k];
                        double DL, DR, dd;
                        interval_distortion(&c, l, g, a, xi, &DL, &dd);
                        interval_distortion(&c, l, g, xi, b, &DR, &dd);
                        double kh = kmax > kmin ? (kappa[xi - 1] - kmin) / (kmax - kmin) : 0.0;
                        double gb = DI - DL - DR + p->lambda_kappa * kh;
                        if (gb > best) { second = best; best = gb; bxi = xi; bDL = DL; bDR = DR; }
                        else if (gb > second) second = gb;
                    }
                    if (nc > 1) nd->m_cut[v] = rel_gap(best, second, DI);
                    }
                    /* salient-token extraction at argmax R_tok (or the floor position) */
                    int ps = a;
                    if (fp >= 0) {
                        ps = fp;
                    } else {
                        double r1 = -INFINITY, r2 = -INFINITY;
                        for (int t = a; t < b; t++) {
                            double r = R[t - c0];
                            if (r > r1) { r2 = r1; r1 = r; ps = t; }
                            else if (r > r2) r2 = r;
                        }
                        nd->m_ext[v] = rel_gap(r1, r2, 0.0);
                    }
                    int ea[3], eb[3], ne = 0;
                    if (ps > a) { ea[ne] = a; eb[ne] = ps; ne++; }
                    ea[ne] = ps; eb[ne] = ps + 1; ne++;
                    if (ps + 1 < b) { ea[ne] = ps + 1; eb[ne] = b; ne++; }
                    double eD[3], gext = DI;
                    for (int k = 0; k < ne; k++) {
                        double dd;
                        interval_distortion(&c, l, g, ea[k], eb[k], &eD[k], &dd);
                        gext -= eD[k];
                    }
                    double rho_ext = gext / (ne - 1);
                    double rho_bin = best;
                    if (fp < 0) nd->m_form[v] = rel_gap(rho_ext, rho_bin, DI);
                    int use_ext = fp >= 0 ? 1 : rho_ext > rho_bin;
                    nd->floor_op[v] = fp >= 0;
                    int ca[3], cb[3], ncl;
                    double cD[3];
                    if (use_ext) {
                        ncl = ne;
                        for (int k = 0; k < ne; k++) { ca[k] = ea[k]; cb[k] = eb[k]; cD[k] = eD[k]; }
                    } else {
                        ncl = 2;
                        ca[0] = a; cb[0] = bxi; cD[0] = bDL;
                        ca[1] = bxi; cb[1] = b; cD[1] = bDR;
                    }
                    nd->form[v] = use_ext;
                    nd->child0[v] = (int32_t)(cnt - root);
                    nd->nchild[v] = ncl;
                    nd->cost[v] = ncl - 1;
                    double dsum = 0.0;
                    for (int k = 0; k < ncl; k++) {
                        int64_t u = cnt++;
                        nd->lg[u] = lg; nd->slot[u] = j; nd->a[u] = ca[k]; nd->b[u] = cb[k];
                        nd->parent[u] = (int32_t)(v - root);
                        nd->D[u] = cD[k]; nd->Ddrop[u] = 0.0;
                        double rr = 0.0;
                        for (int t = ca[k]; t < cb[k]; t++) rr += R[t - c0];
                        nd->R[u] = rr;
                        dsum += cD[k];
                    }
                    double gain = om * nd->R[v] * (DI - dsum);
                    if (gain < 0.0) gain = 0.0;
                    nd->U[v] = gain / (ncl - 1);
                    double own_scale = fabs(om * nd->R[v]) * fmax(fabs(DI), fabs(dsum)) / (ncl - 1);
                    /* bottleneck key: min over the path (creator = parent's split or Add) */
                    double ck, cs_;
                    if (v == root) { ck = unit_fl ? DBL_MAX : dadd; cs_ = add_scale; }
                    else { int64_t pv = root + nd->parent[v]; ck = nd->kappa[pv]; cs_ = nd->kscale[pv]; }
                    if (fp >= 0) { nd->kappa[v] = DBL_MAX; nd->kscale[v] = 0.0; }   /* a floor op */
                    else if (nd->U[v] < ck) { nd->kappa[v] = nd->U[v]; nd->kscale[v] = own_scale; }
                    else { nd->kappa[v] = ck; nd->kscale[v] = cs_; }
                }
                for (int64_t v = root; v < cnt; v++) {
                    if (nd->parent[v] >= 0) nd->parent[v] += (int32_t)root;
                    if (nd->child0[v] >= 0) nd->child0[v] += (int32_t)root;
                }
            }
        }
    nd->count = cnt;
    free(c.kc); free(kv); free(cand);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Greedy allocation, App. A.5 Stage II and App. C.3: one max-priority queue   */
/* keyed by U (Eq. app_unit_utility); seeded with every Add; pop the best;    */
/* an op whose cost exceeds the remaining budget is discarded (its subtree is  */
/* never exposed); executing an op exposes the Split of each non-leaf child;   */
/* stop when the budget is exhausted or the queue is empty.  Heap order:       */
/* U desc, unit (l, g, j) asc, node (a asc, b desc) (reading R12).             */
/* ------------------------------------------------------------------------ */
typedef struct { double U; int64_t unit; int32_t a, b; int64_t node; int is_add; } hitem;

static int hless(const hitem *x, const hitem *y)   /* x has lower priority than y */
{
    if (x->U != y->U) return x->U < y->U;
    if (x->unit != y->unit) return x->unit > y->unit;
    if (x->a != y->a) return x->a > y->a;
    return x->b < y->b;
}

static void hpush(hitem *h, int64_t *n, hitem it)
{
    int64_t i = (*n)++;
    h[i] = it;
    while (i > 0) {
        int64_t pa = (i - 1) / 2;
        if (!hless(&h[pa], &h[i])) break;
        hitem t = h[pa]; h[pa] = h[i]; h[i] = t;
        i = pa;
    }
}

static hitem hpop(hitem *h, int64_t *n)
{
    hitem top = h[0];
    h[0] = h[--(*n)];
    int64_t i = 0;
    for (;;) {
        int64_t l = 2 * i + 1, r = l + 1, b = i;
        if (l < *n && hless(&h[b], &h[l])) b = l;
        if (r < *n && hless(&h[b], &h[r])) b = r;
        if (b == i) break;
        hitem t = h[b]; h[b] = h[i]; h[i] = t;
        i = b;
    }
    return top;
}

int orc_allocate(const orc_params *p, int64_t B_free, int32_t n_slots,
                 const orc_nodes *nd, const double *unit_Uadd, const int64_t *unit_root,
                 const uint8_t *unit_floor, uint8_t *add_sel, uint8_t *split_sel, int64_t *used)
{
    int64_t nu = (int64_t)p->L * p->G * n_slots;
    hitem *h = (hitem *)malloc(sizeof(hitem) * (size_t)(nu + nd->count + 1));
    if (!h) return ORC_ENOMEM;
    int64_t n = 0;
    memset(add_sel, 0, (size_t)nu);
    memset(split_sel, 0, (size_t)nd->count);
    /* remaining capacity: one shared budget, or one per (l, g) (reading R14) */
    int64_t LG = (int64_t)p->L * p->G, nq = p->quota_alloc ? LG : 1;
    int64_t *Rq = (int64_t *)malloc(sizeof(int64_t) * (size_t)nq);
    if (!Rq) { free(h); return ORC_ENOMEM; }
    for (int64_t q = 0; q < nq; q++) Rq[q] = B_free / nq + (q < B_free % nq ? 1 : 0);
    int64_t R = B_free;
    /* the singleton floor's ops execute first (App. A.5 Stage I, reading R15):
       the Add of every floor slot and the forced extractions inside it */
    if (unit_floor)
        for (int64_t u = 0; u < nu; u++) {
            if (!unit_floor[u]) continue;
            int64_t r = unit_root[u], e = u + 1 < nu ? unit_root[u + 1] : nd->count;
            int64_t q = p->quota_alloc ? u / n_slots : 0;
            add_sel[u] = 1;
            Rq[q] -= 1; R -= 1;
            for (int64_t v = r; v < e; v++)
                if (nd->floor_op[v]) { split_sel[v] = 1; Rq[q] -= nd->cost[v]; R -= nd->cost[v]; }
        }
    for (int64_t u = 0; u < nu; u++) {
        int64_t r = unit_root[u];
        if (!add_sel[u]) {
            hitem it = {unit_Uadd[u], u, nd->a[r], nd->b[r], r, 1};
            hpush(h, &n, it);
            continue;
        }
        /* a floor slot: the Split of every frontier node the floor exposed */
        int64_t e = u + 1 < nu ? unit_root[u + 1] : nd->count;
        for (int64_t v = r; v < e; v++) {
            if (split_sel[v] || nd->b[v] - nd->a[v] < 2) continue;
            if (v != r && !split_sel[nd->parent[v]]) continue;
            hitem c = {nd->U[v], u, nd->a[v], nd->b[v], v, 0};
            hpush(h, &n, c);
        }
    }
    while (R > 0 && n > 0) {
        hitem it = hpop(h, &n);
        int64_t v = it.node;
        int cost = it.is_add ? 1 : nd->cost[v];
        int64_t q = p->quota_alloc ? it.unit / n_slots : 0;
        if (cost > Rq[q]) continue;                     /* discard */
        Rq[q] -= cost;
        R -= cost;
        int64_t first, cnt;
        if (it.is_add) {
            add_sel[it.unit] = 1;
            first = v; cnt = 1;                          /* the root joins the frontier */
        } else {
            split_sel[v] = 1;
            first = nd->child0[v]; cnt = nd->nchild[v];
        }
        for (int64_t k = 0; k < cnt; k++) {
            int64_t w = first + k;
            if (nd->b[w] - nd->a[w] < 2) continue;       /* leaves have no Split */
            hitem c = {nd->U[w], it.unit, nd->a[w], nd->b[w], w, 0};
            hpush(h, &n, c);
        }
    }
    if (p->quota_alloc) {                               /* unused capacity is lost */
        R = 0;
        for (int64_t q = 0; q < nq; q++) R += Rq[q] > 0 ? Rq[q] : 0;
    }
    *used = B_free - R;
    free(Rq);
    free(h);
    return ORC_OK;
}

/* ------------------------------------------------------------------------ */
/* Packing, App. A.5 "Frontier updates and physical packing": per (l, g) the  */
/* prefix [0, c_s), the frontier nodes of every covered slot in ascending a   */
/* (non-singletons store ktil, vtil, p, log m_eff; singletons store the       */
/* original K/V, their position and log m = 0), the recent window            */
/* [c_e - r, c_e) and the suffix [c_e, T) as original entries.                 */
/* ------------------------------------------------------------------------ */
static void emit_frontier(const orc_params *p, const double *K, const double *V,
                          const double *rtok, int l, int g, const orc_nodes *nd,
                          const uint8_t *split_sel, int64_t v, int64_t *e, int64_t cap,
                          double *K_out, double *V_out, int32_t *pos, double *log_m,
                          int32_t *src_lo, int32_t *src_hi, proto_t *pr, double *kc, double *mu)
{
    int d = p->d;
    if (nd->b[v] - nd->a[v] >= 2 && split_sel[v]) {
        for (int k = 0; k < nd->nchild[v]; k++)
            emit_frontier(p, K, V, rtok, l, g, nd, split_sel, nd->child0[v] + k, e, cap,
                          K_out, V_out, pos, log_m, src_lo, src_hi, pr, kc, mu);
        return;
    }
    if (*e < cap) {
        prototype(p, K, V, rtok, l, g, nd->a[v], nd->b[v], pr, kc, mu);
        memcpy(K_out + (size_t)(*e) * d, pr->ktil, sizeof(double) * d);
        memcpy(V_out + (size_t)(*e) * d, pr->vtil, sizeof(double) * d);
        pos[*e] = pr->pos;
        log_m[*e] = log(pr->meff);
        src_lo[*e] = nd->a[v];
        src_hi[*e] = nd->b[v];
    }
    (*e)++;
}

static void emit_token(const orc_params *p, const double *K, const double *V, int l, int g, int t,
                       int64_t *e, int64_t cap, double *K_out, double *V_out, int32_t *pos,
                       double *log_m, int32_t *src_lo, int32_t *src_hi)
{
    int d = p->d, T = p->T, G = p->G;
    if (*e < cap) {
        memcpy(K_out + (size_t)(*e) * d, K + (((size_t)l * G + g) * T + t) * d, sizeof(double) * d);
        memcpy(V_out + (size_t)(*e) * d, V + (((size_t)l * G + g) * T + t) * d, sizeof(double) * d);
        pos[*e] = t; log_m[*e] = 0.0; src_lo[*e] = t; src_hi[*e] = t + 1;
    }
    (*e)++;
}

int orc_gather(const orc_params *p, const double *K, const double *V, const double *rtok,
               int32_t n_slots, const orc_nodes *nd, const int64_t *unit_root,
               const uint8_t *add_sel, const uint8_t *split_sel, int64_t cap,
               double *K_out, double *V_out, int32_t *pos, double *log_m,
               int32_t *src_lo, int32_t *src_hi, int64_t *offsets, int64_t *n_entries)
{
    int d = p->d;
    int c_end = p->ctx_end - p->recent;
    double *buf = (double *)malloc(sizeof(double) * d * 4);
    if (!buf) return ORC_ENOMEM;
    proto_t pr;
    pr.ktil = buf; pr.vtil = buf + d;
    int64_t e = 0;
    for (int l = 0; l < p->L; l++)
        for (int g = 0; g < p->G; g++) {
            int lg = l * p->G + g;
            offsets[lg] = e;
            for (int t = 0; t < p->ctx_start; t++)
                emit_token(p, K, V, l, g, t, &e, cap, K_out, V_out, pos, log_m, src_lo, src_hi);
            for (int j = 0; j < n_slots; j++) {
                int64_t u = (int64_t)lg * n_slots + j;
                if (!add_sel[u]) continue;
                emit_frontier(p, K, V, rtok, l, g, nd, split_sel, unit_root[u], &e, cap,
                              K_out, V_out, pos, log_m, src_lo, src_hi, &pr, buf + 2 * d, buf + 3 * d);
            }
            for (int t = c_end; t < p->T; t++)
                emit_token(p, K, V, l, g, t, &e, cap, K_out, V_out, pos, log_m, src_lo, src_hi);
        }
    offsets[p->L * p->G] = e;
    *n_entries = e;
    free(buf);
    return e <= cap ? ORC_OK : ORC_ECAP;
}

/* Decoding on the packed cache, App. A.3 Eq. (app_decode_logit) with the
 * appends of App. A.5 ("Frontier updates and physical packing": a token
 * generated after the compression joins its (l, g) cache with effective
 * multiplicity 1, i.e. log m = 0).  For layer l = l0 + i and query head h of KV
 * head g = h / (Hq / G), the entries of (l, g) are the packed ones
 * [off[lg], off[lg + 1]) followed by the first n_app appended rows; each has
 * the logit  x_e = q . k_e / sqrt(d) + log m_e  and the output is the
 * softmax(x)-weighted sum of the values.  The largest logit is subtracted
 * before exp (the weights are unchanged in exact arithmetic).  An (l, g) with
 * no entry gives a zero output. */
int orc_decode_attention(int32_t L, int32_t G, int32_t Hq, int32_t d, int32_t l0, int32_t nl,
                         const double *q, const double *K, const double *V, const double *log_m,
                         const int64_t *off, const double *K_app, const double *V_app,
                         int32_t app_cap, int32_t n_app, double *out)
{
    if (G <= 0 || Hq % G || d <= 0 || l0 < 0 || nl < 0 || l0 + nl > L || n_app < 0 ||
        n_app > app_cap)
        return ORC_EINVAL;
    int gq = Hq / G;
    int64_t nmax = 0;
    for (int lg = 0; lg < L * G; lg++)
        if (off[lg + 1] - off[lg] > nmax) nmax = off[lg + 1] - off[lg];
    double *x = (double *)malloc(sizeof(double) * (size_t)(nmax + n_app + 1));
    if (!x) return ORC_ENOMEM;
    for (int i = 0; i < nl; i++)
        for (int h = 0; h < Hq; h++) {
            int g = h / gq, lg = (l0 + i) * G + g;
            const double *qh = q + ((size_t)i * Hq + h) * d;
            double *o = out + ((size_t)i * Hq + h) * d;
            int64_t n_pk = off[lg + 1] - off[lg], n = n_pk + n_app;
            for (int c = 0; c < d; c++) o[c] = 0.0;
            if (n == 0) continue;
            double xmax = -DBL_MAX;
            for (int64_t e = 0; e < n; e++) {
                const double *k = e < n_pk ? K + (size_t)(off[lg] + e) * d
                                           : K_app + ((size_t)lg * app_cap + (e - n_pk)) * d;
                double lm = e < n_pk ? log_m[off[lg] + e] : 0.0;
                x[e] = logit(qh, k, d) + lm;       /* logit() divides by sqrt(d) */
                if (x[e] > xmax) xmax = x[e];
            }
            double z = 0.0;
            for (int64_t e = 0; e < n; e++) z += exp(x[e] - xmax);
            for (int64_t e = 0; e < n; e++) {
                const double *v = e < n_pk ? V + (size_t)(off[lg] + e) * d
                                           : V_app + ((size_t)lg * app_cap + (e - n_pk)) * d;
                double w = exp(x[e] - xmax) / z;
                for (int c = 0; c < d; c++) o[c] += w * v[c];
            }
        }
    free(x);
    return ORC_OK;
}

/* Layer-KV-head sensitivity, App. A.4 Eqs. (app_head_sensitivity_raw),
 * (app_head_sensitivity):
 *   static_{l,g} = ( sum_{h in H(g)} ||W_O^{l,h}||_F^2 )^{1/2}
 *   input_{l,g}  = Mean_u || sum_{h in H(g)} W_O^{l,h} o_u^{l,h} ||_2
 *   raw = sqrt(static input),  omega = raw / (Mean_{l,g} raw + eps). */
int orc_head_sensitivity(int32_t L, int32_t G, int32_t Hq, int32_t d, int32_t D, int32_t U,
                         const double *W_O, const double *o, double eps, double *omega)
{
    if (L <= 0 || G <= 0 || Hq % G || d <= 0 || D <= 0 || U <= 0) return ORC_EINVAL;
    int gq = Hq / G;
    size_t row = (size_t)Hq * d;                 /* a row of W_O: all heads' columns */
    double *y = (double *)malloc(sizeof(double) * (size_t)D);
    if (!y) return ORC_ENOMEM;
    double mean = 0.0;
    for (int l = 0; l < L; l++)
        for (int g = 0; g < G; g++) {
            const double *W = W_O + (size_t)l * D * row;
            double st = 0.0;
            for (int r = 0; r < D; r++)
                for (int hh = 0; hh < gq; hh++)
                    for (int i = 0; i < d; i++) {
                        double w = W[(size_t)r * row + (size_t)(g * gq + hh) * d + i];
                        st += w * w;
                    }
            st = sqrt(st);
            double in = 0.0;
            for (int u = 0; u < U; u++) {
                for (int r = 0; r < D; r++) {
                    double acc = 0.0;
                    for (int hh = 0; hh < gq; hh++) {
                        int h = g * gq + hh;
                        const double *ou = o + (((size_t)l * Hq + h) * U + u) * d;
                        for (int i = 0; i < d; i++) acc += W[(size_t)r * row + (size_t)h * d + i] * ou[i];
                    }
                    y[r] = acc;
                }
                double nn = 0.0;
                for (int r = 0; r < D; r++) nn += y[r] * y[r];
                in += sqrt(nn);
            }
            in /= U;
            omega[l * G + g] = sqrt(st * in);
            mean += omega[l * G + g];
        }
    mean /= (double)L * G;
    for (int k = 0; k < L * G; k++) omega[k] /= mean + eps;
    free(y);
    return ORC_OK;
}

/* Graph layers: relative depths 0.50 and 0.75 (reading R16). */
int orc_graph_layers(const orc_params *p, int32_t *out)
{
    static const double rho[2] = {0.50, 0.75};
    int n = 0;
    for (int k = 0; k < 2; k++) {
        int l = (int)floor(rho[k] * p->L);
        if (l > p->L - 1) l = p->L - 1;
        int dup = 0;
        for (int j = 0; j < n; j++) dup |= (out[j] == l);
        if (!dup) out[n++] = l;
    }
    return n;
}

/* Seeds of a hop (reading R16): score sc[Nc] over C, descending (ties lower
 * t), while fewer than m_seed are taken and the running mass is below eta. */
static int pick_seeds(const orc_params *p, const double *sc, int Nc, kv_t *ord, int32_t *sd, double *w)
{
    double tot = 0.0;
    for (int t = 0; t < Nc; t++) { ord[t].v = sc[t]; ord[t].t = t; tot += sc[t]; }
    qsort(ord, (size_t)Nc, sizeof(kv_t), cmp_kv_desc);
    int n = 0;
    double cum = 0.0, ws = 0.0;
    while (n < p->m_seed && n < Nc && cum < p->eta_seed) {
        sd[n] = ord[n].t;
        w[n] = ord[n].v;
        cum += ord[n].v;
        ws += ord[n].v;
        n++;
    }
    for (int k = 0; k < n; k++) w[k] = ws > 0.0 ? w[k] / ws : 1.0 / n;
    (void)tot;
    return n;
}

int orc_multihop(const orc_params *p, const double *shat, const double *Qg, const int32_t *graph_l,
                 int32_t n_graph, const double *K, double *dhat, int32_t *seeds, double *seed_w)
{
    int L = p->L, G = p->G, Hq = p->Hq, T = p->T, d = p->d, gq = Hq / G;
    int c0 = p->ctx_start, Nc = p->ctx_end - p->recent - c0, LG = L * G;
    double *S = (double *)calloc((size_t)Nc, sizeof(double));
    double *sc = (double *)malloc(sizeof(double) * (size_t)Nc);
    double *dk = (double *)malloc(sizeof(double) * (size_t)Nc);
    double *acc = (double *)calloc((size_t)Nc, sizeof(double));
    double *x = (double *)malloc(sizeof(double) * (size_t)T);
    kv_t *ord = (kv_t *)malloc(sizeof(kv_t) * (size_t)Nc);
    int32_t *sd = (int32_t *)malloc(sizeof(int32_t) * (size_t)(p->m_seed + 1));
    double *w = (double *)malloc(sizeof(double) * (size_t)(p->m_seed + 1));
    uint8_t *was = (uint8_t *)calloc((size_t)Nc, 1);
    if (!S || !sc || !dk || !acc || !x || !ord || !sd || !w || !was) {
        free(S); free(sc); free(dk); free(acc); free(x); free(ord); free(sd); free(w); free(was);
        return ORC_ENOMEM;
    }
    if (seeds)
        for (int k = 0; k < p->r_hop * p->m_seed; k++) seeds[k] = -1;
    /* global seed score, Eq. (app_global_seed_score) */
    for (int lg = 0; lg < LG; lg++)
        for (int t = 0; t < Nc; t++) S[t] += shat[(size_t)lg * Nc + t];
    double tot = 0.0;
    for (int t = 0; t < Nc; t++) { S[t] /= LG; tot += S[t]; }
    for (int t = 0; t < Nc; t++) sc[t] = S[t] / (tot + p->eps);
    double decay = 1.0;
    for (int k = 0; k < p->r_hop; k++) {
        int ns = pick_seeds(p, sc, Nc, ord, sd, w);
        if (seeds)
            for (int q = 0; q < ns; q++) { seeds[k * p->m_seed + q] = sd[q] + c0; seed_w[k * p->m_seed + q] = w[q]; }
        for (int q = 0; q < ns; q++) was[sd[q]] = 1;
        /* propagation, Eq. (app_hop_propagation) */
        for (int t = 0; t < Nc; t++) dk[t] = 0.0;
        for (int gi = 0; gi < n_graph; gi++) {
            int l = graph_l[gi];
            for (int h = 0; h < Hq; h++) {
                int g = h / gq;
                const double *Kg = K + (((size_t)l * G + g) * T) * d;
                for (int q = 0; q < ns; q++) {
                    int u = sd[q] + c0;                      /* absolute position of the seed */
                    const double *qu = Qg + (((size_t)gi * Hq + h) * T + u) * d;
                    double mx = -INFINITY;
                    for (int tau = 0; tau <= u; tau++) {     /* visible range [0, u] */
                        x[tau] = logit(qu, Kg + (size_t)tau * d, d);
                        if (x[tau] > mx) mx = x[tau];
                    }
                    double Z = 0.0;
                    for (int tau = 0; tau <= u; tau++) Z += exp(x[tau] - mx);
                    for (int t = c0; t < c0 + Nc && t <= u; t++) dk[t - c0] += w[q] * exp(x[t] - mx) / Z;
                }
            }
        }
        for (int t = 0; t < Nc; t++) if (was[t]) dk[t] = 0.0;
        for (int t = 0; t < Nc; t++) acc[t] += decay * dk[t];
        decay *= p->rho_hop;
        double sk = 0.0;
        for (int t = 0; t < Nc; t++) sk += dk[t];
        for (int t = 0; t < Nc; t++) sc[t] = sk > 0.0 ? dk[t] / sk : 0.0;
    }
    /* Eq. (app_diffused_relevance) */
    double sa = 0.0;
    for (int t = 0; t < Nc; t++) sa += acc[t];
    for (int t = 0; t < Nc; t++) dhat[t] = acc[t] / (sa + p->eps);
    free(S); free(sc); free(dk); free(acc); free(x); free(ord); free(sd); free(w); free(was);
    return ORC_OK;
}
