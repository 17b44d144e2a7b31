/*
 * DendSN oracle: a plain, slow, single-threaded float64 CPU implementation of
 * the dendritic spiking neuron layer and of its BPTT surrogate-gradient
 * backward.  TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the CPU
 * baseline of the benchmark call it; the product path never does.  It shares no
 * code, header, table or helper with the CUDA library.
 *
 * Every neuron m of the M neurons is simulated on its own, step by step in
 * time order, exactly as the Methods define it:
 *
 *   compartment  V^d_i[t] = alpha_i V^d_i[t-1] + X_i[t],  V^d_i[0] = 0
 *                                   (Eq. methods-compartment)
 *   stateless    V^d_i[t] = X_i[t]  (Methods, "Stateless compartment")
 *   branch       r_b[t] = sqrt( sum_{i in C_b} ((V^d_i[t] - xi_i) / zeta_b)^2 )
 *                Y_b[t] = psi(r_b[t])          (Eq. methods-branch-aggregation)
 *   psi          Mexican hat (1 - x^2) exp(-x^2/2)   (Eq. methods-mexican-hat)
 *                or identity psi(x) = x
 *   soma input   Z[t] = sum_b kappa_b m_b Y_b[t]  (Eq. methods-soma-input, with
 *                the branch-gating mask m of Eq. methods-dbg-mask)
 *   residual     Z[t] += (1/P) sum_i X_i[t]       (Eq. methods-residual)
 *   soma (hard)  V^s[t] = beta (1 - S[t-1]) V^s[t-1] + Z[t]
 *                                   (Eq. methods-lif-reset-charge)
 *   soma (soft)  V^s[t] = beta (V^s[t-1] - theta S[t-1]) + Z[t]
 *                (reading: the soft reset subtracts theta inside the leak, the
 *                 same place where the hard reset multiplies by 1 - S)
 *   fire         S[t] = Theta(V^s[t] - theta), Theta(0) = 1
 *                                   (Eq. methods-lif-fire; theta = 1 there)
 *   surrogate    dS/dV approximated by 1 / (1 + pi^2 (V - theta)^2)
 *                                   (Eq. methods-sg)
 *
 * Branch b owns the G consecutive compartments b*G .. b*G+G-1 (the layer
 * constraint that every branch holds P/B compartments, Methods "Dendritic
 * spiking neural networks"; G = P/B).
 *
 * The backward is the chain rule of the recursion above, applied in reverse
 * time order (BPTT, Eq. methods-sg and the text after it):
 *   dS[t]   = gS[t] + dV^s[t+1]/dS[t] * dV[t+1]        (reset path; 0 if detached)
 *   dV[t]   = gV[t] + sg(V^s[t]-theta) dS[t] + dV^s[t+1]/dV^s[t] * dV[t+1]
 *   dZ[t]   = dV[t]
 *   dY_b    = kappa_b m_b dZ;  dr_b = psi'(r_b) dY_b
 *   du_i    = dr_b u_i / r_b   (0 when r_b = 0);  u_i = (V^d_i - xi_i) / zeta_b
 *   A_i[t]  = du_i[t] / zeta_b + alpha_i A_i[t+1]      (dL/dV^d_i[t])
 *   dX_i[t] = A_i[t] (+ dZ[t] / P with the residual)
 *   dalpha_i += A_i[t] V^d_i[t-1];  dxi_i -= du_i / zeta_b
 *   dzeta_b  -= dr_b r_b / zeta_b;  dkappa_b += m_b Y_b dZ
 *
 * Smooth-spike mode (a test mode): S[t] is replaced everywhere by the
 * surrogate's primitive (1/pi) atan(pi (V^s[t] - theta)) + 1/2, so that the
 * backward above is the exact derivative of the forward and can be checked by
 * finite differences.
 *
 * Build: gcc -O2 -std=c99 -ffp-contract=off -shared -fPIC dendsn_oracle.c -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int32_t T, M, K, G, C;     /* steps, neurons, compartments, per branch, channels */
    int32_t psi;               /* 0 identity, 1 Mexican hat */
    int32_t reset;             /* 0 hard, 1 soft */
    int32_t stateless;         /* 1: V^d = X */
    int32_t residual;          /* 1: Z += mean_i X_i */
    int32_t detach_reset;      /* 1: no gradient through the reset term */
    int32_t smooth_spike;      /* 1: S = surrogate primitive (test mode) */
    double theta, beta;
} oracle_cfg;

static const double ORACLE_PI = 3.14159265358979323846;

/* Eq. methods-mexican-hat, or identity. */
static double psi_value(int psi, double r)
{
    if (psi == 1)
        return (1.0 - r * r) * exp(-0.5 * r * r);
    return r;
}

/* Derivative of psi: d/dx (1 - x^2) e^{-x^2/2} = x (x^2 - 3) e^{-x^2/2}. */
static double psi_deriv(int psi, double r)
{
    if (psi == 1)
        return r * (r * r - 3.0) * exp(-0.5 * r * r);
    return 1.0;
}

/* Eq. methods-sg: derivative of (1/pi) atan(pi x) + 1/2. */
static double surrogate_deriv(double x)
{
    return 1.0 / (1.0 + ORACLE_PI * ORACLE_PI * x * x);
}

static double fire(const oracle_cfg *cfg, double v)
{
    if (cfg->smooth_spike)
        return atan(ORACLE_PI * (v - cfg->theta)) / ORACLE_PI + 0.5;
    return (v - cfg->theta >= 0.0) ? 1.0 : 0.0;  /* Theta(0) = 1 */
}

/*
 * One neuron's forward over all T steps.
 *   x      [T][M][K] (this neuron's column is x[t*M*K + m*K + i])
 *   alpha, xi: this neuron's channel rows (K entries); zeta, kappa: Kb entries
 *   km     kappa_b * m_b (Kb entries)
 * Writes vd_hist[(t+1)*K + i] = V^d_i[t] (row 0 is V^d[0] = 0), vs[t], s[t],
 * r_hist[t*Kb + b], y_hist[t*Kb + b].
 */
static void neuron_forward(const oracle_cfg *cfg, const double *x, int64_t m,
                           const double *alpha, const double *xi, const double *zeta,
                           const double *km, double *vd_hist, double *vs, double *s,
                           double *r_hist, double *y_hist)
{
    const int T = cfg->T, K = cfg->K, G = cfg->G, Kb = cfg->K / cfg->G;
    const int64_t M = cfg->M;
    double v_prev = 0.0, s_prev = 0.0;
    for (int i = 0; i < K; ++i)
        vd_hist[i] = 0.0;
    for (int t = 0; t < T; ++t) {
        const double *xt = x + ((int64_t)t * M + m) * K;
        double *vd_prev = vd_hist + (int64_t)t * K;
        double *vd = vd_hist + (int64_t)(t + 1) * K;
        /* Eq. methods-compartment (or the stateless variant). */
        for (int i = 0; i < K; ++i)
            vd[i] = cfg->stateless ? xt[i] : alpha[i] * vd_prev[i] + xt[i];
        /* Eq. methods-branch-aggregation, Eq. methods-soma-input. */
        double z = 0.0;
        for (int b = 0; b < Kb; ++b) {
            double sq = 0.0;
            for (int i = b * G; i < (b + 1) * G; ++i) {
                double u = (vd[i] - xi[i]) / zeta[b];
                sq += u * u;
            }
            double r = sqrt(sq);
            double y = psi_value(cfg->psi, r);
            r_hist[(int64_t)t * Kb + b] = r;
            y_hist[(int64_t)t * Kb + b] = y;
            z += km[b] * y;
        }
        /* Eq. methods-residual. */
        if (cfg->residual) {
            double mean = 0.0;
            for (int i = 0; i < K; ++i)
                mean += xt[i];
            z += mean / K;
        }
        /* Eq. methods-lif-reset-charge (hard) or the soft-reset reading. */
        double v;
        if (cfg->reset == 0)
            v = cfg->beta * (1.0 - s_prev) * v_prev + z;
        else
            v = cfg->beta * (v_prev - cfg->theta * s_prev) + z;
        double sp = fire(cfg, v);          /* Eq. methods-lif-fire */
        vs[t] = v;
        s[t] = sp;
        v_prev = v;
        s_prev = sp;
    }
}

static void gather_params(const oracle_cfg *cfg, int32_t ch, int32_t mrow,
                          const double *alpha, const double *xi, const double *zeta,
                          const double *kappa, const uint8_t *mask,
                          double *a, double *x_, double *z_, double *km, double *mk)
{
    const int K = cfg->K, Kb = cfg->K / cfg->G;
    for (int i = 0; i < K; ++i) {
        a[i] = cfg->stateless ? 0.0 : alpha[(int64_t)ch * K + i];
        x_[i] = xi[(int64_t)ch * K + i];
    }
    for (int b = 0; b < Kb; ++b) {
        double mb = (mask != NULL && mrow >= 0) ? (double)mask[(int64_t)mrow * Kb + b] : 1.0;
        z_[b] = zeta[(int64_t)ch * Kb + b];
        mk[b] = mb;
        km[b] = kappa[(int64_t)ch * Kb + b] * mb;   /* Eq. methods-dbg-mask */
    }
}

/*
 * Forward of M independent neurons.
 *   x [T][M][K]; chan[m] = parameter channel of neuron m; mrow[m] = row of
 *   `mask` ([rows][Kb], 0/1) used by neuron m, or -1 / mask == NULL for none.
 *   alpha, xi [C][K]; zeta, kappa [C][Kb].
 *   s_out, v_out [T][M] (v_out may be NULL).
 * Returns 0 on success, -1 on bad arguments or allocation failure.
 */
int oracle_forward(const oracle_cfg *cfg, const double *x, const int32_t *chan,
                   const int32_t *mrow, const double *alpha, const double *xi,
                   const double *zeta, const double *kappa, const uint8_t *mask,
                   double *s_out, double *v_out)
{
    if (cfg == NULL || cfg->K <= 0 || cfg->G <= 0 || cfg->K % cfg->G != 0 || cfg->T < 0)
        return -1;
    const int T = cfg->T, K = cfg->K, Kb = cfg->K / cfg->G;
    const int64_t M = cfg->M;
    double *work = (double *)malloc(sizeof(double) *
                                    ((size_t)(T + 1) * K + 2 * (size_t)T + 2 * (size_t)T * Kb +
                                     2 * (size_t)K + 3 * (size_t)Kb));
    if (work == NULL)
        return -1;
    double *vd_hist = work;
    double *vs = vd_hist + (size_t)(T + 1) * K;
    double *s = vs + T;
    double *r_hist = s + T;
    double *y_hist = r_hist + (size_t)T * Kb;
    double *a = y_hist + (size_t)T * Kb;
    double *x_ = a + K;
    double *z_ = x_ + K;
    double *km = z_ + Kb;
    double *mk = km + Kb;
    for (int64_t m = 0; m < M; ++m) {
        gather_params(cfg, chan[m], mrow ? mrow[m] : -1, alpha, xi, zeta, kappa, mask,
                      a, x_, z_, km, mk);
        neuron_forward(cfg, x, m, a, x_, z_, km, vd_hist, vs, s, r_hist, y_hist);
        for (int t = 0; t < T; ++t) {
            s_out[(int64_t)t * M + m] = s[t];
            if (v_out != NULL)
                v_out[(int64_t)t * M + m] = vs[t];
        }
    }
    free(work);
    return 0;
}

/*
 * Backward of M independent neurons (the forward is re-run per neuron).
 *   gs [T][M]: dL/dS; gv [T][M] or NULL: direct dL/dV^s.
 *   gx [T][M][K]: dL/dX (overwritten).
 *   galpha, gxi [C][K], gzeta, gkappa [C][Kb]: summed over every neuron of a
 *   channel and every step (overwritten).
 *   dvs [T][M] or NULL: dL/dV^s[t] (a diagnostic output: the tests derive from it
 *   how strongly fp32 rounding of each branch's direction can show in grad_x).
 *   gbeta [C] or NULL: dL/dbeta of the somatic decay, summed the same way, for a
 *   soma whose beta is learnable (the PLIF soma the paper cites, read as
 *   Eq. methods-lif-reset-charge with beta a parameter):
 *     dV^s[t+1]/dbeta = (1 - S[t]) V^s[t]      (hard reset)
 *                     = V^s[t] - theta S[t]     (soft reset)
 */
int oracle_backward(const oracle_cfg *cfg, const double *x, const int32_t *chan,
                    const int32_t *mrow, const double *alpha, const double *xi,
                    const double *zeta, const double *kappa, const uint8_t *mask,
                    const double *gs, const double *gv, double *gx, double *galpha,
                    double *gxi, double *gzeta, double *gkappa, double *gbeta, double *dvs)
{
    if (cfg == NULL || cfg->K <= 0 || cfg->G <= 0 || cfg->K % cfg->G != 0 || cfg->T < 0)
        return -1;
    const int T = cfg->T, K = cfg->K, G = cfg->G, Kb = cfg->K / cfg->G;
    const int64_t M = cfg->M;
    memset(galpha, 0, sizeof(double) * (size_t)cfg->C * K);
    memset(gxi, 0, sizeof(double) * (size_t)cfg->C * K);
    memset(gzeta, 0, sizeof(double) * (size_t)cfg->C * Kb);
    memset(gkappa, 0, sizeof(double) * (size_t)cfg->C * Kb);
    if (gbeta != NULL)
        memset(gbeta, 0, sizeof(double) * (size_t)cfg->C);
    double *work = (double *)malloc(sizeof(double) *
                                    ((size_t)(T + 1) * K + 2 * (size_t)T + 2 * (size_t)T * Kb +
                                     4 * (size_t)K + 3 * (size_t)Kb));
    if (work == NULL)
        return -1;
    double *vd_hist = work;
    double *vs = vd_hist + (size_t)(T + 1) * K;
    double *s = vs + T;
    double *r_hist = s + T;
    double *y_hist = r_hist + (size_t)T * Kb;
    double *a = y_hist + (size_t)T * Kb;
    double *x_ = a + K;
    double *z_ = x_ + K;
    double *km = z_ + Kb;
    double *mk = km + Kb;
    double *A = mk + Kb;          /* dL/dV^d_i[t+1] carried backwards */
    double *direct = A + K;       /* du_i / zeta_b at the current step */
    for (int64_t m = 0; m < M; ++m) {
        const int32_t ch = chan[m];
        gather_params(cfg, ch, mrow ? mrow[m] : -1, alpha, xi, zeta, kappa, mask,
                      a, x_, z_, km, mk);
        neuron_forward(cfg, x, m, a, x_, z_, km, vd_hist, vs, s, r_hist, y_hist);
        for (int i = 0; i < K; ++i)
            A[i] = 0.0;
        double dv_next = 0.0;     /* dL/dV^s[t+1]; zero past the last step */
        for (int t = T - 1; t >= 0; --t) {
            /* Soma: dS[t] collects the reset path of step t+1. */
            double ds = gs[(int64_t)t * M + m];
            double dvdv_next, dvds_next;
            if (cfg->reset == 0) {
                dvdv_next = cfg->beta * (1.0 - s[t]);   /* dV^s[t+1]/dV^s[t] */
                dvds_next = -cfg->beta * vs[t];          /* dV^s[t+1]/dS[t]   */
            } else {
                dvdv_next = cfg->beta;
                dvds_next = -cfg->beta * cfg->theta;
            }
            if (cfg->detach_reset)
                dvds_next = 0.0;
            if (gbeta != NULL) {
                /* beta's direct effect on V^s[t+1] */
                double leak = (cfg->reset == 0) ? (1.0 - s[t]) * vs[t] : vs[t] - cfg->theta * s[t];
                gbeta[ch] += dv_next * leak;
            }
            ds += dvds_next * dv_next;
            double dv = surrogate_deriv(vs[t] - cfg->theta) * ds + dvdv_next * dv_next;
            if (gv != NULL)
                dv += gv[(int64_t)t * M + m];
            if (dvs != NULL)
                dvs[(int64_t)t * M + m] = dv;
            const double dz = dv;
            /* Branches. */
            const double *vd = vd_hist + (int64_t)(t + 1) * K;
            for (int b = 0; b < Kb; ++b) {
                double r = r_hist[(int64_t)t * Kb + b];
                double y = y_hist[(int64_t)t * Kb + b];
                gkappa[(int64_t)ch * Kb + b] += mk[b] * y * dz;
                double dy = km[b] * dz;
                double dr = psi_deriv(cfg->psi, r) * dy;
                gzeta[(int64_t)ch * Kb + b] -= dr * r / z_[b];
                for (int i = b * G; i < (b + 1) * G; ++i) {
                    double u = (vd[i] - x_[i]) / z_[b];
                    double du = (r > 0.0) ? dr * u / r : 0.0;
                    direct[i] = du / z_[b];
                    gxi[(int64_t)ch * K + i] -= direct[i];
                }
            }
            /* Compartments: reverse leaky scan of Eq. methods-compartment. */
            const double *vd_prev = vd_hist + (int64_t)t * K;
            for (int i = 0; i < K; ++i) {
                A[i] = direct[i] + a[i] * A[i];
                double g = A[i];
                if (cfg->residual)
                    g += dz / K;
                gx[((int64_t)t * M + m) * K + i] = g;
                if (!cfg->stateless)
                    galpha[(int64_t)ch * K + i] += A[i] * vd_prev[i];
            }
            dv_next = dv;
        }
    }
    free(work);
    return 0;
}

/*
 * Point-neuron LIF layer: the soma of the DendSN (Eq. methods-lif-reset-charge,
 * Eq. methods-lif-fire) driven directly by one input current per neuron, i.e. the
 * LIF neuron the paper's point-neuron SNNs use and compares its speed against
 * (Results, "Dendritic spiking neural networks" efficiency paragraph):
 *
 *   hard  V[t] = beta (1 - S[t-1]) V[t-1] + X[t]
 *   soft  V[t] = beta (V[t-1] - theta S[t-1]) + X[t]
 *   fire  S[t] = Theta(V[t] - theta), V[-1] = S[-1] = 0
 *
 * Only T, M, reset, detach_reset, smooth_spike, theta and beta of cfg are read.
 *   x [T][M]; s_out, v_out [T][M] (v_out may be NULL).
 */
int oracle_lif_forward(const oracle_cfg *cfg, const double *x, double *s_out, double *v_out)
{
    if (cfg == NULL || cfg->T < 0 || cfg->M < 0)
        return -1;
    const int T = cfg->T;
    const int64_t M = cfg->M;
    for (int64_t m = 0; m < M; ++m) {
        double v = 0.0, s = 0.0;
        for (int t = 0; t < T; ++t) {
            const double xt = x[(int64_t)t * M + m];
            if (cfg->reset == 0)
                v = cfg->beta * (1.0 - s) * v + xt;
            else
                v = cfg->beta * (v - cfg->theta * s) + xt;
            s = fire(cfg, v);
            s_out[(int64_t)t * M + m] = s;
            if (v_out != NULL)
                v_out[(int64_t)t * M + m] = v;
        }
    }
    return 0;
}

/*
 * BPTT of the LIF layer with the arctan surrogate (Eq. methods-sg): the soma
 * part of the DendSN backward, with dX[t] = dV[t] since X enters V linearly.
 *   gs [T][M]; gv [T][M] or NULL; gx [T][M] (overwritten).
 */
int oracle_lif_backward(const oracle_cfg *cfg, const double *x, const double *gs,
                        const double *gv, double *gx)
{
    if (cfg == NULL || cfg->T < 0 || cfg->M < 0)
        return -1;
    const int T = cfg->T;
    const int64_t M = cfg->M;
    double *vt = (double *)malloc(sizeof(double) * 2 * ((size_t)T + 1));
    if (vt == NULL)
        return -1;
    double *st = vt + T + 1;
    for (int64_t m = 0; m < M; ++m) {
        /* forward, keeping V[t] and S[t] */
        double vv = 0.0, ss = 0.0;
        for (int t = 0; t < T; ++t) {
            const double in = x[(int64_t)t * M + m];
            if (cfg->reset == 0)
                vv = cfg->beta * (1.0 - ss) * vv + in;
            else
                vv = cfg->beta * (vv - cfg->theta * ss) + in;
            ss = fire(cfg, vv);
            vt[t] = vv;
            st[t] = ss;
        }
        /* reverse time: g_next = dL/dV[t+1] */
        double g_next = 0.0;
        for (int t = T - 1; t >= 0; --t) {
            double a_vv, a_vs;                    /* dV[t+1]/dV[t], dV[t+1]/dS[t] */
            if (cfg->reset == 0) {
                a_vv = cfg->beta * (1.0 - st[t]);
                a_vs = -cfg->beta * vt[t];
            } else {
                a_vv = cfg->beta;
                a_vs = -cfg->beta * cfg->theta;
            }
            if (cfg->detach_reset)
                a_vs = 0.0;
            const double g_s = gs[(int64_t)t * M + m] + a_vs * g_next;
            double g_v = surrogate_deriv(vt[t] - cfg->theta) * g_s + a_vv * g_next;
            if (gv != NULL)
                g_v += gv[(int64_t)t * M + m];
            gx[(int64_t)t * M + m] = g_v;         /* V[t] is linear in X[t] */
            g_next = g_v;
        }
    }
    free(vt);
    return 0;
}
