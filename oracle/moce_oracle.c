/*
 * MoCE layer forward: CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY. This file is a plain, slow, double-precision
 * restatement of the Mixture of Channel Experts layer of "Mixture of Channel
 * Experts: Static Sparse Supports with Input-Adaptive Mixing for Pointwise
 * Projections" (Sec. 3). Only the tests, the smoke check and the benchmark's
 * CPU-baseline leg load it. The CUDA library never calls it and shares no code,
 * header, table or helper with it.
 *
 * Every step follows the paper's definitions in the paper's order, with no
 * blocking, fusion or reordering:
 *   support   Eq. (support), Sec. 3.2      S_e = TopK(L_e, k)
 *   packing   Sec. 3.5 "Storage", Sec. 3.3  keep the k selected (index, logit)
 *             pairs per expert, ordered by descending logit (the gate input is
 *             positional, Sec. 3.3)
 *   pooling   Sec. 3.3                      z = GAP(X)
 *   gate      Eq. (tau), Sec. 3.3; shape from Sec. 4.1 (two-layer MLP, hidden
 *             width k, ReLU, biases)
 *   weights   Eq. (weights)                 a = softmax(L_S / tau)
 *   routed    Eq. (expert)                  Y_e = sum_i a_i X_i
 *   residual  Eq. (res), Sec. 3.4           mean of X over U, 0 if U is empty
 *   coverage  Sec. 3.4                      L_cov over the full routing matrix and
 *             its gradient with respect to every logit (chain rule, written out)
 *   backward  Sec. 3.2 (the task loss differentiates through the selected logit
 *             values; no gradient through the indices): the gradients of a
 *             scalar loss with respect to x, the selected logits and the gate
 *             parameters, given dy, by the chain rule through the steps above
 *   dynamic   Eq. (dynamic), input-conditioned support variant (Sec. 5): the
 *             example's logits L_e(X) = L_e + <q_e (.) h(z), v_c> with the
 *             router bottleneck h(z) = ReLU(W_h z + b_h); the per-example
 *             TopK, U(X), gate and mixing then reuse the functions above with
 *             that example's supports and logits
 *
 * Readings where the paper is silent (each is listed in the design notes):
 *   - ties between equal logits order by ascending channel index; -0.0 and
 *     +0.0 compare equal; non-finite logits are rejected;
 *   - the gate is h = ReLU(W1 u + b1) with W1 stored row-major [hidden][input],
 *     g = w2 . h + b2, sigma is the logistic function;
 *   - the softmax subtracts the largest support logit before exponentiating,
 *     which leaves Eq. (weights) unchanged;
 *   - U is listed in ascending channel order;
 *   - the coverage loss's epsilon is an argument (the paper does not print it);
 *   - the derivative of ReLU at exactly 0 is taken as 0.
 *
 * Inputs are the exact values the device sees (bf16 inputs are decoded to
 * float first); all arithmetic is in double.
 *
 * Layouts: 0 = NHWC (channel fastest), 1 = NCHW (pixel fastest). The output y
 * has R + 1 channels in the same layout, the residual expert last.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_BAD_ARG 1
#define ORACLE_BAD_SUPPORT 2
#define ORACLE_NO_MEMORY 3

static size_t x_at(int layout, int n, int p, int c, int HW, int C)
{
    if (layout == 0)
        return ((size_t)n * HW + p) * (size_t)C + c;
    return ((size_t)n * C + c) * (size_t)HW + p;
}

/* One (channel, logit) pair of an expert's support. */
typedef struct {
    int32_t idx;
    float logit;
} oracle_pair;

/* Deployment order: larger logit first; equal logits by smaller channel. */
static int pair_order(const void *pa, const void *pb)
{
    const oracle_pair *a = (const oracle_pair *)pa;
    const oracle_pair *b = (const oracle_pair *)pb;
    if (a->logit > b->logit)
        return -1;
    if (a->logit < b->logit)
        return 1;
    return (a->idx > b->idx) - (a->idx < b->idx);
}

/*
 * Eq. (support): S_e = TopK(L_e, k) over a full routing row L_e in R^C.
 * L is [R][C]. Writes the k selected channels and their logits per expert,
 * already in deployment order.
 */
int moce_oracle_topk(int C, int R, int k, const float *L, int32_t *idx_out, float *logit_out)
{
    if (C < 1 || R < 1 || k < 1 || k > C || !L || !idx_out || !logit_out)
        return ORACLE_BAD_ARG;
    oracle_pair *row = (oracle_pair *)malloc(sizeof(oracle_pair) * (size_t)C);
    if (!row)
        return ORACLE_NO_MEMORY;
    for (int e = 0; e < R; ++e) {
        for (int c = 0; c < C; ++c) {
            float v = L[(size_t)e * C + c];
            if (!isfinite(v)) {
                free(row);
                return ORACLE_BAD_SUPPORT;
            }
            row[c].idx = c;
            row[c].logit = v;
        }
        qsort(row, (size_t)C, sizeof(oracle_pair), pair_order);
        for (int i = 0; i < k; ++i) {
            idx_out[(size_t)e * k + i] = row[i].idx;
            logit_out[(size_t)e * k + i] = row[i].logit;
        }
    }
    free(row);
    return ORACLE_OK;
}

/*
 * Deployment packing (Sec. 3.5 "Storage"; order rule of Sec. 3.3; U of
 * Sec. 3.4). support_idx / support_logits are [R][k] in any row order.
 * Outputs: each row sorted into deployment order, the unselected channels U
 * in ascending order (resid, capacity C) and |U|.
 * A support index outside [0, C), a repeated index within one expert, or a
 * non-finite logit is rejected.
 */
int moce_oracle_pack(int C, int R, int k, const int32_t *support_idx, const float *support_logits,
                     int32_t *packed_idx, float *packed_logits, int32_t *resid, int32_t *n_resid)
{
    if (C < 1 || R < 1 || k < 1 || k > C || !support_idx || !support_logits || !packed_idx ||
        !packed_logits || !resid || !n_resid)
        return ORACLE_BAD_ARG;
    unsigned char *covered = (unsigned char *)calloc((size_t)C, 1);
    int *seen_in_row = (int *)malloc(sizeof(int) * (size_t)C);
    oracle_pair *row = (oracle_pair *)malloc(sizeof(oracle_pair) * (size_t)k);
    if (!covered || !seen_in_row || !row) {
        free(covered);
        free(seen_in_row);
        free(row);
        return ORACLE_NO_MEMORY;
    }
    for (int c = 0; c < C; ++c)
        seen_in_row[c] = -1;
    int status = ORACLE_OK;
    for (int e = 0; e < R && status == ORACLE_OK; ++e) {
        for (int i = 0; i < k; ++i) {
            int32_t c = support_idx[(size_t)e * k + i];
            float v = support_logits[(size_t)e * k + i];
            if (c < 0 || c >= C || !isfinite(v) || seen_in_row[c] == e) {
                status = ORACLE_BAD_SUPPORT;
                break;
            }
            seen_in_row[c] = e;
            row[i].idx = c;
            row[i].logit = v;
        }
        if (status != ORACLE_OK)
            break;
        qsort(row, (size_t)k, sizeof(oracle_pair), pair_order);
        for (int i = 0; i < k; ++i) {
            packed_idx[(size_t)e * k + i] = row[i].idx;
            packed_logits[(size_t)e * k + i] = row[i].logit;
            covered[row[i].idx] = 1;
        }
    }
    if (status == ORACLE_OK) {
        int m = 0;
        for (int c = 0; c < C; ++c)
            if (!covered[c])
                resid[m++] = c;
        *n_resid = m;
    }
    free(covered);
    free(seen_in_row);
    free(row);
    return status;
}

/* Sec. 3.3: z = GAP(X), the mean over the H*W positions of each (n, c). */
void moce_oracle_pool(const float *x, int N, int H, int W, int C, int layout, double *z)
{
    int HW = H * W;
    for (int n = 0; n < N; ++n)
        for (int c = 0; c < C; ++c) {
            double s = 0.0;
            for (int p = 0; p < HW; ++p)
                s += (double)x[x_at(layout, n, p, c, HW, C)];
            z[(size_t)n * C + c] = s / (double)HW;
        }
}

/*
 * Eq. (tau): tau_e = tau_min + (tau_max - tau_min) * sigma(g(z_{S_e})).
 * The gate input u is z at the expert's support in deployment order, so u_0
 * is the descriptor of the expert's most preferred channel (Sec. 3.3).
 * g(u) = w2 . ReLU(W1 u + b1) + b2, W1 is [k][k] with row j = hidden unit j.
 * g_out (optional) receives the pre-sigmoid gate value, [N][R].
 */
void moce_oracle_gate(const double *z, int N, int C, int R, int k, const int32_t *packed_idx,
                      const float *W1, const float *b1, const float *w2, float b2,
                      double tau_min, double tau_max, double *g_out, double *tau)
{
    double *u = (double *)malloc(sizeof(double) * (size_t)k);
    double *h = (double *)malloc(sizeof(double) * (size_t)k);
    for (int n = 0; n < N; ++n)
        for (int e = 0; e < R; ++e) {
            for (int i = 0; i < k; ++i)
                u[i] = z[(size_t)n * C + packed_idx[(size_t)e * k + i]];
            for (int j = 0; j < k; ++j) {
                double s = (double)b1[j];
                for (int i = 0; i < k; ++i)
                    s += (double)W1[(size_t)j * k + i] * u[i];
                h[j] = s > 0.0 ? s : 0.0;
            }
            double g = (double)b2;
            for (int j = 0; j < k; ++j)
                g += (double)w2[j] * h[j];
            double sig = 1.0 / (1.0 + exp(-g));
            if (g_out)
                g_out[(size_t)n * R + e] = g;
            tau[(size_t)n * R + e] = tau_min + (tau_max - tau_min) * sig;
        }
    free(u);
    free(h);
}

/*
 * Eq. (weights): a_{e,i} = exp(L_{e,i}/tau_e) / sum_j exp(L_{e,j}/tau_e),
 * evaluated as exp((L_{e,i} - max_j L_{e,j}) / tau_e) / sum (same value).
 * tau is [N][R], packed_logits [R][k], a is [N][R][k].
 */
void moce_oracle_weights(const double *tau, int N, int R, int k, const float *packed_logits,
                         double *a)
{
    for (int n = 0; n < N; ++n)
        for (int e = 0; e < R; ++e) {
            const float *L = packed_logits + (size_t)e * k;
            double t = tau[(size_t)n * R + e];
            double m = (double)L[0];
            for (int i = 1; i < k; ++i)
                if ((double)L[i] > m)
                    m = (double)L[i];
            double *ae = a + ((size_t)n * R + e) * k;
            double s = 0.0;
            for (int i = 0; i < k; ++i) {
                ae[i] = exp(((double)L[i] - m) / t);
                s += ae[i];
            }
            for (int i = 0; i < k; ++i)
                ae[i] /= s;
        }
}

/*
 * Eq. (expert) and Eq. (res): at every position,
 *   y_e = sum_i a_{e,i} x_{S_e[i]}               for e < R,
 *   y_R = |U|^-1 sum_{c in U} x_c, or 0 if U is empty.
 * a is [N][R][k]; y has R + 1 channels in the layout of x.
 */
void moce_oracle_mix(const float *x, int N, int H, int W, int C, int layout, int R, int k,
                     const int32_t *packed_idx, const double *a, const int32_t *resid,
                     int n_resid, double *y)
{
    int HW = H * W;
    int E = R + 1;
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < HW; ++p) {
            for (int e = 0; e < R; ++e) {
                const double *ae = a + ((size_t)n * R + e) * k;
                double s = 0.0;
                for (int i = 0; i < k; ++i)
                    s += ae[i] * (double)x[x_at(layout, n, p, packed_idx[(size_t)e * k + i], HW, C)];
                y[x_at(layout, n, p, e, HW, E)] = s;
            }
            double r = 0.0;
            if (n_resid > 0) {
                for (int j = 0; j < n_resid; ++j)
                    r += (double)x[x_at(layout, n, p, resid[j], HW, C)];
                r /= (double)n_resid;
            }
            y[x_at(layout, n, p, R, HW, E)] = r;
        }
}

/*
 * The whole layer: pool -> gate -> weights -> routed + residual outputs.
 * Supports must already be packed. z_out [N][C], tau_out [N][R] and
 * a_out [N][R][k] are optional copies of the intermediates.
 */
int moce_oracle_forward(const float *x, int N, int H, int W, int C, int layout, int R, int k,
                        const int32_t *packed_idx, const float *packed_logits,
                        const int32_t *resid, int n_resid, const float *W1, const float *b1,
                        const float *w2, float b2, double tau_min, double tau_max, double *y,
                        double *z_out, double *tau_out, double *a_out)
{
    if (N < 0 || H < 0 || W < 0 || C < 1 || R < 1 || k < 1 || k > C || n_resid < 0 ||
        n_resid > C || (layout != 0 && layout != 1))
        return ORACLE_BAD_ARG;
    double *z = z_out ? z_out : (double *)malloc(sizeof(double) * ((size_t)N * C + 1));
    double *tau = tau_out ? tau_out : (double *)malloc(sizeof(double) * ((size_t)N * R + 1));
    double *a = a_out ? a_out : (double *)malloc(sizeof(double) * ((size_t)N * R * k + 1));
    int status = ORACLE_OK;
    if (!z || !tau || !a) {
        status = ORACLE_NO_MEMORY;
    } else {
        moce_oracle_pool(x, N, H, W, C, layout, z);
        moce_oracle_gate(z, N, C, R, k, packed_idx, W1, b1, w2, b2, tau_min, tau_max, NULL, tau);
        moce_oracle_weights(tau, N, R, k, packed_logits, a);
        moce_oracle_mix(x, N, H, W, C, layout, R, k, packed_idx, a, resid, n_resid, y);
    }
    if (!z_out)
        free(z);
    if (!tau_out)
        free(tau);
    if (!a_out)
        free(a);
    return status;
}

/*
 * Brute-force restatement used to pin the oracle above on tiny shapes. It
 * starts from the full routing matrix L [R][C] (the training-time form,
 * Sec. 3.2) and shares no step with the functions above:
 *   - S_e by k rounds of "take the largest remaining logit" (ties: smallest
 *     channel), not by sorting;
 *   - U by counting, over all experts, how often each channel is selected;
 *   - weights as exp(L/tau) / sum exp(L/tau) with no max subtraction;
 *   - the layer as a dense matrix W_eff [R+1][C] per example, applied to the
 *     channel vector of every position with a plain triple loop.
 * Used only with small logits, where exp(L/tau) cannot overflow.
 */
int moce_oracle_bruteforce_forward(const float *x, int N, int H, int W, int C, int layout, int R,
                                   int k, const float *L, const float *W1, const float *b1,
                                   const float *w2, float b2, double tau_min, double tau_max,
                                   double *y)
{
    if (N < 0 || H < 0 || W < 0 || C < 1 || R < 1 || k < 1 || k > C || (layout != 0 && layout != 1))
        return ORACLE_BAD_ARG;
    int HW = H * W;
    int E = R + 1;
    int *sel = (int *)malloc(sizeof(int) * (size_t)R * k);
    int *count = (int *)calloc((size_t)C, sizeof(int));
    unsigned char *taken = (unsigned char *)malloc((size_t)C);
    double *Weff = (double *)malloc(sizeof(double) * (size_t)E * C);
    double *zn = (double *)malloc(sizeof(double) * (size_t)C);
    double *hid = (double *)malloc(sizeof(double) * (size_t)k);
    if (!sel || !count || !taken || !Weff || !zn || !hid) {
        free(sel); free(count); free(taken); free(Weff); free(zn); free(hid);
        return ORACLE_NO_MEMORY;
    }
    for (int e = 0; e < R; ++e) {
        memset(taken, 0, (size_t)C);
        for (int r = 0; r < k; ++r) {
            int best = -1;
            for (int c = 0; c < C; ++c) {
                if (taken[c])
                    continue;
                if (best < 0 || L[(size_t)e * C + c] > L[(size_t)e * C + best])
                    best = c;
            }
            taken[best] = 1;
            sel[(size_t)e * k + r] = best;
            count[best] += 1;
        }
    }
    int nU = 0;
    for (int c = 0; c < C; ++c)
        nU += (count[c] == 0);
    for (int n = 0; n < N; ++n) {
        for (int c = 0; c < C; ++c) {
            double s = 0.0;
            for (int p = 0; p < HW; ++p)
                s += (double)x[x_at(layout, n, p, c, HW, C)];
            zn[c] = s / (double)HW;
        }
        for (size_t q = 0; q < (size_t)E * C; ++q)
            Weff[q] = 0.0;
        for (int e = 0; e < R; ++e) {
            /* gate: input position r is the r-th selected (r-th largest) channel */
            double g = (double)b2;
            for (int j = 0; j < k; ++j) {
                double s = (double)b1[j];
                for (int r = 0; r < k; ++r)
                    s += (double)W1[(size_t)j * k + r] * zn[sel[(size_t)e * k + r]];
                if (s > 0.0)
                    g += (double)w2[j] * s;
            }
            double t = tau_min + (tau_max - tau_min) / (1.0 + exp(-g));
            double den = 0.0;
            for (int r = 0; r < k; ++r)
                den += exp((double)L[(size_t)e * C + sel[(size_t)e * k + r]] / t);
            for (int r = 0; r < k; ++r) {
                int c = sel[(size_t)e * k + r];
                Weff[(size_t)e * C + c] += exp((double)L[(size_t)e * C + c] / t) / den;
            }
        }
        if (nU > 0)
            for (int c = 0; c < C; ++c)
                if (count[c] == 0)
                    Weff[(size_t)R * C + c] = 1.0 / (double)nU;
        for (int p = 0; p < HW; ++p)
            for (int o = 0; o < E; ++o) {
                double s = 0.0;
                for (int c = 0; c < C; ++c)
                    s += Weff[(size_t)o * C + c] * (double)x[x_at(layout, n, p, c, HW, C)];
                y[x_at(layout, n, p, o, HW, E)] = s;
            }
    }
    free(sel); free(count); free(taken); free(Weff); free(zn); free(hid);
    return ORACLE_OK;
}

/*
 * Coverage regularizer, Sec. 3.4: p_{e,c} = softmax(L_e)_c over all C
 * channels of a full routing row, u_c = (1/R) sum_e p_{e,c},
 * ubar = (1/C) sum_c u_c, L_cov = sum_c (u_c - ubar)^2 / (ubar^2 + eps).
 * L is [R][C]. Writes the loss; u [C] and the gradient dL_cov/dL [R][C] when
 * the pointers are not NULL. The softmax subtracts the row maximum first.
 * The gradient is the chain rule of the same definitions:
 *   dL/du_c = 2 (u_c - ubar) / D - (2 / C) sum_c' (u_c' - ubar) / D
 *             - 2 ubar S / (C D^2),     D = ubar^2 + eps, S = sum_c (u_c - ubar)^2
 *   dL/dL_{e,c} = (1/R) p_{e,c} (dL/du_c - sum_c' p_{e,c'} dL/du_c').
 */
int moce_oracle_coverage(int C, int R, const float *L, double eps, double *loss, double *u_out,
                         double *grad)
{
    if (C < 1 || R < 1 || !L || !loss || !(eps >= 0.0))
        return ORACLE_BAD_ARG;
    double *p = (double *)malloc(sizeof(double) * (size_t)R * C);
    double *u = (double *)malloc(sizeof(double) * (size_t)C);
    double *g = (double *)malloc(sizeof(double) * (size_t)C);
    if (!p || !u || !g) {
        free(p);
        free(u);
        free(g);
        return ORACLE_NO_MEMORY;
    }
    for (int e = 0; e < R; ++e) {
        const float *Le = L + (size_t)e * C;
        double m = -INFINITY;
        for (int c = 0; c < C; ++c) {
            if (!isfinite(Le[c])) {
                free(p);
                free(u);
                free(g);
                return ORACLE_BAD_SUPPORT;
            }
            if ((double)Le[c] > m)
                m = (double)Le[c];
        }
        double sum = 0.0;
        for (int c = 0; c < C; ++c)
            sum += exp((double)Le[c] - m);
        for (int c = 0; c < C; ++c)
            p[(size_t)e * C + c] = exp((double)Le[c] - m) / sum;
    }
    for (int c = 0; c < C; ++c) {
        double s = 0.0;
        for (int e = 0; e < R; ++e)
            s += p[(size_t)e * C + c];
        u[c] = s / (double)R;
    }
    double ubar = 0.0;
    for (int c = 0; c < C; ++c)
        ubar += u[c];
    ubar /= (double)C;
    const double D = ubar * ubar + eps;
    double S = 0.0, dev = 0.0;
    for (int c = 0; c < C; ++c) {
        S += (u[c] - ubar) * (u[c] - ubar);
        dev += u[c] - ubar;
    }
    *loss = S / D;
    if (u_out)
        for (int c = 0; c < C; ++c)
            u_out[c] = u[c];
    if (grad) {
        for (int c = 0; c < C; ++c)
            g[c] = 2.0 * (u[c] - ubar) / D - 2.0 * dev / ((double)C * D) -
                   2.0 * ubar * S / ((double)C * D * D);
        for (int e = 0; e < R; ++e) {
            double dot = 0.0;
            for (int c = 0; c < C; ++c)
                dot += p[(size_t)e * C + c] * g[c];
            for (int c = 0; c < C; ++c)
                grad[(size_t)e * C + c] = p[(size_t)e * C + c] * (g[c] - dot) / (double)R;
        }
    }
    free(p);
    free(u);
    free(g);
    return ORACLE_OK;
}

/*
 * Backward of the layer with static supports (Sec. 3.2: gradients reach the
 * selected logit values, never the indices). Given dy = dJ/dy (the layout and
 * shape of y) for a scalar J, returns by the chain rule through pool, gate,
 * weights, routed mix and residual, per example n:
 *   da_{e,i}  = sum_p dy_{p,e} x_{p,S_e[i]}                          Eq. (expert)
 *   ds_{e,i}  = a_{e,i} (da_{e,i} - sum_j a_{e,j} da_{e,j}),  s = L / tau   Eq. (weights)
 *   dL_{e,i} += ds_{e,i} / tau_e;  dtau_e = -sum_i ds_{e,i} L_{e,i} / tau_e^2
 *   dg_e      = dtau_e (tau_max - tau_min) sigma_e (1 - sigma_e)       Eq. (tau)
 *   dw2_j    += dg_e r_{e,j};  db2 += dg_e;  dh_{e,j} = dg_e w2_j [h_{e,j} > 0]
 *   dW1_{j,i}+= dh_{e,j} u_{e,i};  db1_j += dh_{e,j};  du_{e,i} = sum_j W1_{j,i} dh_{e,j}
 *   dz_c      = sum over (e, i) with S_e[i] = c of du_{e,i}            (u = z[S_e])
 *   dx_{p,c}  = sum over (e, i) with S_e[i] = c of a_{e,i} dy_{p,e}
 *               + [c in U] dy_{p,R} / |U| + dz_c / HW                 Eq. (res), GAP
 * dx has the layout of x; dlogit [R][k] (packed order), dW1 [k][k] (row j =
 * hidden unit j), db1 [k], dw2 [k], db2 [1] are sums over the batch.
 */
int moce_oracle_backward(const float *x, const float *dy, int N, int H, int W, int C, int layout,
                         int R, int k, const int32_t *packed_idx, const float *packed_logits,
                         const int32_t *resid, int n_resid, const float *W1, const float *b1,
                         const float *w2, float b2, double tau_min, double tau_max, double *dx,
                         double *dlogit, double *dW1, double *db1, double *dw2, double *db2)
{
    if (N < 0 || H < 0 || W < 0 || C < 1 || R < 1 || k < 1 || k > C || n_resid < 0 ||
        n_resid > C || (layout != 0 && layout != 1) || !dx || !dlogit || !dW1 || !db1 || !dw2 ||
        !db2)
        return ORACLE_BAD_ARG;
    const int HW = H * W, E = R + 1;
    double *z = (double *)malloc(sizeof(double) * (size_t)C);
    double *u = (double *)malloc(sizeof(double) * (size_t)k);
    double *hpre = (double *)malloc(sizeof(double) * (size_t)k);
    double *a = (double *)malloc(sizeof(double) * (size_t)k);
    double *da = (double *)malloc(sizeof(double) * (size_t)k);
    double *dh = (double *)malloc(sizeof(double) * (size_t)k);
    double *dz = (double *)malloc(sizeof(double) * (size_t)C);
    double *aall = (double *)malloc(sizeof(double) * ((size_t)R * k + 1));
    if (!z || !u || !hpre || !a || !da || !dh || !dz || !aall) {
        free(z); free(u); free(hpre); free(a); free(da); free(dh); free(dz); free(aall);
        return ORACLE_NO_MEMORY;
    }
    for (int i = 0; i < R * k; ++i)
        dlogit[i] = 0.0;
    for (int i = 0; i < k * k; ++i)
        dW1[i] = 0.0;
    for (int j = 0; j < k; ++j) {
        db1[j] = 0.0;
        dw2[j] = 0.0;
    }
    *db2 = 0.0;
    for (int n = 0; n < N; ++n) {
        /* forward of example n: z, then per expert u, h, g, sigma, tau, a */
        for (int c = 0; c < C; ++c) {
            double s = 0.0;
            for (int p = 0; p < HW; ++p)
                s += (double)x[x_at(layout, n, p, c, HW, C)];
            z[c] = s / (double)HW;
            dz[c] = 0.0;
        }
        for (int e = 0; e < R; ++e) {
            const int32_t *S = packed_idx + (size_t)e * k;
            const float *L = packed_logits + (size_t)e * k;
            for (int i = 0; i < k; ++i)
                u[i] = z[S[i]];
            double g = (double)b2;
            for (int j = 0; j < k; ++j) {
                double t = (double)b1[j];
                for (int i = 0; i < k; ++i)
                    t += (double)W1[(size_t)j * k + i] * u[i];
                hpre[j] = t;
                g += (double)w2[j] * (t > 0.0 ? t : 0.0);
            }
            const double sig = 1.0 / (1.0 + exp(-g));
            const double tau = tau_min + (tau_max - tau_min) * sig;
            double m = (double)L[0];
            for (int i = 1; i < k; ++i)
                if ((double)L[i] > m)
                    m = (double)L[i];
            double sum = 0.0;
            for (int i = 0; i < k; ++i) {
                a[i] = exp(((double)L[i] - m) / tau);
                sum += a[i];
            }
            for (int i = 0; i < k; ++i) {
                a[i] /= sum;
                aall[(size_t)e * k + i] = a[i];
            }
            /* backward: routed mix -> weights -> temperature -> gate */
            for (int i = 0; i < k; ++i) {
                double s = 0.0;
                for (int p = 0; p < HW; ++p)
                    s += (double)dy[x_at(layout, n, p, e, HW, E)] *
                         (double)x[x_at(layout, n, p, S[i], HW, C)];
                da[i] = s;
            }
            double ada = 0.0;
            for (int i = 0; i < k; ++i)
                ada += a[i] * da[i];
            double dtau = 0.0;
            for (int i = 0; i < k; ++i) {
                const double ds = a[i] * (da[i] - ada);
                dlogit[(size_t)e * k + i] += ds / tau;
                dtau -= ds * (double)L[i] / (tau * tau);
            }
            const double dg = dtau * (tau_max - tau_min) * sig * (1.0 - sig);
            *db2 += dg;
            for (int j = 0; j < k; ++j) {
                const double r = hpre[j] > 0.0 ? hpre[j] : 0.0;
                dw2[j] += dg * r;
                dh[j] = hpre[j] > 0.0 ? dg * (double)w2[j] : 0.0;
                db1[j] += dh[j];
                for (int i = 0; i < k; ++i)
                    dW1[(size_t)j * k + i] += dh[j] * u[i];
            }
            for (int i = 0; i < k; ++i) {
                double du = 0.0;
                for (int j = 0; j < k; ++j)
                    du += (double)W1[(size_t)j * k + i] * dh[j];
                dz[S[i]] += du;
            }
        }
        /* dx: the routed experts' weights, the residual mean and the pool */
        for (int p = 0; p < HW; ++p)
            for (int c = 0; c < C; ++c)
                dx[x_at(layout, n, p, c, HW, C)] = dz[c] / (double)HW;
        for (int p = 0; p < HW; ++p) {
            for (int e = 0; e < R; ++e) {
                const double d = (double)dy[x_at(layout, n, p, e, HW, E)];
                for (int i = 0; i < k; ++i)
                    dx[x_at(layout, n, p, packed_idx[(size_t)e * k + i], HW, C)] +=
                        aall[(size_t)e * k + i] * d;
            }
            if (n_resid > 0) {
                const double d = (double)dy[x_at(layout, n, p, R, HW, E)] / (double)n_resid;
                for (int j = 0; j < n_resid; ++j)
                    dx[x_at(layout, n, p, resid[j], HW, C)] += d;
            }
        }
    }
    free(z); free(u); free(hpre); free(a); free(da); free(dh); free(dz); free(aall);
    return ORACLE_OK;
}

/*
 * Eq. (dynamic): the input-conditioned routing logits of each example.
 *   z = GAP(X) (Sec. 3.3), h(z) = ReLU(W_h z + b_h) in R^d,
 *   L_e(X)_c = L_{e,c} + <q_e (.) h(z), v_c> = L_{e,c} + sum_j q_{e,j} h_j v_{c,j}.
 * L [R][C] is the static routing matrix (row e = L_e), W_h [d][C] row-major,
 * b_h [d], V [C][d] (row c = v_c), Q [R][d] (row e = q_e). Outputs, double:
 * h_out [N][d] (optional) and Ldyn [N][R][C].
 */
int moce_oracle_dynamic_logits(const float *x, int N, int H, int W, int C, int layout, int R,
                               int d, const float *L, const float *Wh, const float *bh,
                               const float *V, const float *Q, double *h_out, double *Ldyn)
{
    if (N < 0 || H < 1 || W < 1 || C < 1 || R < 1 || d < 1 || (layout != 0 && layout != 1) ||
        !L || !Wh || !bh || !V || !Q || !Ldyn)
        return ORACLE_BAD_ARG;
    double *z = (double *)malloc(sizeof(double) * (size_t)C * (N > 0 ? N : 1));
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    if (!z || !h) {
        free(z);
        free(h);
        return ORACLE_NO_MEMORY;
    }
    moce_oracle_pool(x, N, H, W, C, layout, z);
    for (int n = 0; n < N; ++n) {
        const double *zn = z + (size_t)n * C;
        for (int j = 0; j < d; ++j) {
            double s = (double)bh[j];
            for (int c = 0; c < C; ++c)
                s += (double)Wh[(size_t)j * C + c] * zn[c];
            h[j] = (s > 0.0) ? s : 0.0; /* ReLU of the router bottleneck */
            if (h_out)
                h_out[(size_t)n * d + j] = h[j];
        }
        for (int e = 0; e < R; ++e)
            for (int c = 0; c < C; ++c) {
                double off = 0.0;
                for (int j = 0; j < d; ++j)
                    off += (double)Q[(size_t)e * d + j] * h[j] * (double)V[(size_t)c * d + j];
                Ldyn[((size_t)n * R + e) * C + c] = (double)L[(size_t)e * C + c] + off;
            }
    }
    free(z);
    free(h);
    return ORACLE_OK;
}
