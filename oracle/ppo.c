/*
 * Plain fp64 CPU oracle for the PrunePath sparse-FFN path.
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only the test suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load or call this
 * library.  It shares no code, header, table or constant with the CUDA
 * library: it has its own enums, its own bf16 decoding and its own maths.
 *
 * What it computes, step by step, in the order the paper states it
 * (PrunePath, Sec. 3.1 and Sec. 2):
 *   Eq. (routing_logits)        g = W_r^T x                         ppo_logits
 *   Eq. (softmax_prob)          p_j = exp(g_j) / sum_i exp(g_i)     ppo_select
 *   Sec. 3.1 (descending order) pi: p_{pi_1} >= ... >= p_{pi_E}     ppo_select
 *   Eq. (tau_thresh_activate)   A = {pi_1} U {pi_i : S_i < tau}     ppo_select
 *   Eq. (ffn), Eq. (moefication_decomp)  FFN_e(x) on expert block e  ppo_sparse_ffn
 *   Eq. (moe_output)            y = sum_{e in A} sigmoid(g_e) FFN_e(x)
 * and two further activation rules on the same router logits:
 *   Sec. 4.3 (top-k reconstruction analysis): the first k experts of pi
 *   Eq. (lte_hard_set)          A = {e : sigmoid(g_e) > delta}  (LTE's rule)
 * and the router statistics of the training objective (forward values):
 *   Eq. (entropy_loss), Eq. (load_balance_loss), L_gate (Sec. 4.2.3)          ppo_router_stats
 * and, for chaining layers into a decode step, the residual + RMS
 * normalisation x_{l+1} = RMSNorm(x_l + y_l)                                ppo_rmsnorm_residual
 * and the efficiency metric of the experiments:
 *   Sec. 4.1 (s_FFN)  s = 1 - (1/(N L E)) sum_i sum_l |A_l(x_i)|            ppo_ffn_sparsity
 * Every floating-point operation is done in double precision with plain
 * sequential loops; the inputs (fp32 or bf16) are widened exactly.
 *
 * Readings where the paper is silent (each listed in the design notes):
 *  - Tie-break of the descending order: equal logits are ordered by the
 *    lower expert index first.
 *  - Two cut rules.  PAPER is Eq. (tau_thresh_activate) literally: the
 *    ranks whose inclusive prefix mass is strictly below tau, plus rank 1.
 *    MIN_PREFIX is the shortest descending prefix whose mass reaches p,
 *    i.e. it also keeps the rank that crosses p.
 *  - p >= 1 selects all E experts under both rules (the warm-up setting
 *    tau_warm = 1.05 of Sec. 3.2 activates every expert); p NaN is an error.
 *  - TOPK takes k from the same argument p: k = floor(p), at least 1 and
 *    at most E.  LTE takes delta from p; delta <= 0 selects every expert
 *    (a sigmoid is positive everywhere, although in fp64 it underflows to 0
 *    below g = -745), and the set may be empty.  Both list the selected
 *    experts in the order pi.
 *  - Non-gated FFN variants (Sec. 2.1 says the analysis covers any FFN that
 *    is separable along d_ff): h = relu(x W_up) or h = gelu_tanh(x W_up),
 *    the tanh form of GELU being the GPT-2 one.  No biases (Sec. 2.1).
 *  - Storage: W_r is [E][d] (row j is the routing vector of expert j);
 *    W_gate and W_up are [d_ff][d] (row n holds neuron n's input weights),
 *    W_down is [d][d_ff].  Expert e owns neurons [e*d_e, (e+1)*d_e).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define PPO_F32 0
#define PPO_BF16 1
#define PPO_F64 2

#define PPO_ACT_RELU 0
#define PPO_ACT_GELU_TANH 1
#define PPO_ACT_SWIGLU 2

#define PPO_GATE_SIGMOID 0
#define PPO_GATE_NONE 1

#define PPO_RULE_MIN_PREFIX 0
#define PPO_RULE_PAPER 1
#define PPO_RULE_TOPK 2
#define PPO_RULE_LTE 3

#define PPO_OK 0
#define PPO_ERR_ARG 1
#define PPO_ERR_NONFINITE 9

/* Exact widening of one stored element to double. */
static double ld(const void *base, int dtype, size_t i)
{
    if (dtype == PPO_F64)
        return ((const double *)base)[i];
    if (dtype == PPO_F32)
        return (double)((const float *)base)[i];
    /* bf16 is the upper half of an IEEE binary32 word. */
    uint32_t bits = ((uint32_t)((const uint16_t *)base)[i]) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

static int dtype_ok(int dt) { return dt == PPO_F32 || dt == PPO_BF16 || dt == PPO_F64; }

/* ---- activations (Sec. 2.1) --------------------------------------------- */

double ppo_sigmoid(double v) { return 1.0 / (1.0 + exp(-v)); }

double ppo_silu(double v) { return v / (1.0 + exp(-v)); }

double ppo_gelu_tanh(double v)
{
    const double k = sqrt(2.0 / M_PI);
    return 0.5 * v * (1.0 + tanh(k * (v + 0.044715 * v * v * v)));
}

double ppo_relu(double v) { return v > 0.0 ? v : 0.0; }

/* h_n for one intermediate neuron.  a = x W_up[:, n], b = x W_gate[:, n]. */
double ppo_act(int act, double a, double b)
{
    if (act == PPO_ACT_SWIGLU)
        return ppo_silu(b) * a; /* Eq. (ffn): phi(x W_gate) (.) x W_up, phi = SiLU */
    if (act == PPO_ACT_RELU)
        return ppo_relu(a);
    return ppo_gelu_tanh(a);
}

/* ---- Eq. (routing_logits) ------------------------------------------------ */

/* g[t][j] = sum_i W_r[j][i] * x[t][i] for every token t and expert j. */
int ppo_logits(const void *x, int x_dt, int T, int d, const void *Wr, int wr_dt, int E,
               double *g)
{
    if (!dtype_ok(x_dt) || !dtype_ok(wr_dt) || T < 0 || d <= 0 || E <= 0)
        return PPO_ERR_ARG;
#pragma omp parallel for schedule(static)
    for (int t = 0; t < T; t++) {
        for (int j = 0; j < E; j++) {
            double acc = 0.0;
            for (int i = 0; i < d; i++)
                acc += ld(Wr, wr_dt, (size_t)j * d + i) * ld(x, x_dt, (size_t)t * d + i);
            g[(size_t)t * E + j] = acc;
        }
    }
    return PPO_OK;
}

/* ---- softmax, descending order, cumulative-mass cut ---------------------- */

typedef struct {
    double g;
    int j;
} ranked;

/* Descending logit, then ascending expert index (the tie-break reading). */
static int by_rank(const void *pa, const void *pb)
{
    const ranked *a = (const ranked *)pa, *b = (const ranked *)pb;
    if (a->g > b->g)
        return -1;
    if (a->g < b->g)
        return 1;
    return (a->j > b->j) - (a->j < b->j);
}

/*
 * For each token: softmax over its E logits (Eq. softmax_prob), the
 * descending order pi (Sec. 3.1), the inclusive prefix masses
 * S_i = sum_{r<=i} p_{pi_r}, and the activated set (Eq. tau_thresh_activate,
 * under the chosen rule; or the top-k / LTE sets, p then carrying k / delta).
 *
 * Outputs: counts[t] = |A|; ids[t][r] = pi_{r+1} for r < |A|, -1 beyond;
 * cum[t][r] = S_{r+1} for all r < E (nullable); probs[t][j] = p_j (nullable).
 * Returns PPO_ERR_ARG for a NaN p, PPO_ERR_NONFINITE if any logit is not
 * finite (that token then gets counts[t] = 0).
 */
int ppo_select(const double *g, int T, int E, double p, int rule, int *counts, int *ids,
               double *cum, double *probs)
{
    if (isnan(p) || T < 0 || E <= 0 || rule < PPO_RULE_MIN_PREFIX || rule > PPO_RULE_LTE)
        return PPO_ERR_ARG;
    int status = PPO_OK;
    ranked *order = (ranked *)malloc(sizeof(ranked) * (size_t)E);
    double *prob = (double *)malloc(sizeof(double) * (size_t)E);
    if (!order || !prob) {
        free(order);
        free(prob);
        return PPO_ERR_ARG;
    }
    for (int t = 0; t < T; t++) {
        const double *gt = g + (size_t)t * E;
        int *idt = ids + (size_t)t * E;
        int finite = 1;
        for (int j = 0; j < E; j++)
            finite &= isfinite(gt[j]) ? 1 : 0;
        for (int r = 0; r < E; r++)
            idt[r] = -1;
        if (!finite) {
            counts[t] = 0;
            status = PPO_ERR_NONFINITE;
            if (cum)
                for (int r = 0; r < E; r++)
                    cum[(size_t)t * E + r] = NAN;
            continue;
        }
        /* Eq. (softmax_prob).  Dividing numerator and denominator by
           exp(max g) leaves every p_j unchanged and keeps exp() finite. */
        double m = gt[0];
        for (int j = 1; j < E; j++)
            if (gt[j] > m)
                m = gt[j];
        double Z = 0.0;
        for (int j = 0; j < E; j++) {
            prob[j] = exp(gt[j] - m);
            Z += prob[j];
        }
        for (int j = 0; j < E; j++)
            prob[j] /= Z;
        if (probs)
            for (int j = 0; j < E; j++)
                probs[(size_t)t * E + j] = prob[j];

        /* Descending order pi.  Softmax is strictly increasing in g, so the
           order of the logits is the order of the probabilities. */
        for (int j = 0; j < E; j++) {
            order[j].g = gt[j];
            order[j].j = j;
        }
        qsort(order, (size_t)E, sizeof(ranked), by_rank);

        /* Inclusive prefix masses S_i, summed in rank order. */
        double S = 0.0;
        int below = 0; /* #{i : S_i < p}; S is non-decreasing so these are ranks 1..below */
        for (int r = 0; r < E; r++) {
            S += prob[order[r].j];
            if (cum)
                cum[(size_t)t * E + r] = S;
            if (S < p)
                below++;
        }

        if (rule == PPO_RULE_TOPK) {
            /* the k highest-ranked experts; p carries k */
            int k = p >= (double)E ? E : (p >= 1.0 ? (int)floor(p) : 1);
            counts[t] = k;
            for (int r = 0; r < k; r++)
                idt[r] = order[r].j;
            continue;
        }
        if (rule == PPO_RULE_LTE) {
            /* Eq. (lte_hard_set): every expert whose sigmoid score exceeds
               delta = p, each tested on its own, listed in the order pi */
            int k = 0;
            for (int r = 0; r < E; r++)
                if (p <= 0.0 || ppo_sigmoid(order[r].g) > p)
                    idt[k++] = order[r].j;
            counts[t] = k;
            continue;
        }

        int k;
        if (p >= 1.0) {
            k = E; /* warm-up reading: every expert active */
        } else if (rule == PPO_RULE_PAPER) {
            /* {pi_1} U {pi_i : S_i < tau} */
            k = below > 1 ? below : 1;
        } else {
            /* shortest prefix with S_k >= p (all E if rounding keeps S_E < p) */
            k = below + 1 < E ? below + 1 : E;
        }
        counts[t] = k;
        for (int r = 0; r < k; r++)
            idt[r] = order[r].j;
    }
    free(order);
    free(prob);
    return status;
}

/* ---- Eq. (ffn), Eq. (moefication_decomp), Eq. (moe_output) ---------------- */

/*
 * y[t] = sum_{r < counts[t]} w(t, ids[t][r]) * FFN_e(x_t), e = ids[t][r], with
 * FFN_e(x) = sum_{n in block e} h_n(x) * W_down[:, n]
 * and w = sigmoid(g[t][e]) (PPO_GATE_SIGMOID, Eq. moe_output) or 1
 * (PPO_GATE_NONE: the plain MoEfication sum of Eq. moefication_decomp).
 * Wg is ignored (may be NULL) unless act == PPO_ACT_SWIGLU.
 */
int ppo_sparse_ffn(const void *x, int x_dt, int T, int d, int E, int de, int act, int gate_mode,
                   const void *Wg, const void *Wu, const void *Wd, int w_dt, const int *counts,
                   const int *ids, const double *g, double *y)
{
    if (!dtype_ok(x_dt) || !dtype_ok(w_dt) || T < 0 || d <= 0 || E <= 0 || de <= 0)
        return PPO_ERR_ARG;
    if (act == PPO_ACT_SWIGLU && !Wg)
        return PPO_ERR_ARG;
    const int dff = E * de;
    int bad_id = 0;
#pragma omp parallel for schedule(dynamic) reduction(| : bad_id)
    for (int t = 0; t < T; t++) {
        double *yt = y + (size_t)t * d;
        for (int j = 0; j < d; j++)
            yt[j] = 0.0;
        for (int r = 0; r < counts[t]; r++) {
            const int e = ids[(size_t)t * E + r];
            if (e < 0 || e >= E) {
                bad_id = 1;
                continue;
            }
            const double w =
                gate_mode == PPO_GATE_NONE ? 1.0 : ppo_sigmoid(g[(size_t)t * E + e]);
            for (int n = e * de; n < (e + 1) * de; n++) {
                double a = 0.0, b = 0.0;
                for (int i = 0; i < d; i++) {
                    const double xi = ld(x, x_dt, (size_t)t * d + i);
                    a += ld(Wu, w_dt, (size_t)n * d + i) * xi;
                    if (act == PPO_ACT_SWIGLU)
                        b += ld(Wg, w_dt, (size_t)n * d + i) * xi;
                }
                const double h = ppo_act(act, a, b);
                for (int j = 0; j < d; j++)
                    yt[j] += w * h * ld(Wd, w_dt, (size_t)j * dff + n);
            }
        }
    }
    return bad_id ? PPO_ERR_ARG : PPO_OK;
}

/* Eq. (ffn) on the whole intermediate dimension, no routing. */
int ppo_dense_ffn(const void *x, int x_dt, int T, int d, int dff, int act, const void *Wg,
                  const void *Wu, const void *Wd, int w_dt, double *y)
{
    if (!dtype_ok(x_dt) || !dtype_ok(w_dt) || T < 0 || d <= 0 || dff <= 0)
        return PPO_ERR_ARG;
    if (act == PPO_ACT_SWIGLU && !Wg)
        return PPO_ERR_ARG;
#pragma omp parallel for schedule(dynamic)
    for (int t = 0; t < T; t++) {
        double *yt = y + (size_t)t * d;
        for (int j = 0; j < d; j++)
            yt[j] = 0.0;
        for (int n = 0; n < dff; n++) {
            double a = 0.0, b = 0.0;
            for (int i = 0; i < d; i++) {
                const double xi = ld(x, x_dt, (size_t)t * d + i);
                a += ld(Wu, w_dt, (size_t)n * d + i) * xi;
                if (act == PPO_ACT_SWIGLU)
                    b += ld(Wg, w_dt, (size_t)n * d + i) * xi;
            }
            const double h = ppo_act(act, a, b);
            for (int j = 0; j < d; j++)
                yt[j] += h * ld(Wd, w_dt, (size_t)j * dff + n);
        }
    }
    return PPO_OK;
}

/* The whole layer for T tokens: logits, selection, sparse FFN.  g, counts,
   ids are outputs too (g is [T][E] doubles, ids [T][E]). */
int ppo_layer(const void *x, int x_dt, int T, int d, int E, int de, int act, int gate_mode,
              int rule, double p, const void *Wr, const void *Wg, const void *Wu, const void *Wd,
              int w_dt, double *g, int *counts, int *ids, double *y)
{
    int s = ppo_logits(x, x_dt, T, d, Wr, w_dt, E, g);
    if (s != PPO_OK)
        return s;
    s = ppo_select(g, T, E, p, rule, counts, ids, NULL, NULL);
    if (s == PPO_ERR_ARG)
        return s;
    int s2 = ppo_sparse_ffn(x, x_dt, T, d, E, de, act, gate_mode, Wg, Wu, Wd, w_dt, counts, ids,
                            g, y);
    return s != PPO_OK ? s : s2;
}

/* ---- router statistics (Sec. 3.2 and Sec. 4.2.3) --------------------------- */

/*
 * Over a batch of B = T tokens with router logits g[t][j] and softmax
 * probabilities p_tj (Eq. softmax_prob):
 *   out[0] = L_ent  = -(1/B) sum_t sum_j p_tj log(p_tj + eps)   (Eq. entropy_loss)
 *   out[1] = L_bal  = E sum_j ((1/B) sum_t p_tj)^2              (Eq. load_balance_loss)
 *   out[2] = L_gate = (1/(B E)) sum_t sum_j sigmoid(g_tj)        (the gate-magnitude
 *            regulariser of the instruction-tuning experiments)
 * Forward values only.  Returns PPO_ERR_ARG for T < 1 or E < 1 and
 * PPO_ERR_NONFINITE if a logit is not finite (out is then NaN).
 */
int ppo_router_stats(const double *g, int T, int E, double eps, double *out)
{
    if (T < 1 || E < 1 || isnan(eps))
        return PPO_ERR_ARG;
    double *colsum = (double *)calloc((size_t)E, sizeof(double));
    double *prob = (double *)malloc(sizeof(double) * (size_t)E);
    if (!colsum || !prob) {
        free(colsum);
        free(prob);
        return PPO_ERR_ARG;
    }
    double ent = 0.0, gate = 0.0;
    int status = PPO_OK;
    for (int t = 0; t < T; t++) {
        const double *gt = g + (size_t)t * E;
        int finite = 1;
        for (int j = 0; j < E; j++)
            finite &= isfinite(gt[j]) ? 1 : 0;
        if (!finite) {
            status = PPO_ERR_NONFINITE;
            break;
        }
        double m = gt[0];
        for (int j = 1; j < E; j++)
            if (gt[j] > m)
                m = gt[j];
        double Z = 0.0;
        for (int j = 0; j < E; j++) {
            prob[j] = exp(gt[j] - m);
            Z += prob[j];
        }
        for (int j = 0; j < E; j++) {
            const double pj = prob[j] / Z;
            ent -= pj * log(pj + eps);
            colsum[j] += pj;
            gate += ppo_sigmoid(gt[j]);
        }
    }
    if (status == PPO_OK) {
        double bal = 0.0;
        for (int j = 0; j < E; j++) {
            const double f = colsum[j] / (double)T;
            bal += f * f;
        }
        out[0] = ent / (double)T;
        out[1] = (double)E * bal;
        out[2] = gate / ((double)T * (double)E);
    } else {
        out[0] = out[1] = out[2] = NAN;
    }
    free(colsum);
    free(prob);
    return status;
}

/* ---- chained decode step ------------------------------------------------- */

/*
 * Input of the next layer of a stack of MoEfied FFN layers with a residual
 * connection and RMS normalisation (the post-norm form x_{l+1} =
 * RMSNorm(x_l + y_l)):
 *   v = x_prev + y_prev                  (y_prev NULL: v = x_prev)
 *   out = v / sqrt(mean(v^2) + eps) * gamma   (gamma NULL: unit weights)
 * per token (row of d elements), in fp64.
 */
int ppo_rmsnorm_residual(const void *x_prev, const void *y_prev, const void *gamma, int dt, int T, int d,
                         double eps, double *out)
{
    if (!dtype_ok(dt) || !x_prev || T < 0 || d <= 0 || isnan(eps))
        return PPO_ERR_ARG;
    for (int t = 0; t < T; t++) {
        double ss = 0.0;
        for (int i = 0; i < d; i++) {
            double v = ld(x_prev, dt, (size_t)t * d + i);
            if (y_prev)
                v += ld(y_prev, dt, (size_t)t * d + i);
            out[(size_t)t * d + i] = v;
            ss += v * v;
        }
        const double r = 1.0 / sqrt(ss / (double)d + eps);
        for (int i = 0; i < d; i++) {
            const double g = gamma ? ld(gamma, dt, (size_t)i) : 1.0;
            out[(size_t)t * d + i] *= r * g;
        }
    }
    return PPO_OK;
}

/* ---- FFN sparsity (Sec. 4.1) --------------------------------------------- */

/*
 * The average FFN sparsity of N tokens through L layers of E experts each:
 *   s_FFN = 1 - (1 / (N L E)) sum_{i=1..N} sum_{l=1..L} |A_l(x_i)|
 * where |A_l(x_i)| = counts[l * N + i], the number of experts activated for
 * token i at layer l (0 <= count <= E; LTE's rule can activate none).
 * Also returns the total sum of |A| (k_sum) and a histogram of the set sizes,
 * hist[c] = #{(i, l) : |A_l(x_i)| = c} for c = 0..E (E + 1 entries).
 * Returns PPO_ERR_ARG for N < 1, L < 1, E < 1 or a count outside [0, E].
 */
int ppo_ffn_sparsity(const int *counts, int N, int L, int E, unsigned long long *k_sum, unsigned long long *hist,
                     double *s_ffn)
{
    if (!counts || N < 1 || L < 1 || E < 1)
        return PPO_ERR_ARG;
    for (int c = 0; c <= E; c++)
        hist[c] = 0ull;
    unsigned long long total = 0ull;
    for (int i = 0; i < N; i++) {
        for (int l = 0; l < L; l++) {
            const int c = counts[(size_t)l * N + i];
            if (c < 0 || c > E)
                return PPO_ERR_ARG;
            total += (unsigned long long)c;
            hist[c] += 1ull;
        }
    }
    *k_sum = total;
    *s_ffn = 1.0 - (double)total / ((double)N * (double)L * (double)E);
    return PPO_OK;
}
