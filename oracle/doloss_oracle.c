/*
 * DO-loss oracle: a plain, slow, single-threaded CPU statement of what the
 * DO-loss hot path computes, written from "Function Over Form: Distributional
 * Orthogonalization in Mixture-of-Experts with Replica Expert Mechanism".
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call this file:
 * only the tests, the package smoke check and the CPU-baseline leg of the
 * benchmark use it.  It shares no code, header, table or helper with the CUDA
 * library; it is compiled on its own with gcc, without fast-math.
 *
 * Notation follows Sec. 3.1: n experts (E), K selected per token (k), a batch
 * of m tokens (T).  f_it is the binary load bit, F_i the load signature,
 * G_ij the Hamming distance, C_ij the direction term, p_it the normalized
 * routing probability.  Every floating-point quantity is computed in double
 * from the fp32 logits it is given.  Each function works on one problem (one
 * layer); batched layers are independent problems.
 *
 * Readings of the paper that the code takes where the text is silent:
 *  - Top-K is taken over the raw logits, larger value first, equal values
 *    resolved in favour of the lower expert index (sigmoid and softmax are
 *    monotone, so the set is the Top-K of the scores in exact arithmetic).
 *  - p_it is the dense normalized probability over all n experts (Sec. 3.1.1:
 *    sum_i p_it = 1; App. A keeps the Top-K mass s_K below one).
 *  - G may be a summed distance matrix from several data-parallel replicas,
 *    entering the loss as d_scale * D (Sec. 3.1.4, Eq. global_do).
 *  - grad_scale multiplies the gradient only (the lambda of Eq. 10 or an
 *    upstream gradient); the loss value is unscaled.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define GATE_SIGMOID_NORM 0
#define GATE_SOFTMAX 1

/* Sec. 3.1.1, Eq. (1): f_it = 1(i in Top-K(x_t)).
 * K passes of an argmax over the experts not yet chosen; a strict '>' while
 * scanning i upward keeps the lowest index among equal maxima.  f is [T][E]. */
void oracle_select(const float *z, int64_t T, int32_t E, int32_t k, uint8_t *f)
{
    for (int64_t t = 0; t < T; ++t) {
        const float *zt = z + t * (int64_t)E;
        uint8_t *ft = f + t * (int64_t)E;
        for (int32_t i = 0; i < E; ++i) ft[i] = 0;
        for (int32_t pass = 0; pass < k; ++pass) {
            int32_t best = -1;
            double bv = 0.0;
            for (int32_t i = 0; i < E; ++i) {
                if (ft[i]) continue;
                double v = (double)zt[i];
                if (best < 0 || v > bv) { best = i; bv = v; }
            }
            ft[best] = 1;
        }
    }
}

/* Load signature F_i in {0,1}^m stored as 32-bit words, [E][W], W=ceil(T/32):
 * bit (t mod 32) of word t/32 is f_it; bits past T are zero. */
void oracle_pack(const uint8_t *f, int64_t T, int32_t E, uint32_t *bits)
{
    int64_t W = (T + 31) / 32;
    memset(bits, 0, sizeof(uint32_t) * (size_t)(W * E));
    for (int64_t t = 0; t < T; ++t)
        for (int32_t i = 0; i < E; ++i)
            if (f[t * E + i]) bits[(int64_t)i * W + t / 32] |= (uint32_t)1u << (t % 32);
}

/* n_i = ||F_i||_1, the tokens routed to expert i (App. C.3). */
void oracle_counts(const uint8_t *f, int64_t T, int32_t E, int32_t *counts)
{
    for (int32_t i = 0; i < E; ++i) counts[i] = 0;
    for (int64_t t = 0; t < T; ++t)
        for (int32_t i = 0; i < E; ++i) counts[i] += f[t * E + i];
}

/* Eq. gij_cij (Sec. 3.1.3): G_ij = ||F_i - F_j||_1 = sum_t |f_it - f_jt|,
 * accumulated over tokens [t0, t1) into D (the caller zeroes D first). */
void oracle_hamming(const uint8_t *f, int64_t t0, int64_t t1, int32_t E, int32_t *D)
{
    for (int64_t t = t0; t < t1; ++t) {
        const uint8_t *ft = f + t * E;
        for (int32_t i = 0; i < E; ++i)
            for (int32_t j = 0; j < E; ++j)
                D[(int64_t)i * E + j] += abs((int)ft[i] - (int)ft[j]);
    }
}

/* The same distance read off the packed signatures: the number of positions
 * where F_i and F_j differ is the population count of their XOR. */
static int popcount32(uint32_t x)
{
    return __builtin_popcount(x);   /* the compiler's population count */
}

void oracle_hamming_bits(const uint32_t *bits, int64_t T, int32_t E, int32_t *D)
{
    int64_t W = (T + 31) / 32;
    for (int32_t i = 0; i < E; ++i)
        for (int32_t j = 0; j < E; ++j) {
            int64_t acc = 0;
            for (int64_t w = 0; w < W; ++w)
                acc += popcount32(bits[(int64_t)i * W + w] ^ bits[(int64_t)j * W + w]);
            D[(int64_t)i * E + j] = (int32_t)acc;
        }
}

/* Routing probability of one token (Sec. 3.1.1; App. A):
 *  sigmoid-norm: s_i = 1/(1+exp(-z_i)), p_i = s_i / sum_i' s_i'
 *  softmax:      p_i = exp(z_i - max z) / sum_i' exp(z_i' - max z)     */
static void gate_row(const float *zt, int32_t E, int32_t gate, double *p)
{
    double sum = 0.0;
    if (gate == GATE_SOFTMAX) {
        double mx = (double)zt[0];
        for (int32_t i = 1; i < E; ++i)
            if ((double)zt[i] > mx) mx = (double)zt[i];
        for (int32_t i = 0; i < E; ++i) { p[i] = exp((double)zt[i] - mx); sum += p[i]; }
    } else {
        for (int32_t i = 0; i < E; ++i) { p[i] = 1.0 / (1.0 + exp(-(double)zt[i])); sum += p[i]; }
    }
    for (int32_t i = 0; i < E; ++i) p[i] /= sum;
}

void oracle_gate(const float *z, int64_t T, int32_t E, int32_t gate, double *p)
{
    for (int64_t t = 0; t < T; ++t) gate_row(z + t * E, E, gate, p + t * E);
}

/* Eq. gij_cij: C_ij = sum_t p_it (f_it - f_jt), accumulated over tokens
 * [t0, t1) into C ([E][E], zeroed by the caller). */
void oracle_direction(const float *z, const uint8_t *f, int64_t t0, int64_t t1,
                      int32_t E, int32_t gate, double *C)
{
    double *p = (double *)malloc(sizeof(double) * (size_t)E);
    for (int64_t t = t0; t < t1; ++t) {
        const uint8_t *ft = f + t * E;
        gate_row(z + t * E, E, gate, p);
        for (int32_t i = 0; i < E; ++i)
            for (int32_t j = 0; j < E; ++j)
                C[(int64_t)i * E + j] += p[i] * ((double)ft[i] - (double)ft[j]);
    }
    free(p);
}

/* Eq. do_loss: L_DO = 1/(m^2 k) sum_i sum_j G_ij C_ij, with G = d_scale * D
 * (Eq. global_do when D is a sum over replicas; d_scale = 1 locally). */
double oracle_loss(const int32_t *D, const double *C, int32_t E, int64_t m, int32_t k,
                   double d_scale)
{
    double acc = 0.0;
    for (int32_t i = 0; i < E; ++i)
        for (int32_t j = 0; j < E; ++j)
            acc += d_scale * (double)D[(int64_t)i * E + j] * C[(int64_t)i * E + j];
    return acc / ((double)m * (double)m * (double)k);
}

/* Gradient of Eq. do_loss with G (and F) held constant (Sec. 3.1.3: G is
 * detached).  C_ij is linear in p_it and no other C_i'j depends on p_it, so
 * dL/dp_it = 1/(m^2 k) sum_j G_ij (f_it - f_jt).  Tokens [t0, t1); g is [T][E]. */
void oracle_dloss_dp(const int32_t *D, const uint8_t *f, int64_t t0, int64_t t1,
                     int32_t E, int64_t m, int32_t k, double d_scale, double *g)
{
    double norm = 1.0 / ((double)m * (double)m * (double)k);
    for (int64_t t = t0; t < t1; ++t) {
        const uint8_t *ft = f + t * E;
        for (int32_t i = 0; i < E; ++i) {
            double acc = 0.0;
            for (int32_t j = 0; j < E; ++j)
                acc += d_scale * (double)D[(int64_t)i * E + j] * ((double)ft[i] - (double)ft[j]);
            g[t * E + i] = acc * norm;
        }
    }
}

/* Chain rule through the router gate, with the Jacobian written out entry by
 * entry: dz_lt = grad_scale * sum_i (d p_it / d z_lt) g_it.
 *  sigmoid-norm: d p_i / d z_l = (delta_il - p_i) / S * s_l (1 - s_l), S = sum s,
 *                with 1 - s_l evaluated as sigmoid(-z_l) (no cancellation for
 *                large z_l)
 *  softmax:      d p_i / d z_l = p_i (delta_il - p_l)                          */
void oracle_gate_backward(const float *z, const double *g, int64_t t0, int64_t t1,
                          int32_t E, int32_t gate, double grad_scale, double *dz)
{
    double *p = (double *)malloc(sizeof(double) * (size_t)E);
    double *s = (double *)malloc(sizeof(double) * (size_t)E);
    for (int64_t t = t0; t < t1; ++t) {
        const float *zt = z + t * E;
        const double *gt = g + t * E;
        gate_row(zt, E, gate, p);
        double S = 0.0;
        for (int32_t i = 0; i < E; ++i) { s[i] = 1.0 / (1.0 + exp(-(double)zt[i])); S += s[i]; }
        for (int32_t l = 0; l < E; ++l) {
            double acc = 0.0;
            for (int32_t i = 0; i < E; ++i) {
                double delta = (i == l) ? 1.0 : 0.0;
                double J;
                if (gate == GATE_SOFTMAX)
                    J = p[i] * (delta - p[l]);
                else
                    J = (delta - p[i]) / S * s[l] * (1.0 / (1.0 + exp((double)zt[l])));
                acc += J * gt[i];
            }
            dz[t * E + l] = grad_scale * acc;
        }
    }
    free(p);
    free(s);
}

/* Eq. origin_do: L_origin_DO = sum_{i != j} ||F_i - F_j||_1^2, exact in int64. */
int64_t oracle_origin_do(const int32_t *D, int32_t E)
{
    int64_t acc = 0;
    for (int32_t i = 0; i < E; ++i)
        for (int32_t j = 0; j < E; ++j)
            if (i != j) acc += (int64_t)D[(int64_t)i * E + j] * (int64_t)D[(int64_t)i * E + j];
    return acc;
}

/* One problem end to end, the steps in the paper's order: Top-K and the load
 * signatures (Sec. 3.1.1), the detached Hamming matrix and the direction term
 * (Eq. gij_cij), the loss (Eq. do_loss) and its gradient to the logits.
 * dz may be NULL (forward only).  Returns 0, or -1 if memory ran out. */
int oracle_forward_backward(const float *z, int64_t T, int32_t E, int32_t k, int32_t gate,
                            double d_scale, double grad_scale, uint32_t *bits, int32_t *counts,
                            int32_t *D, double *loss, int64_t *origin_do, double *dz)
{
    uint8_t *f = (uint8_t *)malloc((size_t)(T * E));
    double *C = (double *)calloc((size_t)E * (size_t)E, sizeof(double));
    if (!f || !C) { free(f); free(C); return -1; }
    oracle_select(z, T, E, k, f);
    oracle_pack(f, T, E, bits);
    oracle_counts(f, T, E, counts);
    oracle_hamming_bits(bits, T, E, D);
    oracle_direction(z, f, 0, T, E, gate, C);
    *loss = oracle_loss(D, C, E, T, k, d_scale);
    *origin_do = oracle_origin_do(D, E);
    if (dz) {
        double *g = (double *)malloc(sizeof(double) * (size_t)(T * E));
        if (!g) { free(f); free(C); return -1; }
        oracle_dloss_dp(D, f, 0, T, E, T, k, d_scale, g);
        oracle_gate_backward(z, g, 0, T, E, gate, grad_scale, dz);
        free(g);
    }
    free(f);
    free(C);
    return 0;
}

/* Routing outputs of the router (Sec. 3.1.1): of the dense p_t, only the K
 * chosen entries keep their value, and those K are re-normalized to sum to
 * one; they weight the chosen experts' outputs.  Per token t, ids[t][q] is the
 * q-th expert chosen by the argmax passes of oracle_select (largest logit
 * first, equal logits lower index first) and
 *     combine[t][q] = p_{ids[t][q],t} / sum_{q'} p_{ids[t][q'],t},
 * with p from gate_row.  ids and combine are [T][k]. */
void oracle_route(const float *z, int64_t T, int32_t E, int32_t k, int32_t gate, int32_t *ids,
                  double *combine)
{
    double *p = (double *)malloc(sizeof(double) * (size_t)E);
    uint8_t *taken = (uint8_t *)malloc((size_t)E);
    for (int64_t t = 0; t < T; ++t) {
        const float *zt = z + t * (int64_t)E;
        int32_t *it = ids + t * (int64_t)k;
        double *ct = combine + t * (int64_t)k;
        for (int32_t i = 0; i < E; ++i) taken[i] = 0;
        for (int32_t pass = 0; pass < k; ++pass) {
            int32_t best = -1;
            double bv = 0.0;
            for (int32_t i = 0; i < E; ++i) {
                if (taken[i]) continue;
                double v = (double)zt[i];
                if (best < 0 || v > bv) { best = i; bv = v; }
            }
            taken[best] = 1;
            it[pass] = best;
        }
        gate_row(zt, E, gate, p);
        double kept = 0.0;
        for (int32_t q = 0; q < k; ++q) kept += p[it[q]];
        for (int32_t q = 0; q < k; ++q) ct[q] = p[it[q]] / kept;
    }
    free(p);
    free(taken);
}

/* Dispatch order of the routed (token, choice) pairs: grouped by expert,
 * expert 0 first, and by token inside an expert (a stable counting sort of
 * the pairs, taken in token order, by expert id).
 *   offsets [E+1]: rows of expert e are offsets[e] .. offsets[e+1]-1
 *                  (offsets[e+1] - offsets[e] = n_e, offsets[E] = T k)
 *   rows [T k]:    the token of each row
 *   pos [T][k]:    the row of the pair (t, q); rows[pos[t][q]] = t        */
void oracle_dispatch(const int32_t *ids, int64_t T, int32_t E, int32_t k, int32_t *offsets,
                     int32_t *rows, int32_t *pos)
{
    int64_t *fill = (int64_t *)calloc((size_t)E, sizeof(int64_t));
    for (int32_t e = 0; e <= E; ++e) offsets[e] = 0;
    for (int64_t t = 0; t < T; ++t)
        for (int32_t q = 0; q < k; ++q) offsets[ids[t * k + q] + 1] += 1;
    for (int32_t e = 0; e < E; ++e) offsets[e + 1] += offsets[e];
    for (int64_t t = 0; t < T; ++t)
        for (int32_t q = 0; q < k; ++q) {
            int32_t e = ids[t * k + q];
            int64_t r = offsets[e] + fill[e]++;
            rows[r] = (int32_t)t;
            pos[t * k + q] = (int32_t)r;
        }
    free(fill);
}

/* bf16 is the upper half of an IEEE binary32: widening it is exact. */
static double bf16_value(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

void oracle_bf16_to_double(const uint16_t *h, int64_t n, double *out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = bf16_value(h[i]);
}

/* The router that produces the logits of Eq. 1 (Sec. 4.1: a linear map from
 * the hidden size to the n experts, no bias, as in the Qwen3-MoE architecture
 * the paper trains): z_te = sum_h X_th W_eh, with X [T][H] and W [E][H] in
 * bf16 and every product and sum in double.  z is [T][E]. */
void oracle_router_logits(const uint16_t *X, const uint16_t *Wr, int64_t T, int32_t H, int32_t E,
                          double *z)
{
    for (int64_t t = 0; t < T; ++t)
        for (int32_t e = 0; e < E; ++e) {
            double acc = 0.0;
            for (int32_t h = 0; h < H; ++h)
                acc += bf16_value(X[t * H + h]) * bf16_value(Wr[(int64_t)e * H + h]);
            z[t * E + e] = acc;
        }
}

/* Gradients of that linear map for an upstream gradient dz [T][E] (double):
 * dW_eh = sum_t dz_te X_th ([E][H]) and, when dX is not NULL,
 * dX_th = sum_e dz_te W_eh ([T][H]). */
void oracle_router_grad(const uint16_t *X, const uint16_t *Wr, const double *dz, int64_t T,
                        int32_t H, int32_t E, double *dW, double *dX)
{
    for (int32_t e = 0; e < E; ++e)
        for (int32_t h = 0; h < H; ++h) {
            double acc = 0.0;
            for (int64_t t = 0; t < T; ++t) acc += dz[t * E + e] * bf16_value(X[t * H + h]);
            dW[(int64_t)e * H + h] = acc;
        }
    if (!dX) return;
    for (int64_t t = 0; t < T; ++t)
        for (int32_t h = 0; h < H; ++h) {
            double acc = 0.0;
            for (int32_t e = 0; e < E; ++e) acc += dz[t * E + e] * bf16_value(Wr[(int64_t)e * H + h]);
            dX[t * H + h] = acc;
        }
}

/* The other reading of which p enters C_ij (Sec. 3.1.1 describes both the
 * dense normalized p and, after Top-K, the K chosen values re-normalized):
 * mode 0 takes the dense p of gate_row, mode 1 the re-normalized top-K
 * weights (zero for the experts not chosen).  C is [E][E], accumulated over
 * tokens [t0, t1).  The path implements mode 0; mode 1 is kept so that the
 * reading can be checked against App. C.2 (idle experts receive gradient). */
void oracle_direction_mode(const float *z, const uint8_t *f, int64_t t0, int64_t t1, int32_t E,
                           int32_t gate, int32_t mode, double *C)
{
    double *p = (double *)malloc(sizeof(double) * (size_t)E);
    for (int64_t t = t0; t < t1; ++t) {
        const uint8_t *ft = f + t * E;
        gate_row(z + t * E, E, gate, p);
        if (mode == 1) {
            double kept = 0.0;
            for (int32_t i = 0; i < E; ++i) kept += ft[i] ? p[i] : 0.0;
            for (int32_t i = 0; i < E; ++i) p[i] = ft[i] ? p[i] / kept : 0.0;
        }
        for (int32_t i = 0; i < E; ++i)
            for (int32_t j = 0; j < E; ++j)
                C[(int64_t)i * E + j] += p[i] * ((double)ft[i] - (double)ft[j]);
    }
    free(p);
}

/* Gradient of the combine weights (Sec. 3.1.1: w_tq = p_{e_q,t} / sum_q' p_{e_q',t})
 * to the logits, for an upstream gradient g [T][k] of the weights: with the
 * dense p written out, dz_tl = sum_q g_tq d w_tq / d z_tl for every expert l
 * (the experts not chosen have a zero derivative, the dense normaliser
 * cancelling), computed entry by entry in double:
 *   sigmoid-norm: w_q = s_q / S,  S = sum of the chosen s,
 *                 d w_q / d z_l = [l chosen] s_l (1 - s_l) (delta_ql - w_q) / S,
 *                 with 1 - s_l evaluated as sigmoid(-z_l)
 *   softmax:      w_q = exp(z_q) / sum of the chosen exp(z),
 *                 d w_q / d z_l = [l chosen] w_q (delta_ql - w_l)
 * ids [T][k] are the chosen experts; dz is [T][E]. */
void oracle_route_backward(const float *z, const int32_t *ids, const double *g, int64_t T,
                           int32_t E, int32_t k, int32_t gate, double *dz)
{
    double *w = (double *)malloc(sizeof(double) * (size_t)k);
    double *sv = (double *)malloc(sizeof(double) * (size_t)k);
    for (int64_t t = 0; t < T; ++t) {
        const float *zt = z + t * (int64_t)E;
        const int32_t *it = ids + t * (int64_t)k;
        const double *gt = g + t * (int64_t)k;
        double *dt = dz + t * (int64_t)E;
        for (int32_t l = 0; l < E; ++l) dt[l] = 0.0;
        double S = 0.0, zmax = (double)zt[it[0]];
        for (int32_t q = 0; q < k; ++q)
            if ((double)zt[it[q]] > zmax) zmax = (double)zt[it[q]];
        for (int32_t q = 0; q < k; ++q) {
            double v = (double)zt[it[q]];
            sv[q] = gate == GATE_SOFTMAX ? exp(v - zmax) : 1.0 / (1.0 + exp(-v));
            S += sv[q];
        }
        for (int32_t q = 0; q < k; ++q) w[q] = sv[q] / S;
        for (int32_t m = 0; m < k; ++m) {     /* l = ids[m], a chosen expert */
            double acc = 0.0;
            for (int32_t q = 0; q < k; ++q) {
                double delta = (q == m) ? 1.0 : 0.0;
                /* 1 - sigmoid(v) written as sigmoid(-v): no cancellation for large v */
                double J = gate == GATE_SOFTMAX
                               ? w[q] * (delta - w[m])
                               : sv[m] * (1.0 / (1.0 + exp((double)zt[it[m]]))) * (delta - w[q]) / S;
                acc += gt[q] * J;
            }
            dt[it[m]] = acc;
        }
    }
    free(w);
    free(sv);
}
