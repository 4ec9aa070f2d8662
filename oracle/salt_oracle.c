/*
 * SALT serving-phase oracle: plain, slow, fp64 CPU reference.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path links, loads or
 * calls this file; only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark do.  It shares no code, header, table or helper with the
 * CUDA library: every conversion below is written out here on its own.
 *
 * What it computes (paper, Section "Multi-Tenant Serving"): the final weight
 * of request i is W_final = W_base + gamma * Wbar + delta_i.  With the
 * centroid Wbar = A_c B_c and the residual delta_i = a_u b_u in low-rank form
 * (Section "The Centroid-Residual Decomposition", delta_i = B'_i A'_i read
 * in row-vector convention), one token's LoRA output is
 *
 *   y[t, j] = y_in[t, j]
 *           + [d >= 0] * s_c(d) * sum_k (sum_i x[t,i] A_c[i,k]) B_c[k,j]
 *           + [u >= 0] * s_u(u) * sum_k (sum_i x[t,i] a_u[i,k]) b_u[k,j]
 *
 * where y_in already holds x W_base, or, when a base weight is passed, the
 * base product x W_base is added here as well (y = y_in + x W_final, the
 * whole of W_final = W_base + gamma Wbar + delta_i),
 * d is the token's domain (centroid) and u its residual slot, and -1 drops
 * the term (a token routed out of distribution falls back, Section
 * "Automated Centroid Routing", Stage 1).  A is stored transposed, At[k][i].
 * Every operand is the exact bf16 value widened to double; nothing is
 * rounded until the caller compares.
 *
 * Grouping (Section "Multi-Tenant Serving": requests are grouped by their
 * centroid; heterogeneous batching of residuals as in SGMV, Section
 * "Multi-Tenant LoRA Serving"): tokens are sorted stably by (domain, slot),
 * -1 first, ties kept in token order; a domain segment is a maximal run of
 * equal domain and a user segment a maximal run of equal (domain, slot).
 *
 * gamma (same section): the centroid of a request is scaled by a
 * per-request coefficient taken from a small fixed set of values (bins), and requests are
 * grouped by their (centroid, gamma) pair.  Here gamma is a per-token factor
 * on the centroid term (1 when absent), and the grouping key is
 * (domain, gamma bin, slot); a token without a centroid has no bin.
 *
 * Also here: the alignment regulariser of Phase 1 (Eq. 2), a matrix cosine
 * between a task update Delta W and the centroid Wbar, evaluated from the
 * dense matrices entry by entry; and the fold of a scaled centroid into a
 * base weight (same section: high-frequency centroids are fused into the
 * base weights when a node starts), W + gamma * s_c * A_c B_c entry by entry.
 *
 * All functions here are pinned by tests/test_oracle_pins.py against the
 * dense closed form, the concatenation identity, special cases, invariants,
 * a library sort, a hand-worked example, the paper's printed adapter
 * footprints, rank-one closed forms and dense brute force.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* bf16 is the top 16 bits of an IEEE binary32; widening is exact. */
static double oracle_bf16_value(uint16_t h)
{
    uint32_t bits = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

/*
 * One projection, every listed token.
 *
 * x      [T][d_in]  bf16 bits, row-major
 * y_in   [T][d_out] bf16 bits (may be NULL: zeros)
 * W_base base weight, bf16 bits, [d_in][d_out] (w_layout 0) or [d_out][d_in]
 *        (w_layout 1), or NULL (no base term)
 * dom    [T] centroid index or -1;  slot [T] residual slot or -1
 * gamma  [T] per-token factor on the centroid term (NULL: 1 for every token)
 * For domain d: rc[d] ranks, s_c[d], At_c[d] -> [rc][d_in], B_c[d] -> [rc][d_out]
 * For slot u:   r_u[u] ranks, s_u[u], At_u[u] -> [r][d_in],  B_u[u] -> [r][d_out]
 * rows   [n_rows] token indices to evaluate (NULL: all T tokens in order)
 * y_out  [n_rows][d_out] doubles
 * Returns 0, or -1 on an id outside its table or a w_layout other than 0 / 1.
 */
int oracle_apply(int64_t T, int64_t d_in, int64_t d_out,
                 const uint16_t *x, const uint16_t *y_in, const uint16_t *W_base, int32_t w_layout,
                 const int32_t *dom, const int32_t *slot, const double *gamma,
                 int32_t n_domains, const int32_t *rc, const double *s_c,
                 const uint16_t *const *At_c, const uint16_t *const *B_c,
                 int32_t n_slots, const int32_t *r_u, const double *s_u,
                 const uint16_t *const *At_u, const uint16_t *const *B_u,
                 int64_t n_rows, const int64_t *rows, double *y_out)
{
    int64_t count = rows ? n_rows : T;
    double *v = NULL;
    if (w_layout != 0 && w_layout != 1) return -1;
    int32_t max_rank = 1;
    for (int32_t d = 0; d < n_domains; ++d)
        if (rc[d] > max_rank) max_rank = rc[d];
    for (int32_t u = 0; u < n_slots; ++u)
        if (r_u[u] > max_rank) max_rank = r_u[u];
    v = (double *)malloc(sizeof(double) * (size_t)max_rank);
    if (!v) return -2;

    for (int64_t n = 0; n < count; ++n) {
        int64_t t = rows ? rows[n] : n;
        double *out = y_out + n * d_out;
        const uint16_t *xt = x + t * d_in;
        int32_t d = dom[t], u = slot[t];
        if (t < 0 || t >= T || d < -1 || d >= n_domains || u < -1 || u >= n_slots) {
            free(v);
            return -1;
        }
        for (int64_t j = 0; j < d_out; ++j)
            out[j] = y_in ? oracle_bf16_value(y_in[t * d_out + j]) : 0.0;

        /* base term: x W_base */
        if (W_base) {
            for (int64_t j = 0; j < d_out; ++j) {
                double base = 0.0;
                for (int64_t i = 0; i < d_in; ++i)
                    base += oracle_bf16_value(xt[i]) * oracle_bf16_value(W_base[w_layout ? j * d_in + i : i * d_out + j]);
                out[j] += base;
            }
        }

        /* centroid term: gamma * s_c * (x A_c) B_c */
        if (d >= 0) {
            int32_t R = rc[d];
            double gt = gamma ? gamma[t] : 1.0;
            for (int32_t k = 0; k < R; ++k) {
                double acc = 0.0;
                for (int64_t i = 0; i < d_in; ++i)
                    acc += oracle_bf16_value(xt[i]) * oracle_bf16_value(At_c[d][k * d_in + i]);
                v[k] = acc;
            }
            for (int64_t j = 0; j < d_out; ++j) {
                double acc = 0.0;
                for (int32_t k = 0; k < R; ++k)
                    acc += v[k] * oracle_bf16_value(B_c[d][k * d_out + j]);
                out[j] += gt * s_c[d] * acc;
            }
        }
        /* residual term: s_u * (x a_u) b_u */
        if (u >= 0) {
            int32_t R = r_u[u];
            for (int32_t k = 0; k < R; ++k) {
                double acc = 0.0;
                for (int64_t i = 0; i < d_in; ++i)
                    acc += oracle_bf16_value(xt[i]) * oracle_bf16_value(At_u[u][k * d_in + i]);
                v[k] = acc;
            }
            for (int64_t j = 0; j < d_out; ++j) {
                double acc = 0.0;
                for (int32_t k = 0; k < R; ++k)
                    acc += v[k] * oracle_bf16_value(B_u[u][k * d_out + j]);
                out[j] += s_u[u] * acc;
            }
        }
    }
    free(v);
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Grouping of a heterogeneous batch into domain and user segments.        */

typedef struct {
    int32_t d, g, u, t;
} oracle_key;

static int oracle_key_cmp(const void *pa, const void *pb)
{
    const oracle_key *a = (const oracle_key *)pa, *b = (const oracle_key *)pb;
    if (a->d != b->d) return a->d < b->d ? -1 : 1;
    if (a->g != b->g) return a->g < b->g ? -1 : 1;
    if (a->u != b->u) return a->u < b->u ? -1 : 1;
    if (a->t != b->t) return a->t < b->t ? -1 : 1;
    return 0;
}

/*
 * gbin      [T]      gamma bin of each token, or NULL (no bins); the bin of
 *                    a token without a centroid (dom = -1) is taken as -1
 * perm      [T]      token index of the i-th token in grouped order
 * dseg_ptr  [T + 1]  domain segment i spans [dseg_ptr[i], dseg_ptr[i+1]):
 *                    a maximal run of equal (domain, bin)
 * dseg_dom, dseg_gbin [T]  its (domain, bin)
 * useg_ptr  [T + 1]  user segment i spans [useg_ptr[i], useg_ptr[i+1]):
 *                    a maximal run of equal (domain, bin, slot)
 * useg_dom, useg_gbin, useg_slot [T]  its (domain, bin, slot)
 * counts    [2]      number of domain segments, number of user segments
 */
int oracle_segments(int32_t T, const int32_t *dom, const int32_t *gbin, const int32_t *slot,
                    int32_t *perm, int32_t *dseg_ptr, int32_t *dseg_dom, int32_t *dseg_gbin,
                    int32_t *useg_ptr, int32_t *useg_dom, int32_t *useg_gbin, int32_t *useg_slot,
                    int32_t *counts)
{
    oracle_key *keys;
    int32_t nd = 0, nu = 0;
    if (T < 0) return -1;
    counts[0] = counts[1] = 0;
    if (T == 0) {
        dseg_ptr[0] = 0;
        useg_ptr[0] = 0;
        return 0;
    }
    keys = (oracle_key *)malloc(sizeof(oracle_key) * (size_t)T);
    if (!keys) return -2;
    for (int32_t t = 0; t < T; ++t) {
        keys[t].d = dom[t];
        keys[t].g = (gbin && dom[t] >= 0) ? gbin[t] : -1;
        keys[t].u = slot[t];
        keys[t].t = t;
    }
    qsort(keys, (size_t)T, sizeof(oracle_key), oracle_key_cmp);
    for (int32_t i = 0; i < T; ++i) {
        perm[i] = keys[i].t;
        int new_dom = i == 0 || keys[i].d != keys[i - 1].d || keys[i].g != keys[i - 1].g;
        if (new_dom) {
            dseg_ptr[nd] = i;
            dseg_dom[nd] = keys[i].d;
            dseg_gbin[nd] = keys[i].g;
            ++nd;
        }
        if (new_dom || keys[i].u != keys[i - 1].u) {
            useg_ptr[nu] = i;
            useg_dom[nu] = keys[i].d;
            useg_gbin[nu] = keys[i].g;
            useg_slot[nu] = keys[i].u;
            ++nu;
        }
    }
    dseg_ptr[nd] = T;
    useg_ptr[nu] = T;
    counts[0] = nd;
    counts[1] = nu;
    free(keys);
    return 0;
}

/*
 * Bytes one rank-r adapter occupies over a list of adapted weight matrices
 * (bf16, 2 bytes per parameter): r * sum_l (d_in_l + d_out_l) * 2.  This is
 * the quantity the paper's "Swap" and "Pin" memory columns report (Table 1
 * and the appendix tables for Llama-3.2-3B and Pythia-12B).
 */
int64_t oracle_adapter_bytes(int32_t n_layers, const int32_t *d_in, const int32_t *d_out, int32_t rank)
{
    int64_t params = 0;
    for (int32_t l = 0; l < n_layers; ++l)
        params += (int64_t)rank * ((int64_t)d_in[l] + (int64_t)d_out[l]);
    return params * 2;
}

/* ---------------------------------------------------------------------- */
/* Phase 1 alignment regulariser (Eq. 2).                                  */

/*
 * L_align(Delta W, Wbar) = 1 - Tr(Delta W^T Wbar) / (||Delta W||_F ||Wbar||_F + eps)
 * with Delta W = s * A B (rank r) and Wbar = s_c * A_c B_c (rank rc), both
 * d_in x d_out, the A factors stored transposed (At[k][i]).  Evaluated from
 * the dense matrices: each row i of both is formed in doubles and its
 * entries enter the trace and the two squared norms.
 *
 * out[0] = L_align, out[1] = the cosine term Tr / (norms + eps),
 * out[2] = Tr(Delta W^T Wbar), out[3] = ||Delta W||_F, out[4] = ||Wbar||_F.
 */
int oracle_align_loss(int64_t d_in, int64_t d_out,
                      int32_t r, const uint16_t *At, const uint16_t *B, double s,
                      int32_t rc, const uint16_t *At_c, const uint16_t *B_c, double s_c,
                      double eps, double *out)
{
    double *dw = (double *)malloc(sizeof(double) * (size_t)(d_out > 0 ? d_out : 1));
    double *wb = (double *)malloc(sizeof(double) * (size_t)(d_out > 0 ? d_out : 1));
    double tr = 0.0, nn_dw = 0.0, nn_wb = 0.0;
    if (!dw || !wb) {
        free(dw);
        free(wb);
        return -2;
    }
    for (int64_t i = 0; i < d_in; ++i) {
        /* row i of A B and of A_c B_c, summed over k in ascending order */
        for (int64_t j = 0; j < d_out; ++j) dw[j] = wb[j] = 0.0;
        for (int32_t k = 0; k < r; ++k) {
            double a = oracle_bf16_value(At[k * d_in + i]);
            for (int64_t j = 0; j < d_out; ++j) dw[j] += a * oracle_bf16_value(B[k * d_out + j]);
        }
        for (int32_t k = 0; k < rc; ++k) {
            double c = oracle_bf16_value(At_c[k * d_in + i]);
            for (int64_t j = 0; j < d_out; ++j) wb[j] += c * oracle_bf16_value(B_c[k * d_out + j]);
        }
        for (int64_t j = 0; j < d_out; ++j) {
            dw[j] *= s;
            wb[j] *= s_c;
        }
        for (int64_t j = 0; j < d_out; ++j) {
            tr += dw[j] * wb[j];
            nn_dw += dw[j] * dw[j];
            nn_wb += wb[j] * wb[j];
        }
    }
    free(dw);
    free(wb);
    {
        double n_dw = sqrt(nn_dw), n_wb = sqrt(nn_wb);
        double cosine = tr / (n_dw * n_wb + eps);
        out[0] = 1.0 - cosine;
        out[1] = cosine;
        out[2] = tr;
        out[3] = n_dw;
        out[4] = n_wb;
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Fold of a scaled centroid into a base weight.                          */

/*
 * W_out = W + scale * A_c B_c entry by entry, in doubles (scale = gamma * s_c).
 * layout 0: W is [d_in][d_out] (y = x W, the row-vector convention above);
 * layout 1: W is [d_out][d_in] (y = x W^T, the weight of a linear layer).
 * W holds bf16 bits; W_out gets the unrounded doubles in W's layout.
 */
int oracle_fold(int64_t d_in, int64_t d_out, int32_t rc, const uint16_t *At_c, const uint16_t *B_c,
                double scale, const uint16_t *W, int32_t layout, double *W_out)
{
    double *row = (double *)malloc(sizeof(double) * (size_t)(d_out > 0 ? d_out : 1));
    if (layout != 0 && layout != 1) {
        free(row);
        return -1;
    }
    if (!row) return -2;
    for (int64_t i = 0; i < d_in; ++i) {
        /* row i of A_c B_c, summed over k in ascending order */
        for (int64_t j = 0; j < d_out; ++j) row[j] = 0.0;
        for (int32_t k = 0; k < rc; ++k) {
            double a = oracle_bf16_value(At_c[k * d_in + i]);
            for (int64_t j = 0; j < d_out; ++j) row[j] += a * oracle_bf16_value(B_c[k * d_out + j]);
        }
        for (int64_t j = 0; j < d_out; ++j) {
            int64_t idx = layout ? j * d_in + i : i * d_out + j;
            W_out[idx] = oracle_bf16_value(W[idx]) + scale * row[j];
        }
    }
    free(row);
    return 0;
}
