/*
 * entropy.c -- oracle for the entropy-guided adaptive trigger.
 *
 * TEST INFRASTRUCTURE ONLY (see rsref.h).
 *
 * Follows Section 3.2.1: Eq. 1 (mean predictive entropy of a suffix key),
 * Eq. 2 (confidence score C_k = H_k + lambda_e / k), Eq. 3 (k* = argmin C_k)
 * and the trigger decision (trigger iff H_{k*} <= theta_entropy), in the
 * order Algorithm 1's entropy-guided triggering evaluates them: k runs
 * upward from 1 and a later k replaces the
 * current best only when its C_k is strictly smaller.
 */
#include <math.h>
#include <stdlib.h>
#include "rsref.h"

/* Eq. 1, inner term: -sum_v P(v) log P(v) with P = softmax(z), in nats.
 * P is formed explicitly; a zero probability contributes nothing (the
 * limit of p log p at 0). */
double rsref_row_entropy(const float *z, long V)
{
    double zmax = -INFINITY;
    for (long v = 0; v < V; ++v)
        if ((double)z[v] > zmax) zmax = (double)z[v];
    if (zmax == -INFINITY) return 0.0; /* every logit -inf: degenerate row */

    double s = 0.0; /* softmax normaliser, relative to zmax */
    for (long v = 0; v < V; ++v) s += exp((double)z[v] - zmax);

    double h = 0.0;
    for (long v = 0; v < V; ++v) {
        double p = exp((double)z[v] - zmax) / s;
        if (p > 0.0) h -= p * log(p);
    }
    return h;
}

void rsref_entropy_rows(const float *logits, long R, long V, double *H)
{
    for (long r = 0; r < R; ++r) H[r] = rsref_row_entropy(logits + r * V, V);
}

/* Section 3.2.1 (entropy, confidence score, key selection, trigger decision)
 * over the per-request entropy history.
 * The history holds one entropy per committed token: the entropy of the
 * distribution that predicted it (the verify step's root row and the rows
 * of its accepted nodes), oldest first. */
void rsref_gate(const double *H, const long *row_off, const unsigned char *row_commit,
                int B, int l, double lambda_e, double theta,
                double *hist, int *hist_n,
                int *k_star, double *h_best, unsigned char *ok)
{
    for (int b = 0; b < B; ++b) {
        double *hb = hist + (long)b * l;
        int n = hist_n[b];
        if (n < 0) n = 0;
        if (n > l) n = l;

        /* append the committed rows' entropies, dropping the oldest */
        for (long r = row_off[b]; r < row_off[b + 1]; ++r) {
            if (!row_commit[r]) continue;
            if (n == l) {
                for (int i = 1; i < l; ++i) hb[i - 1] = hb[i];
                hb[l - 1] = H[r];
            } else {
                hb[n++] = H[r];
            }
        }
        hist_n[b] = n;

        /* Algorithm 1, entropy-guided triggering */
        double c_min = INFINITY, best = INFINITY;
        int kbest = 0;
        int kmax = n < l ? n : l;
        for (int k = 1; k <= kmax; ++k) {
            /* Eq. 1: mean over the newest k entries, summed oldest to newest */
            double s = 0.0;
            for (int i = n - k; i < n; ++i) s += hb[i];
            double hk = s / (double)k;
            double ck = hk + lambda_e / (double)k; /* Eq. 2 */
            if (ck < c_min) {                      /* Eq. 3, strict: ties keep the smaller k */
                c_min = ck;
                best = hk;
                kbest = k;
            }
        }
        k_star[b] = kbest;
        h_best[b] = best;
        ok[b] = (unsigned char)(kbest > 0 && best <= theta); /* trigger decision */
    }
}
