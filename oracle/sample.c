/*
 * sample.c -- lossless verification of model-drafted tree nodes by sampling
 * (Section 3.4, "For Drafter Module outputs": standard lossless speculative
 * sampling).  TEST INFRASTRUCTURE ONLY (see rsref.h).
 *
 * Reading.  The draft tree's model children are deterministic expansions of
 * their parent (a point-mass proposal per child).  Speculative sampling's
 * acceptance min(1, p(x)/q(x)) with such proposals, applied to the siblings
 * in turn with the residual renormalised after each rejection, emits a token
 * with exactly the target law p_T; its outcome has the same law as: draw
 * y ~ p_T( . | node); if a model child of the node carries token y, accept it
 * and continue from it, otherwise y is the correction token and the walk
 * stops.  The oracle states that form directly.
 *
 * The row law at temperature T > 0 is p_T(v) = exp((z_v - max z) / T) / Z,
 * and the draw for a uniform u in [0, 1) is the smallest token id v with
 * sum_{w <= v} p_T(w) > u (the inverse of the CDF taken in token-id order),
 * all in fp64.
 */
#include <math.h>

#include "rsref.h"

int rsref_sample_row(const float *z, long V, double T, double u)
{
    double m = -INFINITY;
    for (long v = 0; v < V; ++v)
        if ((double)z[v] > m) m = (double)z[v];
    if (m == -INFINITY) return 0; /* no mass anywhere: the first id */

    double Z = 0.0;
    for (long v = 0; v < V; ++v) Z += exp(((double)z[v] - m) / T);

    const double target = u * Z; /* CDF(v) > u  <=>  partial sum > u Z */
    double c = 0.0;
    long last = 0;
    for (long v = 0; v < V; ++v) {
        const double e = exp(((double)z[v] - m) / T);
        if (e > 0.0) last = v;
        c += e;
        if (c > target) return (int)v;
    }
    return (int)last; /* rounding left u Z at the total: the last id with mass */
}

void rsref_tree_sample(const float *logits, long V, const int *node_off, int B,
                       const int *tokens, const int *parents,
                       const unsigned char *source, double T, const double *u,
                       int acc_cap, int *draw, int *acc_len, int *acc_nodes,
                       int *bonus, int *status)
{
    for (int b = 0; b < B; ++b) {
        const int n0 = node_off[b], N = node_off[b + 1] - n0;

        for (int i = 0; i < N; ++i)
            draw[n0 + i] = rsref_sample_row(logits + (long)(n0 + i) * V, V, T, u[n0 + i]);

        int bad = N < 1;
        for (int i = 0; i < N && !bad; ++i) {
            if (i == 0)
                bad = parents[n0] != -1 || source[n0] != 0;
            else
                bad = parents[n0 + i] < 0 || parents[n0 + i] >= i ||
                      source[n0 + i] < 1 || source[n0 + i] > 2;
        }
        for (int j = 0; j < acc_cap; ++j) acc_nodes[(long)b * acc_cap + j] = -1;
        if (bad) {
            acc_len[b] = 0;
            bonus[b] = -1;
            status[b] = RSREF_ST_BAD_TREE;
            continue;
        }

        /* walk: from the root, follow the model child that carries the draw */
        int cur = 0, len = 0;
        for (;;) {
            const int y = draw[n0 + cur];
            int next = -1;
            for (int i = 1; i < N; ++i)
                if (source[n0 + i] == 1 && parents[n0 + i] == cur && tokens[n0 + i] == y) {
                    next = i;
                    break;
                }
            if (next < 0) {
                bonus[b] = y;
                break;
            }
            if (len < acc_cap) acc_nodes[(long)b * acc_cap + len] = next;
            ++len;
            cur = next;
        }
        acc_len[b] = len;
        status[b] = len > acc_cap ? RSREF_ST_TRUNCATED : 0;
    }
}
