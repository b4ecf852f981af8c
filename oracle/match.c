/*
 * match.c -- oracle for retrieval and feedback-driven candidate selection.
 *
 * TEST INFRASTRUCTURE ONLY (see rsref.h).
 *
 * Follows Section 3.3 ("Selection Algorithm": retrieve every match position
 * of the key, drop those whose score is below theta_score, keep the top
 * candidates by score) and Algorithm 1's retrieval (Contains / RetrievePositions /
 * quality filter S_p >= theta_score / SelectTopK).  The suffix automaton of
 * the paper is an index over the same position set; here the set is found by
 * comparing the key with every window of the buffer.
 *
 * Readings (the paper leaves these open):
 *   - a position p is the buffer index of the LAST token of an earlier
 *     occurrence of the key; the trailing occurrence itself (p = t-1) is not
 *     a match; overlapping occurrences are all matches;
 *   - equal scores are ordered most recent first (larger p first);
 *   - the continuation of p is tokens[p+1 .. p+span_len], cut at the end of
 *     the buffer (so it is never empty, because p <= t-2).
 */
#include <stdlib.h>
#include "rsref.h"

typedef struct { float s; int p; } cand_t;

/* (score desc, position desc) */
static int cand_cmp(const void *a, const void *b)
{
    const cand_t *x = (const cand_t *)a, *y = (const cand_t *)b;
    if (x->s > y->s) return -1;
    if (x->s < y->s) return 1;
    if (x->p > y->p) return -1;
    if (x->p < y->p) return 1;
    return 0;
}

int rsref_match_scan(const int *tokens, const long *tok_off, int B,
                     const int *k_star, const unsigned char *gate_ok,
                     const float *scores, double theta_score,
                     int top_c, int span_len, int pos_cap,
                     int *count, int *pos, int *sel_pos, int *sel_len,
                     int *spans, int *n_sel, int *status)
{
    for (int b = 0; b < B; ++b) {
        const int *X = tokens + tok_off[b];
        const float *S = scores + tok_off[b];
        long t = tok_off[b + 1] - tok_off[b];
        int k = k_star[b];

        count[b] = 0;
        n_sel[b] = 0;
        status[b] = 0;
        for (int i = 0; i < pos_cap; ++i) pos[(long)b * pos_cap + i] = -1;
        for (int c = 0; c < top_c; ++c) {
            sel_pos[b * top_c + c] = -1;
            sel_len[b * top_c + c] = 0;
            for (int j = 0; j < span_len; ++j)
                spans[((long)b * top_c + c) * span_len + j] = -1;
        }
        if (k <= 0) continue;
        if (gate_ok && !gate_ok[b]) continue;
        if ((long)k > t) continue; /* the key itself does not fit */

        /* RetrievePositions: every p in [k-1, t-2] whose window matches */
        cand_t *cand = (cand_t *)malloc(sizeof(cand_t) * (size_t)(t > 0 ? t : 1));
        int nf = 0;
        int cnt = 0;
        for (long p = k - 1; p <= t - 2; ++p) {
            int match = 1;
            for (int i = 0; i < k; ++i)
                if (X[p - k + 1 + i] != X[t - k + i]) { match = 0; break; }
            if (!match) continue;
            if (cnt < pos_cap) pos[(long)b * pos_cap + cnt] = (int)p;
            ++cnt;
            if ((double)S[p] >= theta_score) { /* quality filter (Algorithm 1) */
                cand[nf].s = S[p];
                cand[nf].p = (int)p;
                ++nf;
            }
        }
        count[b] = cnt;
        if (cnt > pos_cap) status[b] |= RSREF_ST_TRUNCATED;

        /* SelectTopK: best scores first, ties to the most recent position */
        qsort(cand, (size_t)nf, sizeof(cand_t), cand_cmp);
        int ns = nf < top_c ? nf : top_c;
        for (int c = 0; c < ns; ++c) {
            int p = cand[c].p;
            long len = t - 1 - p;
            if (len > span_len) len = span_len;
            sel_pos[b * top_c + c] = p;
            sel_len[b * top_c + c] = (int)len;
            for (long j = 0; j < len; ++j)
                spans[((long)b * top_c + c) * span_len + j] = X[p + 1 + j];
        }
        n_sel[b] = ns;
        free(cand);
    }
    return 0;
}
