/*
 * accept.c -- oracle for source-aware verification, longest-path selection
 * and the EMA feedback update.
 *
 * TEST INFRASTRUCTURE ONLY (see rsref.h).
 *
 * Follows:
 *   - Section 3.4: strict verification of model drafts (greedy decoding, as
 *     in the experiments of Section 4.1: a draft token is accepted iff it is
 *     the argmax of its parent's distribution and its parent is accepted);
 *     relaxed verification of retrieved drafts (Eq. 6: the token is among the
 *     beta most likely tokens; Eq. 7: log p(x1) - log p(x~) <= tau) and the
 *     look-ahead tolerance procedure;
 *   - Algorithm 1 (verification): the longest accepted path over all branches gives
 *     X_accepted and the winning position;
 *   - Eq. 4-5 and Algorithm 1's score update: S_p <- (1-alpha) S_p + alpha R_p with
 *     R_p = L_accepted / L_draft for the winner and 0 for every other
 *     selected position.
 *
 * Readings (the paper is silent or garbled there):
 *   - argmax takes the lowest token id among equal maxima; TopK_beta is the
 *     first beta ids in (logit desc, id asc) order;
 *   - Eq. 7's difference of log-probabilities equals the difference of the
 *     two logits (the softmax normaliser cancels); it is evaluated as that
 *     logit gap in fp64;
 *   - look-ahead: starting at the first greedy mismatch l0 (cur = last = l0),
 *     each of at most phi attempts stops the procedure if the token at cur
 *     fails the relaxed check; otherwise it counts the consecutive greedy
 *     matches xi that FOLLOW cur; if xi >= m the acceptance extends over the
 *     relaxed token and those matches (last = cur + 1 + xi, cur = last),
 *     else cur advances by one.  The accepted length is last.  This reading
 *     is parity unpinned against the paper, which prints no worked example
 *     of the procedure; the tests pin it to hand-worked cases of the reading
 *     and to its closed special cases (phi = 0, beta = 1 or tau = 0 reduce
 *     it to strict verification; an all-greedy chain is accepted whole);
 *   - the winner is the longest accepted path; ties go to the model tree,
 *     then to the chain that was selected first; all zero -> no winner;
 *   - the bonus token is the argmax of the last accepted node's row (the
 *     root's row when nothing was accepted);
 *   - the score table is stored in fp32; the update is evaluated in fp64 and
 *     rounded once.
 */
#include <math.h>
#include <stdlib.h>
#include "rsref.h"

static double lse_row(const float *z, long V)
{
    double m = -INFINITY;
    for (long v = 0; v < V; ++v)
        if ((double)z[v] > m) m = (double)z[v];
    if (m == -INFINITY) return -INFINITY;
    double s = 0.0;
    for (long v = 0; v < V; ++v) s += exp((double)z[v] - m);
    return m + log(s);
}

/* true when (za, a) comes before (zb, b) in (logit desc, id asc) order */
static int before(float za, long a, float zb, long b)
{
    if (za > zb) return 1;
    if (za < zb) return 0;
    return a < b;
}

/* TopK_beta: beta selection passes, each taking the best id not yet taken */
static void topk_row(const float *z, long V, int beta, int *out)
{
    for (int j = 0; j < beta; ++j) {
        long best = -1;
        for (long v = 0; v < V; ++v) {
            int taken = 0;
            for (int i = 0; i < j; ++i)
                if (out[i] == (int)v) { taken = 1; break; }
            if (taken) continue;
            if (best < 0 || before(z[v], v, z[best], best)) best = v;
        }
        out[j] = (int)best; /* -1 once the row has fewer than beta ids */
    }
}

void rsref_accept(const float *logits, long V, const int *node_off, int B,
                  const int *tokens, const int *parents,
                  const unsigned char *source, const signed char *chain,
                  const int *sel_pos, int top_c, const long *tok_off,
                  int beta, double tau, int phi, int m, double alpha,
                  int acc_cap,
                  int *argmax, int *topk, double *lse, double *p_tok,
                  int *acc_len, int *acc_nodes, int *bonus, int *winner,
                  unsigned char *commit, float *scores, int *status)
{
    long R = node_off[B];

    /* ---- per-row statistics ---- */
    for (long r = 0; r < R; ++r) {
        const float *z = logits + r * V;
        topk_row(z, V, beta, topk + r * beta);
        argmax[r] = topk[r * beta]; /* first in (logit desc, id asc) order */
        lse[r] = lse_row(z, V);
    }

    for (int b = 0; b < B; ++b) {
        int n0 = node_off[b];
        int N = node_off[b + 1] - n0;
        const int *par = parents + n0;
        const int *tok = tokens + n0;
        const unsigned char *src = source + n0;
        const signed char *chn = chain + n0;

        status[b] = 0;
        acc_len[b] = 0;
        winner[b] = -2;
        bonus[b] = -1;
        for (int j = 0; j < acc_cap; ++j) acc_nodes[(long)b * acc_cap + j] = -1;
        for (int i = 0; i < N; ++i) { commit[n0 + i] = 0; p_tok[n0 + i] = 0.0; }

        /* ---- tree layout check ---- */
        int bad = (N < 1);
        int *last_of = (int *)malloc(sizeof(int) * (size_t)(top_c > 0 ? top_c : 1));
        for (int c = 0; c < top_c; ++c) last_of[c] = -1;
        if (!bad && (par[0] != -1 || src[0] != 0 || chn[0] != -1)) bad = 1;
        for (int i = 1; i < N && !bad; ++i) {
            int p = par[i];
            if (p < 0 || p >= i) { bad = 1; break; }
            if (tok[i] < 0 || (long)tok[i] >= V) { bad = 1; break; } /* not a vocabulary id */
            if (src[i] == 1) {
                if (src[p] > 1 || chn[i] != -1) bad = 1;
            } else if (src[i] == 2) {
                int c = chn[i];
                if (c < 0 || c >= top_c) { bad = 1; break; }
                if (p != (last_of[c] < 0 ? 0 : last_of[c])) bad = 1;
                last_of[c] = i;
            } else {
                bad = 1;
            }
        }
        free(last_of);
        if (bad) { status[b] |= RSREF_ST_BAD_TREE; continue; }

        /* probability of each node's token under its parent's row */
        p_tok[n0] = 1.0;
        for (int i = 1; i < N; ++i) {
            long pr = n0 + par[i];
            p_tok[n0 + i] = exp((double)logits[pr * V + tok[i]] - lse[pr]);
        }

        /* ---- strict verification of the model subtree ---- */
        unsigned char *acc = (unsigned char *)calloc((size_t)N, 1);
        int *depth = (int *)calloc((size_t)N, sizeof(int));
        acc[0] = 1;
        int best_model = 0, model_len = 0;
        for (int i = 1; i < N; ++i) {
            if (src[i] != 1) continue;
            int p = par[i];
            depth[i] = depth[p] + 1;
            acc[i] = acc[p] && tok[i] == argmax[n0 + p];
            if (acc[i] && depth[i] > model_len) { model_len = depth[i]; best_model = i; }
        }

        /* ---- relaxed verification with look-ahead tolerance, per chain ---- */
        int *chain_len = (int *)calloc((size_t)(top_c > 0 ? top_c : 1), sizeof(int));
        int *chain_acc = (int *)calloc((size_t)(top_c > 0 ? top_c : 1), sizeof(int));
        int *d = (int *)malloc(sizeof(int) * (size_t)N);
        for (int c = 0; c < top_c; ++c) {
            int L = 0;
            for (int i = 1; i < N; ++i)
                if (src[i] == 2 && chn[i] == c) d[L++] = i;
            chain_len[c] = L;
            if (L == 0) continue;

            /* g(j): greedy match; rx(j): Eq. 6 and Eq. 7 */
#define G_(j) (tok[d[j]] == argmax[n0 + par[d[j]]])
            int l0 = 0;
            while (l0 < L && G_(l0)) ++l0;
            int cur = l0, last = l0;
            for (int attempt = 0; attempt < phi; ++attempt) {
                if (cur >= L) break;
                long row = n0 + par[d[cur]];
                int x = tok[d[cur]];
                int in_top = 0;
                for (int j = 0; j < beta; ++j)
                    if (topk[row * beta + j] == x) in_top = 1;
                double gap = (double)logits[row * V + argmax[row]] - (double)logits[row * V + x];
                if (!(in_top && gap <= tau)) break; /* relaxed-verify failure ends it */
                int xi = 0;
                while (cur + 1 + xi < L && G_(cur + 1 + xi)) ++xi;
                if (xi >= m) { last = cur + 1 + xi; cur = last; }
                else { cur = cur + 1; }
            }
#undef G_
            chain_acc[c] = last;
        }

        /* ---- longest accepted path and its winner ---- */
        int best_len = model_len, win = model_len > 0 ? -1 : -2;
        for (int c = 0; c < top_c; ++c)
            if (chain_acc[c] > best_len) { best_len = chain_acc[c]; win = c; }
        if (best_len == 0) win = -2;

        int *path = (int *)malloc(sizeof(int) * (size_t)(best_len > 0 ? best_len : 1));
        if (win == -1) {
            int a = best_model;
            for (int j = best_len - 1; j >= 0; --j) { path[j] = a; a = par[a]; }
        } else if (win >= 0) {
            int L = 0;
            for (int i = 1; i < N && L < best_len; ++i)
                if (src[i] == 2 && chn[i] == win) path[L++] = i;
        }
        acc_len[b] = best_len;
        winner[b] = win;
        if (best_len > acc_cap) status[b] |= RSREF_ST_TRUNCATED;
        for (int j = 0; j < best_len && j < acc_cap; ++j) acc_nodes[(long)b * acc_cap + j] = path[j];
        int last_node = best_len > 0 ? path[best_len - 1] : 0;
        bonus[b] = argmax[n0 + last_node];
        commit[n0] = 1;
        for (int j = 0; j < best_len; ++j) commit[n0 + path[j]] = 1;

        /* ---- EMA update of the selected positions (Eq. 4-5) ---- */
        long t = tok_off[b + 1] - tok_off[b];
        for (int c = 0; c < top_c; ++c) {
            int p = sel_pos[b * top_c + c];
            if (p < 0 || chain_len[c] == 0) continue;
            if ((long)p >= t) { status[b] |= RSREF_ST_BAD_POS; continue; }
            double Rp = (win == c) ? (double)chain_acc[c] / (double)chain_len[c] : 0.0;
            float *S = scores + tok_off[b] + p;
            double upd = (1.0 - alpha) * (double)(*S) + alpha * Rp;
            *S = (float)upd;
        }

        free(path);
        free(d);
        free(chain_len);
        free(chain_acc);
        free(acc);
        free(depth);
    }
}
