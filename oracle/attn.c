/*
 * attn.c -- oracle for tree-verification attention.
 *
 * TEST INFRASTRUCTURE ONLY (see rsref.h).
 *
 * The paper verifies the packed draft tree with one target forward
 * ("parallel verification", Section 3.3; both verifications of Algorithm 1) but does
 * not spell out the attention.  The standard reading is used: each tree node
 * attends to the whole committed prefix and to the tree slots of its
 * ancestors and itself (the draft tokens on its own root-to-node path), with
 * scaled dot-product softmax attention; grouped-query heads share a KV head
 * (KV head = q head / (Hq/Hkv)).
 *
 * Written out per (node, head): one score per allowed key, one softmax, one
 * weighted sum of values, all in fp64.
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#include "rsref.h"

/* bf16 bit pattern -> double (exact) */
static double bf16_to_double(unsigned short h)
{
    unsigned int u = (unsigned int)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

int rsref_tree_attn(const unsigned short *q, const unsigned short *k,
                    const unsigned short *v, const long *kv_off,
                    const int *ctx_len, const int *node_off,
                    const int *parents, int B, int Hq, int Hkv, int D,
                    double scale, long n_rows, const long *row_node,
                    const int *row_head, double *out, double *lse)
{
    int G = Hq / Hkv;
    int rc = 0;
    for (long n = 0; n < n_rows; ++n) {
        long r = row_node[n];
        int h = row_head[n];
        int b = 0;
        while (b < B && !(node_off[b] <= r && r < node_off[b + 1])) ++b;
        double *o = out + n * D;
        for (int d = 0; d < D; ++d) o[d] = 0.0;
        lse[n] = NAN;
        if (b == B) { rc = 1; continue; }

        int N = node_off[b + 1] - node_off[b];
        int i = (int)(r - node_off[b]);
        const int *par = parents + node_off[b];
        long S = ctx_len[b];
        int kvh = h / G;

        /* ancestors-or-self of node i, by walking the parent links */
        unsigned char *on_path = (unsigned char *)calloc((size_t)N, 1);
        int bad = 0, a = i, steps = 0;
        while (a != -1) {
            if (a < 0 || a >= N || steps > N) { bad = 1; break; }
            on_path[a] = 1;
            int pa = par[a];
            if (a == 0 ? pa != -1 : (pa < 0 || pa >= a)) { bad = 1; break; }
            a = pa;
            ++steps;
        }
        if (bad) { free(on_path); rc = 1; continue; }

        /* allowed key slots: prefix 0..S-1, then S+a for a on the path */
        long nkeys = S;
        for (int j = 0; j < N; ++j) nkeys += on_path[j];
        long *slot = (long *)malloc(sizeof(long) * (size_t)(nkeys > 0 ? nkeys : 1));
        double *s = (double *)malloc(sizeof(double) * (size_t)(nkeys > 0 ? nkeys : 1));
        long c = 0;
        for (long j = 0; j < S; ++j) slot[c++] = j;
        for (int j = 0; j < N; ++j)
            if (on_path[j]) slot[c++] = S + j;

        const unsigned short *qr = q + ((long)r * Hq + h) * D;
        double smax = -INFINITY;
        for (long j = 0; j < nkeys; ++j) {
            const unsigned short *kr = k + ((kv_off[b] + slot[j]) * Hkv + kvh) * D;
            double dot = 0.0;
            for (int d = 0; d < D; ++d) dot += bf16_to_double(qr[d]) * bf16_to_double(kr[d]);
            s[j] = scale * dot;
            if (s[j] > smax) smax = s[j];
        }
        double z = 0.0;
        for (long j = 0; j < nkeys; ++j) z += exp(s[j] - smax);
        for (long j = 0; j < nkeys; ++j) {
            double p = exp(s[j] - smax) / z;
            const unsigned short *vr = v + ((kv_off[b] + slot[j]) * Hkv + kvh) * D;
            for (int d = 0; d < D; ++d) o[d] += p * bf16_to_double(vr[d]);
        }
        lse[n] = smax + log(z);
        free(slot);
        free(s);
        free(on_path);
    }
    return rc;
}
