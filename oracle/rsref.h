/*
 * rsref.h -- plain, slow CPU oracle for the ReSpec verify-and-draft step
 * (arXiv 2511.01282, "When, What, and How: Rethinking Retrieval-Enhanced
 * Speculative Decoding").
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load this library.  The product path
 * (the CUDA library in the package) never calls it, links it or shares a
 * line of code with it.
 *
 * Every quantity is computed in fp64 from the fp32 / bf16 inputs (both convert
 * to double exactly), straight from the paper's definitions, one request,
 * one row, one head at a time.  No blocking, fusion or reordering beyond what
 * a definition states.
 *
 * Conventions shared with the product ABI (restated here, not included):
 *   - row_off / node_off / tok_off are [B+1] prefix offsets;
 *   - tree node 0 of a request is its root (last committed token),
 *     parents[i] < i (local indices), parents[0] = -1;
 *   - source: 0 root, 1 model draft, 2 retrieved draft; chain: retrieved
 *     chain id (0..top_c-1) or -1;
 *   - the logits row of node i is the target's distribution for the token
 *     that follows node i.
 */
#ifndef RSREF_H
#define RSREF_H

#ifdef __cplusplus
extern "C" {
#endif

/* per-request status bits written by the oracle (same meaning as the
 * product's status word; the values are restated, not shared) */
#define RSREF_ST_BAD_TREE   1  /* parents / source / chain layout invalid      */
#define RSREF_ST_TRUNCATED  2  /* an output list was longer than its capacity  */
#define RSREF_ST_BAD_POS    4  /* a selected position lies outside the buffer  */

/* ---- Section 3.2.1, Eq. 1 (inner term) -------------------------------- */
/* Shannon entropy, in nats, of softmax(z) over one row of V logits. */
double rsref_row_entropy(const float *z, long V);

/* H[r] = rsref_row_entropy(logits + r*V, V) for r < R. */
void rsref_entropy_rows(const float *logits, long R, long V, double *H);

/* ---- Section 3.2.1, Eq. 1-3; Algorithm 1's entropy-guided triggering -- */
/* Pushes the entropies of the committed rows (row_commit[r] != 0, in row
 * order) of each request into its history (hist[b*l .. b*l+l-1], oldest
 * first, hist_n[b] valid entries, the newest at index hist_n[b]-1), then
 * evaluates H_k (mean of the newest k entries), C_k = H_k + lambda_e/k for
 * k = 1..min(l, hist_n), k* = first strict minimum of C_k, and
 * ok = (k* > 0 and H_{k*} <= theta). k* = 0 and h_best = +inf when the
 * history is empty. */
void rsref_gate(const double *H, const long *row_off, const unsigned char *row_commit,
                int B, int l, double lambda_e, double theta,
                double *hist, int *hist_n,
                int *k_star, double *h_best, unsigned char *ok);

/* ---- Section 3.3 (retrieval, filtering, top-3); Algorithm 1 retrieval -- */
/* For request b with key length k = k_star[b] (skipped when k <= 0, or when
 * gate_ok is given and gate_ok[b] == 0): every buffer index p with
 * k-1 <= p <= t-2 whose trailing k tokens equal the buffer's last k tokens,
 * ascending (count[b] = how many; pos[b*pos_cap ..] = the first pos_cap).
 * Of those, positions with scores[p] >= theta_score, ordered by
 * (score desc, p desc), the first top_c are selected; each selected p
 * yields the continuation tokens[p+1 .. min(p+span_len, t-1)].
 * Returns 0. */
int rsref_match_scan(const int *tokens, const long *tok_off, int B,
                     const int *k_star, const unsigned char *gate_ok,
                     const float *scores, double theta_score,
                     int top_c, int span_len, int pos_cap,
                     int *count, int *pos, int *sel_pos, int *sel_len,
                     int *spans, int *n_sel, int *status);

/* ---- Tree-verification attention (the verify forward of Algorithm 1) -- */
/* For each requested (global node r, q-head h): request b owns r; the keys
 * are every prefix slot j < ctx_len[b] and the tree slot ctx_len[b]+a of
 * every ancestor-or-self a of the node; K/V rows live at kv_off[b] + slot.
 * out[n*D ..] = sum_j softmax_j(scale * q.k_j) v_j, lse[n] = log sum_j
 * exp(scale * q.k_j).  q, k, v are bf16 bit patterns.  KV head = h / (Hq/Hkv).
 * Returns 0, or 1 if a node's parent chain is malformed. */
int rsref_tree_attn(const unsigned short *q, const unsigned short *k,
                    const unsigned short *v, const long *kv_off,
                    const int *ctx_len, const int *node_off,
                    const int *parents, int B, int Hq, int Hkv, int D,
                    double scale, long n_rows, const long *row_node,
                    const int *row_head, double *out, double *lse);

/* ---- Section 3.4 (Eq. 6-7, look-ahead tolerance), Eq. 4-5, Algorithm 1 */
/* Row statistics for every node row, then per request: strict acceptance of
 * model drafts, relaxed acceptance with look-ahead for retrieved chains,
 * longest accepted path, winner, bonus token, commit flags and the EMA
 * update of the selected positions' scores (in place, fp32 storage). */
void rsref_accept(const float *logits, long V, const int *node_off, int B,
                  const int *tokens, const int *parents,
                  const unsigned char *source, const signed char *chain,
                  const int *sel_pos, int top_c, const long *tok_off,
                  int beta, double tau, int phi, int m, double alpha,
                  int acc_cap,
                  int *argmax, int *topk, double *lse, double *p_tok,
                  int *acc_len, int *acc_nodes, int *bonus, int *winner,
                  unsigned char *commit, float *scores, int *status);

/* ---- Section 3.4, drafter outputs: lossless speculative sampling ------- */
/* The draw from one row at temperature T > 0 for a uniform u in [0, 1): the
 * smallest token id v with sum_{w <= v} p_T(w) > u, where p_T = softmax(z/T)
 * (the inverse CDF in token-id order).  Rows without mass give 0. */
int rsref_sample_row(const float *z, long V, double T, double u);

/* draw[r] = rsref_sample_row(row r, u[r]) for every node row; then per
 * request, from the root: while a model child (source 1) of the current node
 * carries the current node's draw, accept it (acc_nodes, in depth order) and
 * move to it; the first draw without such a child is the correction token
 * (bonus).  acc_len counts every accepted node (TRUNCATED when more than
 * acc_cap); a malformed tree gives BAD_TREE, acc_len 0, bonus -1. */
void rsref_tree_sample(const float *logits, long V, const int *node_off, int B,
                       const int *tokens, const int *parents,
                       const unsigned char *source, double T, const double *u,
                       int acc_cap, int *draw, int *acc_len, int *acc_nodes,
                       int *bonus, int *status);

#ifdef __cplusplus
}
#endif
#endif
