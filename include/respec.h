/*
 * respec.h -- C ABI of the GB300 (sm_103a) verify-and-draft hot path of
 * ReSpec (arXiv 2511.01282, "When, What, and How: Rethinking
 * Retrieval-Enhanced Speculative Decoding").
 *
 * One decoding step of Algorithm 1, as four calls:
 *
 *   rs_entropy_gate     Section 3.2.1, Eq. 1-3, trigger decision (Alg. 1 triggering)
 *   rs_match_scan       Section 3.3 retrieval + selection   (Alg. 1 retrieval)
 *   rs_tree_verify_attn tree attention of the verify pass   (Alg. 1 verification)
 *   rs_accept           Section 3.4 verification, Eq. 4-5  (Alg. 1 verify + EMA)
 *
 * General rules (every entry point):
 *   - All array arguments are DEVICE pointers owned by the caller, unless a
 *     comment says otherwise.  The library allocates nothing: scratch space
 *     comes from the caller's `workspace`, at least rs_*_workspace_size()
 *     bytes, 256-byte aligned; its contents need not be initialised and are
 *     garbage after the call.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Calls only enqueue kernels on it: they never synchronise and
 *     never copy to or from the host, so they can be captured in a CUDA graph.
 *     Calls that share a workspace must be ordered on one stream.
 *   - Arguments that the host can check (sizes, null pointers, parameter
 *     ranges, alignment) are checked before anything is launched; a failure
 *     returns a non-zero rs_status and rs_last_error() describes it.
 *   - Errors that depend on device data (a malformed tree, a capacity
 *     overflow) never trap: they set bits of the caller's per-request
 *     int32 `status` word (each call OVERWRITES status[b] with its own bits,
 *     0 when the request is fine) and the request's decision outputs are set
 *     to their empty values.
 *   - Offsets arrays are prefix sums with B+1 entries (offset[0] = 0).
 *   - bf16 tensors are passed as uint16_t bit patterns.
 *   - Thread safety: calls are re-entrant; rs_last_error() is per thread.
 */
#ifndef RESPEC_H
#define RESPEC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ------------------------------------------------------------------ limits */
#define RS_MAX_L      8    /* longest retrieval key (the paper uses l = 3)     */
#define RS_MAX_TOPC   8    /* candidates kept per request (the paper uses 3)  */
#define RS_MAX_SPAN   256  /* retrieved continuation length                   */
#define RS_MAX_BETA   16   /* TopK size of Eq. 6                              */
#define RS_MAX_NODES  256  /* draft-tree nodes per request, root included     */

/* ------------------------------------------------------------------ status */
typedef enum {
    RS_OK = 0,
    RS_ERR_INVALID_ARG = 1, /* null pointer, negative size, parameter out of range */
    RS_ERR_UNSUPPORTED = 2, /* e.g. head dim not in {64, 128}, Hq % Hkv != 0       */
    RS_ERR_CAPACITY = 3,    /* workspace too small                                 */
    RS_ERR_CUDA = 4         /* a CUDA launch failed (message from the runtime)     */
} rs_status;

/* per-request status bits (device int32 status[b]) */
#define RS_ST_BAD_TREE   1  /* parents not topological, root not -1, source/chain
                               layout broken, or a node count out of range     */
#define RS_ST_TRUNCATED  2  /* an output list was longer than its capacity     */
#define RS_ST_BAD_POS    4  /* a selected position lies outside the buffer     */
#define RS_ST_TOO_LARGE  8  /* more than RS_MAX_NODES tree nodes               */
#define RS_ST_TIMEOUT   16  /* a pipeline wait inside a kernel gave up (bounded
                               wait, ~2 s; the environment variable
                               RS_DEBUG_WAIT_LIMIT, in clock cycles, shortens it
                               for tests); the request's outputs are invalid   */
#define RS_ST_BAD_OFFSET 32 /* the request's range in an offsets array lies
                               outside the arrays it indexes (a negative start
                               or length, or an end past R, kv_rows, t_total or
                               the array's last entry): the kernels check every
                               range they read from device memory before they
                               index with it, skip the request and leave every
                               array outside their own outputs untouched     */

/* -------------------------------------------------------------- parameters */
/* Hyper-parameters of Algorithm 1 (its inputs), Eq. 6-7 and Section 3.4.
 * Passed by value.  Defaults used by this project where the paper gives no
 * value: lambda_e 0.5, alpha 0.3, theta_score 0.3, beta 5, tau 3, phi 2,
 * m 2; the paper fixes theta_entropy = 1.5, top_c = 3 and l = 3. */
typedef struct {
    int   l;              /* maximum key length, 1..RS_MAX_L                       */
    float lambda_e;       /* Eq. 2 length penalty                                  */
    float theta_entropy;  /* trigger threshold of Section 3.2.1, nats              */
    float alpha;          /* Eq. 4 EMA rate, in [0, 1]                             */
    float theta_score;    /* Section 3.3 score threshold                           */
    int   top_c;          /* candidates kept, 1..RS_MAX_TOPC                       */
    int   span_len;       /* retrieved continuation length L, 1..RS_MAX_SPAN       */
    int   beta;           /* Eq. 6 TopK size, 1..RS_MAX_BETA (and <= V)             */
    float tau;            /* Eq. 7 tolerance, >= 0                                  */
    int   phi;            /* relaxed attempts of the look-ahead procedure, >= 0    */
    int   m;              /* greedy matches the look-ahead needs, >= 0             */
} rs_params;

/* Message for the last failing call on this thread ("" if none). */
const char *rs_last_error(void);

/* Library version string. */
const char *rs_version(void);

/* Number of kernels this library has launched in this process. */
uint64_t rs_launch_count(void);

/* Offsets arrays hold device data the host cannot check, so each kernel
 * checks the ranges it reads (see RS_ST_BAD_OFFSET): node_off / row_off
 * against R (or their last entry), tok_off against its last entry (the token
 * and score buffers hold tok_off[B] entries) or the index's t_total, kv_off +
 * ctx_len + node count against kv_rows.  rs_entropy_gate and
 * rs_entropy_gate_rows have no status output: a request whose row range is
 * out of bounds pushes no entropies (its trigger is evaluated on its history
 * as it was). */

/* ===================================================== rs_entropy_gate ====
 * Section 3.2.1 (Eq. 1: mean predictive entropy of a key; Eq. 2: C_k =
 * H_k + lambda_e / k; Eq. 3: k* = argmin C_k; trigger decision: iff
 * H_{k*} <= theta_entropy), evaluated as Algorithm 1's triggering does (k upward,
 * strict '<', so ties keep the shorter key).
 *
 *   logits     [R, V] fp32 row-major: the verify pass's next-token logits,
 *              one row per tree node (row r of request b for r in
 *              [row_off[b], row_off[b+1])).  16-byte aligned rows take the
 *              vector path; any V >= 1 works.
 *   row_off    [B+1] int32 row offsets per request.
 *   row_commit [R] uint8: 1 for the rows whose entropy enters the history,
 *              i.e. the rows that predicted a committed token (the root row
 *              and the rows of the accepted nodes, as rs_accept's `commit`
 *              output gives them), pushed in row order.
 *   hist       [B, p.l] fp32 in/out: per request the newest entropies, oldest
 *              first; hist_n [B] int32 in/out: how many are valid (0..l).
 *   entropy    [R] fp32 out: H(softmax(row)) in nats for every row.
 *   k_star     [B] int32 out: chosen key length (0 when the history is empty).
 *   h_best     [B] fp32 out: H_{k*} (+inf when k* = 0).
 *   entropy_ok [B] uint8 out: 1 iff k* > 0 and H_{k*} <= theta_entropy.
 * H_k and C_k are evaluated in fp64 from the fp32 history.  The row entropy
 * is accumulated in fp32 (one online max/sum pass per row).
 */
size_t rs_entropy_gate_workspace_size(int R, int V);
rs_status rs_entropy_gate(const float *logits, int R, int V, const int32_t *row_off,
                          const uint8_t *row_commit, int B, rs_params p,
                          float *hist, int32_t *hist_n, float *entropy,
                          int32_t *k_star, float *h_best, uint8_t *entropy_ok,
                          void *workspace, size_t workspace_bytes, void *stream);

/* ================================================ rs_entropy_gate_rows ====
 * The trigger of rs_entropy_gate (history push, H_k, C_k, k*, decision) from
 * row entropies computed elsewhere -- rs_accept's `entropy` output over the
 * same logits -- instead of from the logits.  Arguments as rs_entropy_gate;
 * `entropy` is an input here.  One kernel, no workspace.
 */
rs_status rs_entropy_gate_rows(const float *entropy, const int32_t *row_off,
                               const uint8_t *row_commit, int B, rs_params p,
                               float *hist, int32_t *hist_n, int32_t *k_star,
                               float *h_best, uint8_t *entropy_ok, void *stream);

/* ============================================= rs_entropy_gate_noalloc ====
 * Not from the paper (it has no counterpart): rs_entropy_gate for callers
 * that cannot allocate device memory -- for example code embedded in a
 * serving engine whose memory pool owns all of the GPU's memory and hands out
 * no scratch buffers, or code that must not call cudaMalloc because that
 * would synchronise the device in the middle of its work.  The caller still
 * passes every input and output (same meaning as rs_entropy_gate); the
 * library's scratch is a fixed device array of RS_GATE_NOALLOC_MAX_PARTIALS
 * (max, sum, weighted-sum) triples (768 KiB) that every GPU loading the
 * library holds until the process exits.  It supports
 * R * ceil(V / 8192) <= RS_GATE_NOALLOC_MAX_PARTIALS (e.g. R <= 4096 rows at
 * V = 128256); larger calls return RS_ERR_CAPACITY without launching.
 * The first call on each device looks the array's device address up
 * (cudaGetSymbolAddress), so make that first call before any stream capture;
 * the address is remembered per CUDA context, so the first call after a
 * device reset (or from another context on the same device) looks it up
 * again.
 * Nothing in the array needs to start at zero.  All calls share the array:
 * calls that overlap on the GPU (other streams, or unordered host threads)
 * race on it.  This call allocates nothing.
 */
#define RS_GATE_NOALLOC_MAX_PARTIALS 65536
rs_status rs_entropy_gate_noalloc(const float *logits, int R, int V, const int32_t *row_off,
                                  const uint8_t *row_commit, int B, rs_params p,
                                  float *hist, int32_t *hist_n, float *entropy,
                                  int32_t *k_star, float *h_best, uint8_t *entropy_ok,
                                  void *stream);

/* ======================================================= rs_match_scan ====
 * Section 3.3 "Selection Algorithm" and Algorithm 1's retrieval: find every
 * earlier occurrence of the key (the buffer's last k = k_star[b] tokens),
 * drop positions whose score is below theta_score, keep the top_c best by
 * score and gather their continuations.
 *
 *   tokens   [sum t_b] int32: per request the committed token buffer
 *            (prompt + generated, ending with the root token), request b at
 *            tokens[tok_off[b] .. tok_off[b+1]).
 *   tok_off  [B+1] int64.
 *   k_star   [B] int32 key lengths (rs_entropy_gate's output); k <= 0 skips
 *            the request, k > RS_MAX_L skips it with RS_ST_TOO_LARGE.
 *   gate_ok  [B] uint8 or NULL: when given, requests with gate_ok[b] == 0
 *            are skipped (Algorithm 1 retrieves only when the entropy half
 *            of the trigger holds).
 *   scores   [sum t_b] fp32 feedback scores, parallel to tokens (score of a
 *            match = score of its end position; initialise to S0 = 0.5).
 *   pos_cap  capacity of `pos` per request (>= 0).
 * Outputs (per request b):
 *   count [B]           number of match positions p, k-1 <= p <= t-2, whose
 *                       trailing k tokens equal the key (Contains <=> > 0);
 *   pos   [B, pos_cap]  the first min(count, pos_cap) of them, ascending,
 *                       -1 padded (RS_ST_TRUNCATED when count > pos_cap; the
 *                       selection still considers every match);
 *   sel_pos [B, top_c]  selected positions, best first: score desc, then
 *                       most recent first; -1 padded;
 *   sel_len [B, top_c]  continuation lengths min(span_len, t-1-p), 0 padded;
 *   spans [B, top_c, span_len] continuation tokens tokens[p+1 ..], -1 padded;
 *   n_sel [B]           number selected;  status [B] as above.
 */
size_t rs_match_scan_workspace_size(int B);
rs_status rs_match_scan(const int32_t *tokens, const int64_t *tok_off, int B,
                        const int32_t *k_star, const uint8_t *gate_ok,
                        const float *scores, rs_params p, int pos_cap,
                        int32_t *count, int32_t *pos, int32_t *sel_pos,
                        int32_t *sel_len, int32_t *spans, int32_t *n_sel,
                        int32_t *status, void *workspace, size_t workspace_bytes,
                        void *stream);

/* ================================================= rs_tree_verify_attn ====
 * Attention of the verify pass over the packed draft tree (the verify
 * forward of Algorithm 1; the paper's "parallel verification", Section 3.3): every
 * tree node attends to its request's whole committed prefix and to the
 * tree slots of its ancestors and itself.
 *
 *   q        [R, Hq, D] bf16: one row per tree node (R = node_off[B]).
 *   k, v     [kv_rows, Hkv, D] bf16 KV cache; request b's prefix slot j
 *            (j < ctx_len[b]) is row kv_off[b] + j and its tree node i is row
 *            kv_off[b] + ctx_len[b] + i.  k and v must be 16-byte aligned.
 *   kv_off   [B] int64;  ctx_len [B] int32 (>= 0);  node_off [B+1] int32;
 *            B <= 3840 requests per call; kv_rows < 2^31 and
 *            (2 Hq + Hkv) (kv_rows / 128 + B) < 2.2e8 (the work split's
 *            32-bit prefixes; RS_ERR_UNSUPPORTED otherwise, far beyond a KV
 *            cache that fits in memory at common head counts).
 *   parents  [R] int32 local parent index per node; parents of node 0 is -1,
 *            0 <= parents[i] < i otherwise.
 *   D in {64, 128}; Hq a multiple of Hkv (grouped-query heads h share KV
 *   head h / (Hq / Hkv)); scale > 0 is the softmax scale (1/sqrt(D) usually).
 *   out      [R, Hq, D] fp32 attention outputs;  lse [R, Hq] fp32 natural-log
 *            sum of exp(scale * q.k) over the attended keys.  out and the
 *            workspace must be 16-byte aligned.
 *   status   [B]: RS_ST_BAD_TREE / RS_ST_TOO_LARGE for a malformed request
 *            (its out/lse rows are zeroed).
 * QK^T and PV run on the tensor cores with fp32 accumulation.  The call
 * picks one of two kernel forms from its sizes (one 128-row tile per work
 * segment, or a pair of tiles sharing each K/V tile when the requests
 * average more than 128 (node, q-head-in-group) rows per KV head); the
 * workspace size depends on that choice, so size it with the same five
 * sizes as the call.  Environment: RS_DEBUG_ATTN_FORM=one|pair (a test
 * hook) forces either form; both compute the same function.
 */
size_t rs_tree_verify_attn_workspace_size(int B, int R, int Hq, int Hkv, int D);
rs_status rs_tree_verify_attn(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                              int64_t kv_rows, const int64_t *kv_off, const int32_t *ctx_len,
                              const int32_t *node_off, const int32_t *parents, int B, int R,
                              int Hq, int Hkv, int D, float scale, float *out, float *lse,
                              int32_t *status, void *workspace, size_t workspace_bytes,
                              void *stream);

/* =========================================================== rs_accept ====
 * Section 3.4 source-aware verification, the longest accepted path of
 * Algorithm 1 and the EMA feedback of Eq. 4-5 (Algorithm 1's score update).
 *
 *   logits   [R, V] fp32 verify logits (row of node i predicts its children).
 *   node_off [B+1] int32;  tokens [R] int32 draft token of every node, in
 *            [0, V) (the root's is ignored; an id outside the vocabulary makes
 *            the request RS_ST_BAD_TREE);  parents [R] int32 as for
 *            rs_tree_verify_attn.
 *   source   [R] uint8: 0 root (node 0 only), 1 model draft, 2 retrieved.
 *   chain    [R] int8: retrieved chain id (0..top_c-1) of source-2 nodes, -1
 *            otherwise.  Model nodes hang from the root or model nodes; the
 *            nodes of chain c, in index order, form a path from the root.
 *   sel_pos  [B, top_c] int32: buffer position that chain c was retrieved
 *            from (rs_match_scan's sel_pos), -1 when none.
 *   tok_off  [B+1] int64 and scores [sum t_b] fp32 in/out: the feedback
 *            table updated in place for the selected positions.
 *   acc_cap  capacity of acc_nodes per request (>= 1).
 * Row outputs, for every node row r:
 *   argmax [R]        lowest id among the maximal logits;
 *   topk   [R, beta]  ids in (logit desc, id asc) order;
 *   lse    [R] fp32   log-sum-exp of the row;
 *   p_tok  [R] fp32   probability of node r's token under its parent's row
 *                     (1 for the root, 0 in a malformed request);
 *   entropy [R] fp32 or NULL: when given, the row entropy in nats (Eq. 1,
 *                     as rs_entropy_gate computes it) from the same pass over
 *                     the logits.  The verify step's logits are the next
 *                     step's trigger input, so passing this to
 *                     rs_entropy_gate_rows saves the gate's own logits pass.
 * Decision outputs, per request b:
 *   acc_len [B]            accepted draft tokens on the winning path;
 *   acc_nodes [B, acc_cap] their local node indices in depth order, -1 padded;
 *   bonus [B]              argmax of the last accepted node's row (root's row
 *                          when nothing was accepted);
 *   winner [B]             -1 model tree, c = chain c, -2 nothing accepted;
 *   commit [R] uint8       1 for the root and the accepted nodes (feed it to
 *                          the next rs_entropy_gate as row_commit);
 *   status [B].
 * Model drafts: greedy strict verification (accepted iff token == argmax of
 * the parent row and the parent is accepted).  Retrieved chains: relaxed
 * check (token in TopK_beta and z_max - z_token <= tau, Eq. 6-7, as an fp64
 * logit gap) with the look-ahead tolerance procedure.  Ties: model tree
 * first, then chains in selection order.  EMA: S <- (1-alpha) S + alpha R,
 * R = acc_len / chain length for the winning chain and 0 for every other
 * chain with a selected position (evaluated in fp64, stored in fp32).
 */
size_t rs_accept_workspace_size(int R, int V, int beta);
rs_status rs_accept(const float *logits, int R, int V, const int32_t *node_off, int B,
                    const int32_t *tokens, const int32_t *parents, const uint8_t *source,
                    const int8_t *chain, const int32_t *sel_pos, const int64_t *tok_off,
                    rs_params p, int acc_cap, int32_t *argmax, int32_t *topk, float *lse,
                    float *p_tok, float *entropy, int32_t *acc_len, int32_t *acc_nodes,
                    int32_t *bonus, int32_t *winner, uint8_t *commit, float *scores,
                    int32_t *status, void *workspace, size_t workspace_bytes, void *stream);

/* ============================================ rs_match_index (NEXT-4) ====
 * An index for Section 3.3's retrieval on long buffers, kept current step by
 * step.  Algorithm 1 asks its suffix automaton two things about the key (the
 * buffer's last k <= RS_MAX_L tokens), Contains and RetrievePositions, and
 * after each step adds the committed tokens to it (Update).  Both questions
 * are answered exactly from an inverted index: for every token id, the
 * ascending list of positions holding it; the positions holding the key's
 * last token are the candidates, verified against the key's other tokens.  A
 * query costs O(occurrences of that token) instead of rs_match_scan's O(t);
 * an update costs O(tokens added).
 *
 * rs_match_index_bytes(B, V, t_total): device bytes of an index over B
 *   buffers of ids in [0, V) (others share one bucket) holding t_total tokens
 *   in all at build time (tok_off[B] then), including the build's scratch.
 *   Each id's list has room for a quarter more positions than it held at
 *   build time (plus two), and each request has an overflow list of 4096
 *   positions for ids whose room is used up.
 * rs_match_index_build: indexes tokens[tok_off[b] .. tok_off[b+1]) of every
 *   request (the index remembers each request's length and offset).  The
 *   caller owns `index`; nothing in it needs initialising.  Requires
 *   ceil(log2(V + 1)) + ceil(log2(B)) <= 32 (RS_ERR_UNSUPPORTED otherwise).
 * rs_match_index_append: adds the tokens appended to each request's buffer
 *   since the build or the last append: positions built .. t_b - 1, where t_b
 *   = tok_off[b+1] - tok_off[b] now (positions are relative to the request's
 *   first token, so the buffers may be laid out anew between calls; the
 *   tokens already indexed must not change).  V and t_total as given to the
 *   build.  status [B] int32 (or NULL): RS_ST_TRUNCATED when some positions
 *   could not be indexed (an id's room and the overflow list both full): they
 *   and every later position are then tested one by one by the queries until
 *   the next build.  One CTA per request.
 * rs_match_scan_indexed: rs_match_scan's inputs, outputs and meaning, plus
 *   V, t_total (as given to the build) and the index.  Positions the index
 *   does not hold (appended without rs_match_index_append, or left out as
 *   above) are tested one by one.  One CTA per request.
 */
size_t rs_match_index_bytes(int B, int V, int64_t t_total);
rs_status rs_match_index_build(const int32_t *tokens, const int64_t *tok_off, int B, int V, int64_t t_total,
                               void *index, size_t index_bytes, void *stream);
rs_status rs_match_index_append(const int32_t *tokens, const int64_t *tok_off, int B, int V, int64_t t_total,
                                void *index, size_t index_bytes, int32_t *status, void *stream);
rs_status rs_match_scan_indexed(const int32_t *tokens, const int64_t *tok_off, int B, const int32_t *k_star,
                                const uint8_t *gate_ok, const float *scores, rs_params p, int pos_cap,
                                int32_t *count, int32_t *pos, int32_t *sel_pos, int32_t *sel_len,
                                int32_t *spans, int32_t *n_sel, int32_t *status, int V, int64_t t_total,
                                const void *index, size_t index_bytes, void *stream);

/* ======================================================= rs_tree_sample ===
 * Section 3.4, "For Drafter Module outputs": lossless speculative sampling
 * of the model-drafted nodes (the non-greedy counterpart of rs_accept's
 * strict check).  The model children of a node are deterministic expansions
 * (a point-mass proposal each); speculative sampling over them has the law
 * of: draw y from the target row at temperature T, accept the model child
 * carrying y and continue from it, otherwise y is the correction token.
 * Every row's draw is the inverse CDF, in token-id order, of the caller's
 * uniform: the smallest id v with sum_{w <= v} softmax(z / T)(w) > u.
 * Retrieved nodes (source 2) are not proposals here; they are verified by
 * rs_accept's relaxed procedure.
 *
 *   logits, R, V, node_off, B, tokens, parents, source: as for rs_accept.
 *   temperature  T > 0 (finite), RS_ERR_INVALID_ARG otherwise.
 *   uniforms [R] fp32 in [0, 1): one per row, drawn by the caller (e.g. a
 *            counter-based generator); a value >= 1 selects the row's last
 *            id with mass.
 *   acc_cap  capacity of acc_nodes per request (>= 1).
 * Outputs:
 *   draw    [R] int32     every row's draw (0 for a row without mass);
 *   acc_len [B] int32     accepted model nodes from the root (RS_ST_TRUNCATED
 *                         when above acc_cap: acc_nodes keeps the first ones);
 *   acc_nodes [B, acc_cap] int32  local node indices in depth order, -1 padded;
 *   bonus   [B] int32     the correction token (the draw of the last accepted
 *                         node, or of the root);
 *   status  [B] int32     RS_ST_BAD_TREE (parents / source layout) or
 *                         RS_ST_TOO_LARGE (more than RS_MAX_NODES nodes):
 *                         acc_len 0, bonus -1.
 * Draws are exact: each is the fp64 inverse CDF above (exp and sums in fp64,
 * token-id order), up to rounding at the 1e-12 level of Z.  An fp32 pass
 * settles each row under a rigorous error bound; rows whose u Z lies within
 * that bound of a CDF step (a few percent of high-entropy rows) are redone
 * in double-float arithmetic, spread over the GPU.
 * Workspace: rs_tree_sample_workspace_size(R, V) bytes (per 8192-logit chunk
 * of every row its maximum and mass terms; the list of redone rows; per
 * 512-id slice of every row a double-float sum).  Stream-ordered: a call
 * must not share its workspace with a call in flight on another stream.
 * Environment: RS_DEBUG_SAMPLE_EXACT=1 (a test hook) redoes every row with
 * mass.
 */
size_t rs_tree_sample_workspace_size(int R, int V);
rs_status rs_tree_sample(const float *logits, int R, int V, const int32_t *node_off, int B,
                         const int32_t *tokens, const int32_t *parents, const uint8_t *source,
                         float temperature, const float *uniforms, int acc_cap, int32_t *draw,
                         int32_t *acc_len, int32_t *acc_nodes, int32_t *bonus, int32_t *status,
                         void *workspace, size_t workspace_bytes, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* RESPEC_H */
