// scan.cu -- rs_match_scan: retrieval and feedback-driven candidate
// selection (Section 3.3 "Selection Algorithm"; Algorithm 1 l.9-11).
//
// One CTA of 1024 threads per request.  The buffer is swept in windows of
// 32768 positions: warp w, step j tests positions window + 32 (w + 32 j) +
// lane against the key (kept in shared memory) and its ballot is one 32-bit
// word of the window's match bitmask.  Thread i then owns bitmask word i
// (32 consecutive positions): a block-wide exclusive scan of the words'
// popcounts gives every match its rank, so positions are written in
// ascending order with no sort.  Each thread keeps its best top_c matches
// (score desc, position desc) in a small register list; top_c rounds of a
// block-wide reduction pick the selected positions, whose continuations are
// then gathered.
#include <math.h>

#include "common.cuh"

namespace rs {
namespace {

constexpr int kScanThreads = 1024;
constexpr int kWin = kScanThreads * 32;  // positions per window

// (s, p) before (s2, p2): higher score first, then the more recent position
__device__ __forceinline__ bool sp_before(float s, int p, float s2, int p2) {
    return s > s2 || (s == s2 && p > p2);
}

__device__ __forceinline__ int block_excl_scan(int v, int *s_warp, int &total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = s_warp[lane];
        int z = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, z, o);
            if (lane >= o) z += y;
        }
        s_warp[lane] = z - w;  // exclusive prefix of warp totals
        if (lane == 31) s_warp[32] = z;
    }
    __syncthreads();
    int r = s_warp[warp] + x - v;
    total = s_warp[32];
    __syncthreads();  // s_warp reusable
    return r;
}

__global__ void __launch_bounds__(kScanThreads)
match_scan_kernel(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off,
                  const int32_t *__restrict__ k_star, const uint8_t *__restrict__ gate_ok,
                  const float *__restrict__ scores, float theta_score, int top_c, int span_len, int pos_cap,
                  int32_t *__restrict__ count, int32_t *__restrict__ pos, int32_t *__restrict__ sel_pos,
                  int32_t *__restrict__ sel_len, int32_t *__restrict__ spans, int32_t *__restrict__ n_sel,
                  int32_t *__restrict__ status) {
    const int b = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const long long t0 = tok_off[b];
    const long long t = tok_off[b + 1] - t0;
    const int32_t *X = tokens + t0;
    const float *S = scores + t0;
    int k = k_star[b];

    __shared__ int s_key[RS_MAX_L];
    __shared__ uint32_t s_bits[kWin / 32];
    __shared__ int s_warp[33];
    __shared__ float s_wv[32];
    __shared__ int s_wp[32];
    __shared__ int s_sel[RS_MAX_TOPC];

    int st = 0;
    bool run = k > 0 && (gate_ok == nullptr || gate_ok[b] != 0);
    if (run && k > RS_MAX_L) {
        st = RS_ST_TOO_LARGE;
        run = false;
    }
    if (run && (long long)k > t) run = false;
    if (run && tid < k) s_key[tid] = X[t - k + tid];
    __syncthreads();

    // per-thread best list (score desc, position desc), kept sorted
    float ls[RS_MAX_TOPC];
    int lp[RS_MAX_TOPC];
#pragma unroll
    for (int i = 0; i < RS_MAX_TOPC; ++i) {
        ls[i] = -INFINITY;
        lp[i] = -1;
    }

    long long cnt = 0;
    if (run) {
        const long long pend = t - 1;  // positions p in [k-1, t-2]
        for (long long w0 = 0; w0 < pend; w0 += kWin) {
            // match bitmask of this window
#pragma unroll 4
            for (int j = 0; j < 32; ++j) {
                const long long p = w0 + (long long)(warp + 32 * j) * 32 + lane;
                bool m = false;
                if (p >= k - 1 && p < pend) {
                    m = true;
                    for (int i = 0; i < k; ++i) m = m && (X[p - k + 1 + i] == s_key[i]);
                }
                unsigned bal = __ballot_sync(0xffffffffu, m);
                if (lane == 0) s_bits[warp + 32 * j] = bal;
            }
            __syncthreads();
            const uint32_t word = s_bits[tid];
            int total = 0;
            const int rank = block_excl_scan(__popc(word), s_warp, total);
            uint32_t rem = word;
            int i = 0;
            while (rem) {
                const int bit = __ffs(rem) - 1;
                rem &= rem - 1;
                const long long p = w0 + (long long)tid * 32 + bit;
                const long long idx = cnt + rank + i++;
                if (idx < pos_cap) pos[(long long)b * pos_cap + idx] = (int32_t)p;
                const float s = S[p];
                if (s >= theta_score && sp_before(s, (int)p, ls[RS_MAX_TOPC - 1], lp[RS_MAX_TOPC - 1])) {
                    // insert into the sorted register list (fully unrolled)
                    float cs = s;
                    int cp = (int)p;
#pragma unroll
                    for (int q = 0; q < RS_MAX_TOPC; ++q) {
                        if (sp_before(cs, cp, ls[q], lp[q])) {
                            float ts = ls[q];
                            int tp = lp[q];
                            ls[q] = cs;
                            lp[q] = cp;
                            cs = ts;
                            cp = tp;
                        }
                    }
                }
            }
            cnt += total;
            __syncthreads();  // s_bits reusable
        }
    }

    // pad the position list
    const long long stored = cnt < pos_cap ? cnt : pos_cap;
    for (long long i = stored + tid; i < pos_cap; i += kScanThreads) pos[(long long)b * pos_cap + i] = -1;
    if (cnt > pos_cap) st |= RS_ST_TRUNCATED;

    // top_c rounds of a block-wide best-head reduction
    int nsel = 0;
    for (int c = 0; c < top_c; ++c) {
        float hv = ls[0];
        int hp = lp[0];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            float ov = __shfl_xor_sync(0xffffffffu, hv, o);
            int op = __shfl_xor_sync(0xffffffffu, hp, o);
            if (sp_before(ov, op, hv, hp)) {
                hv = ov;
                hp = op;
            }
        }
        if (lane == 0) {
            s_wv[warp] = hv;
            s_wp[warp] = hp;
        }
        __syncthreads();
        hv = s_wv[lane];
        hp = s_wp[lane];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            float ov = __shfl_xor_sync(0xffffffffu, hv, o);
            int op = __shfl_xor_sync(0xffffffffu, hp, o);
            if (sp_before(ov, op, hv, hp)) {
                hv = ov;
                hp = op;
            }
        }
        __syncthreads();  // s_wv / s_wp reusable
        if (hp < 0) break;  // no candidate left
        if (tid == 0) s_sel[c] = hp;
        nsel = c + 1;
        if (lp[0] == hp) {  // the owner pops its head
#pragma unroll
            for (int q = 0; q < RS_MAX_TOPC - 1; ++q) {
                ls[q] = ls[q + 1];
                lp[q] = lp[q + 1];
            }
            ls[RS_MAX_TOPC - 1] = -INFINITY;
            lp[RS_MAX_TOPC - 1] = -1;
        }
    }
    __syncthreads();

    // selected positions, lengths and continuations
    for (int i = tid; i < top_c * span_len; i += kScanThreads) {
        const int c = i / span_len, j = i - c * span_len;
        int v = -1;
        if (c < nsel) {
            const long long p = s_sel[c];
            long long len = t - 1 - p;
            if (len > span_len) len = span_len;
            if (j < len) v = X[p + 1 + j];
        }
        spans[(long long)b * top_c * span_len + i] = v;
    }
    if (tid < top_c) {
        const int c = tid;
        int sp = -1, sl = 0;
        if (c < nsel) {
            sp = s_sel[c];
            long long len = t - 1 - sp;
            sl = (int)(len > span_len ? span_len : len);
        }
        sel_pos[(long long)b * top_c + c] = sp;
        sel_len[(long long)b * top_c + c] = sl;
    }
    if (tid == 0) {
        count[b] = (int32_t)cnt;
        n_sel[b] = nsel;
        status[b] = st;
    }
}

}  // namespace
}  // namespace rs

using namespace rs;

extern "C" size_t rs_match_scan_workspace_size(int B) {
    (void)B;
    return 0;
}

extern "C" rs_status rs_match_scan(const int32_t *tokens, const int64_t *tok_off, int B, const int32_t *k_star,
                                   const uint8_t *gate_ok, const float *scores, rs_params p, int pos_cap,
                                   int32_t *count, int32_t *pos, int32_t *sel_pos, int32_t *sel_len,
                                   int32_t *spans, int32_t *n_sel, int32_t *status, void *workspace,
                                   size_t workspace_bytes, void *stream) {
    clear_error();
    (void)workspace;
    (void)workspace_bytes;
    RS_CHECK_ARG(B >= 0, "rs_match_scan: negative B");
    RS_CHECK_ARG(pos_cap >= 0, "rs_match_scan: negative pos_cap");
    RS_CHECK_ARG(p.top_c >= 1 && p.top_c <= RS_MAX_TOPC, "rs_match_scan: top_c=%d outside [1, %d]", p.top_c,
                 RS_MAX_TOPC);
    RS_CHECK_ARG(p.span_len >= 1 && p.span_len <= RS_MAX_SPAN, "rs_match_scan: span_len=%d outside [1, %d]",
                 p.span_len, RS_MAX_SPAN);
    RS_CHECK_ARG(B == 0 || (tokens && tok_off && k_star && scores && count && sel_pos && sel_len && spans &&
                            n_sel && status && (pos || pos_cap == 0)),
                 "rs_match_scan: null pointer");
    if (B == 0) return RS_OK;
    match_scan_kernel<<<B, kScanThreads, 0, (cudaStream_t)stream>>>(
        tokens, tok_off, k_star, gate_ok, scores, p.theta_score, p.top_c, p.span_len, pos_cap, count, pos,
        sel_pos, sel_len, spans, n_sel, status);
    RS_CHECK_LAUNCH("rs_match_scan");
    return RS_OK;
}
