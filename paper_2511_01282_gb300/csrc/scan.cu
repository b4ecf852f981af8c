// scan.cu -- rs_match_scan: retrieval and feedback-driven candidate
// selection (Section 3.3 "Selection Algorithm"; Algorithm 1 l.9-11).
//
// One cluster of 8 CTAs (256 threads each) per request; CTA c scans the c-th
// eighth of the candidate positions [k-1, t-2].  Per window of 8192
// positions, warp w, step j tests positions 32 (w + 8 j) + lane against the
// key (both staged in shared memory) and its ballot is one 32-bit word of
// the window's match bitmask; thread i owns word i.  Pass 1 counts the slice's
// matches and keeps each thread's best top_c matches (score desc, position
// desc) in a small register list, merged per CTA.  After a cluster barrier
// every CTA reads its peers' counts through distributed shared memory, so
// pass 2 writes its positions at their global ascending rank (a block scan
// of word popcounts orders them within a window) -- no sort.  CTA 0 merges
// the eight per-CTA top_c lists and gathers the selected continuations.  The
// cluster's CTAs are co-scheduled and all of them pass the same two cluster
// barriers, so nothing waits on a CTA that is not running.
#include <cooperative_groups.h>
#include <math.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace rs {
namespace {

constexpr int kScanCluster = 8;
constexpr int kScanThreads = 256;
constexpr int kScanWarps = kScanThreads / 32;
constexpr int kWin = kScanThreads * 32;  // positions per window

// (s, p) before (s2, p2): higher score first, then the more recent position
__device__ __forceinline__ bool sp_before(float s, int p, float s2, int p2) {
    return s > s2 || (s == s2 && p > p2);
}

struct ScanShared {
    int tok[kWin + RS_MAX_L];       // buffer tokens [w0 - (k - 1), w0 + kWin) of the current window
    uint32_t bits[kWin / 32];
    int warp_sums[kScanWarps + 1];
    float wv[kScanWarps];
    int wp[kScanWarps];
    int key[RS_MAX_L];
    long long cnt;                  // this CTA's match count (read by the peers)
    float top_s[RS_MAX_TOPC];       // this CTA's best top_c (read by CTA 0)
    int top_p[RS_MAX_TOPC];
    int ntop;
    int sel[RS_MAX_TOPC];
};

// Exclusive scan of one int per thread over the block; *total gets the sum.
__device__ __forceinline__ int block_excl_scan(int v, ScanShared &sh, int *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh.warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const int w = lane < kScanWarps ? sh.warp_sums[lane] : 0;
        int z = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, z, o);
            if (lane >= o) z += y;
        }
        if (lane < kScanWarps) sh.warp_sums[lane] = z - w;
        if (lane == kScanWarps - 1) sh.warp_sums[kScanWarps] = z;
    }
    __syncthreads();
    const int r = sh.warp_sums[warp] + x - v;
    *total = sh.warp_sums[kScanWarps];
    __syncthreads();  // warp_sums reusable
    return r;
}

// The match bitmask of window [w0, w0 + kWin) restricted to [lo, hi).  The
// window's tokens (and the k - 1 before it) are first staged in shared
// memory with independent coalesced loads.
__device__ __forceinline__ void window_bits(const int32_t *__restrict__ X, long long t, int k, long long w0,
                                            long long lo, long long hi, ScanShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const long long t_lo = w0 - (k - 1);
    for (int j = threadIdx.x; j < kWin + k - 1; j += kScanThreads) {
        const long long idx = t_lo + j;
        sh.tok[j] = (idx >= 0 && idx < t) ? X[idx] : -1;
    }
    __syncthreads();
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
        const int word = warp + kScanWarps * j;
        const long long p = w0 + (long long)word * 32 + lane;
        const int base = word * 32 + lane;  // tokens of p: tok[base .. base + k - 1]
        bool m = p >= lo && p < hi;
        for (int i = 0; i < k; ++i) m &= (sh.tok[base + i] == sh.key[i]);
        const unsigned bal = __ballot_sync(0xffffffffu, m);
        if (lane == 0) sh.bits[word] = bal;
    }
    __syncthreads();
}

// Best head of the block's register lists; every thread gets it.
__device__ __forceinline__ void block_best(float hv, int hp, ScanShared &sh, float *bv, int *bp) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, hv, o);
        const int op = __shfl_xor_sync(0xffffffffu, hp, o);
        if (sp_before(ov, op, hv, hp)) {
            hv = ov;
            hp = op;
        }
    }
    if (lane == 0) {
        sh.wv[warp] = hv;
        sh.wp[warp] = hp;
    }
    __syncthreads();
    hv = lane < kScanWarps ? sh.wv[lane] : -INFINITY;
    hp = lane < kScanWarps ? sh.wp[lane] : -1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, hv, o);
        const int op = __shfl_xor_sync(0xffffffffu, hp, o);
        if (sp_before(ov, op, hv, hp)) {
            hv = ov;
            hp = op;
        }
    }
    __syncthreads();  // wv / wp reusable
    *bv = hv;
    *bp = hp;
}

__global__ void __cluster_dims__(kScanCluster, 1, 1) __launch_bounds__(kScanThreads)
match_scan_kernel(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off,
                  const int32_t *__restrict__ k_star, const uint8_t *__restrict__ gate_ok,
                  const float *__restrict__ scores, float theta_score, int top_c, int span_len, int pos_cap,
                  int32_t *__restrict__ count, int32_t *__restrict__ pos, int32_t *__restrict__ sel_pos,
                  int32_t *__restrict__ sel_len, int32_t *__restrict__ spans, int32_t *__restrict__ n_sel,
                  int32_t *__restrict__ status) {
    cg::cluster_group cluster = cg::this_cluster();
    const int crank = (int)cluster.block_rank();
    const int b = blockIdx.y;
    const int tid = threadIdx.x;
    const long long t0 = tok_off[b];
    const long long t = tok_off[b + 1] - t0;
    const int32_t *X = tokens + t0;
    const float *S = scores + t0;
    const int k = k_star[b];
    __shared__ ScanShared sh;

    int st = 0;
    bool run = k > 0 && (gate_ok == nullptr || gate_ok[b] != 0);
    if (run && k > RS_MAX_L) {
        st = RS_ST_TOO_LARGE;
        run = false;
    }
    if (run && (long long)k > t) run = false;
    if (run && tid < k) sh.key[tid] = X[t - k + tid];

    // this CTA's slice of the candidate positions [k-1, t-2]
    long long lo = 0, hi = 0;
    if (run) {
        const long long first = k - 1, n = (t - 1) - first;
        long long per = (n + kScanCluster - 1) / kScanCluster;
        per = (per + 31) / 32 * 32;
        lo = first + (long long)crank * per;
        hi = lo + per < t - 1 ? lo + per : t - 1;
        if (lo > hi) lo = hi;
    }
    __syncthreads();

    // ---- pass 1: count, and each thread's best matches ----
    float ls[RS_MAX_TOPC];
    int lp[RS_MAX_TOPC];
#pragma unroll
    for (int i = 0; i < RS_MAX_TOPC; ++i) {
        ls[i] = -INFINITY;
        lp[i] = -1;
    }
    long long cnt = 0;
    for (long long w0 = lo; w0 < hi; w0 += kWin) {
        window_bits(X, t, k, w0, lo, hi, sh);
        uint32_t rem = sh.bits[tid];
        cnt += __popc(rem);
        while (rem) {
            const int bit = __ffs(rem) - 1;
            rem &= rem - 1;
            const long long p = w0 + (long long)tid * 32 + bit;
            const float s = S[p];
            if (s >= theta_score && sp_before(s, (int)p, ls[RS_MAX_TOPC - 1], lp[RS_MAX_TOPC - 1])) {
                float cs = s;
                int cp = (int)p;
#pragma unroll
                for (int q = 0; q < RS_MAX_TOPC; ++q) {
                    if (sp_before(cs, cp, ls[q], lp[q])) {
                        const float ts = ls[q];
                        const int tp = lp[q];
                        ls[q] = cs;
                        lp[q] = cp;
                        cs = ts;
                        cp = tp;
                    }
                }
            }
        }
        __syncthreads();  // bits and tok reusable
    }
    // the CTA's count and best top_c
    {
        int c32 = (int)cnt, total = 0;
        (void)block_excl_scan(c32, sh, &total);
        if (tid == 0) sh.cnt = total;
    }
    int ntop = 0;
    for (int c = 0; c < top_c; ++c) {
        float bv;
        int bp;
        block_best(ls[0], lp[0], sh, &bv, &bp);
        if (bp < 0) break;
        if (tid == 0) {
            sh.top_s[c] = bv;
            sh.top_p[c] = bp;
        }
        ntop = c + 1;
        if (lp[0] == bp) {  // the owner pops its head
#pragma unroll
            for (int q = 0; q < RS_MAX_TOPC - 1; ++q) {
                ls[q] = ls[q + 1];
                lp[q] = lp[q + 1];
            }
            ls[RS_MAX_TOPC - 1] = -INFINITY;
            lp[RS_MAX_TOPC - 1] = -1;
        }
    }
    if (tid == 0) sh.ntop = ntop;
    cluster.sync();

    // ---- the slice's global rank; pass 2 writes positions in order ----
    long long offset = 0, total = 0;
    for (int r = 0; r < kScanCluster; ++r) {
        const long long c = *cluster.map_shared_rank(&sh.cnt, r);
        if (r < crank) offset += c;
        total += c;
    }
    if (run && offset < pos_cap) {
        long long base = offset;
        for (long long w0 = lo; w0 < hi && base < pos_cap; w0 += kWin) {
            window_bits(X, t, k, w0, lo, hi, sh);
            uint32_t rem = sh.bits[tid];
            int wtotal = 0;
            const int rank = block_excl_scan(__popc(rem), sh, &wtotal);
            int i = 0;
            while (rem) {
                const int bit = __ffs(rem) - 1;
                rem &= rem - 1;
                const long long idx = base + rank + i++;
                if (idx < pos_cap) pos[(long long)b * pos_cap + idx] = (int32_t)(w0 + (long long)tid * 32 + bit);
            }
            base += wtotal;
            __syncthreads();  // bits reusable
        }
    }

    // ---- CTA 0: merge the per-CTA lists, selection outputs ----
    if (crank == 0) {
        const long long stored = total < pos_cap ? total : pos_cap;
        for (long long i = stored + tid; i < pos_cap; i += kScanThreads) pos[(long long)b * pos_cap + i] = -1;
        if (total > pos_cap) st |= RS_ST_TRUNCATED;
        if (tid < 32) {
            // up to kScanCluster * RS_MAX_TOPC = 64 candidates, two per lane
            float cv[2];
            int cpos[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int e = tid + 32 * h, r = e / RS_MAX_TOPC, q = e % RS_MAX_TOPC;
                cv[h] = -INFINITY;
                cpos[h] = -1;
                if (q < *cluster.map_shared_rank(&sh.ntop, r)) {
                    cv[h] = *cluster.map_shared_rank(&sh.top_s[q], r);
                    cpos[h] = *cluster.map_shared_rank(&sh.top_p[q], r);
                }
            }
            int nsel = 0;
            float pv = INFINITY;
            int pp = 0x7fffffff;
            for (int c = 0; c < top_c; ++c) {
                float hv = -INFINITY;
                int hp = -1;
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    if (cpos[h] >= 0 && sp_before(pv, pp, cv[h], cpos[h]) && sp_before(cv[h], cpos[h], hv, hp)) {
                        hv = cv[h];
                        hp = cpos[h];
                    }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const float ov = __shfl_xor_sync(0xffffffffu, hv, o);
                    const int op = __shfl_xor_sync(0xffffffffu, hp, o);
                    if (sp_before(ov, op, hv, hp)) {
                        hv = ov;
                        hp = op;
                    }
                }
                if (hp < 0) break;
                if (tid == 0) sh.sel[c] = hp;
                nsel = c + 1;
                pv = hv;
                pp = hp;
            }
            if (tid == 0) sh.ntop = nsel;  // own copy: the peers have been read
        }
        __syncthreads();
        const int nsel = sh.ntop;
        for (int i = tid; i < top_c * span_len; i += kScanThreads) {
            const int c = i / span_len, j = i - c * span_len;
            int v = -1;
            if (c < nsel) {
                const long long p = sh.sel[c];
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
                sp = sh.sel[c];
                const long long len = t - 1 - sp;
                sl = (int)(len > span_len ? span_len : len);
            }
            sel_pos[(long long)b * top_c + c] = sp;
            sel_len[(long long)b * top_c + c] = sl;
        }
        if (tid == 0) {
            count[b] = (int32_t)total;
            n_sel[b] = nsel;
            status[b] = st;
        }
    }
    cluster.sync();  // the peers' shared memory stays valid until CTA 0 is done
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
    RS_CHECK_ARG(B <= 65535, "rs_match_scan: B=%d above 65535", B);
    RS_CHECK_ARG(pos_cap >= 0, "rs_match_scan: negative pos_cap");
    RS_CHECK_ARG(p.top_c >= 1 && p.top_c <= RS_MAX_TOPC, "rs_match_scan: top_c=%d outside [1, %d]", p.top_c,
                 RS_MAX_TOPC);
    RS_CHECK_ARG(p.span_len >= 1 && p.span_len <= RS_MAX_SPAN, "rs_match_scan: span_len=%d outside [1, %d]",
                 p.span_len, RS_MAX_SPAN);
    RS_CHECK_ARG(B == 0 || (tokens && tok_off && k_star && scores && count && sel_pos && sel_len && spans &&
                            n_sel && status && (pos || pos_cap == 0)),
                 "rs_match_scan: null pointer");
    if (B == 0) return RS_OK;
    match_scan_kernel<<<dim3(kScanCluster, B), kScanThreads, 0, (cudaStream_t)stream>>>(
        tokens, tok_off, k_star, gate_ok, scores, p.theta_score, p.top_c, p.span_len, pos_cap, count, pos,
        sel_pos, sel_len, spans, n_sel, status);
    RS_CHECK_LAUNCH("rs_match_scan");
    return RS_OK;
}
