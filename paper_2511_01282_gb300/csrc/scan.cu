// scan.cu -- rs_match_scan: retrieval and feedback-driven candidate
// selection (Section 3.3 "Selection Algorithm"; Algorithm 1's retrieval).
//
// One cluster of 8 CTAs (256 threads each) per request.  A buffer whose
// candidate positions [0, t-2] fit one window of 8192 is handled by CTA 0
// alone (the other seven leave at once and no cluster barrier is used);
// otherwise CTA c scans the c-th eighth of the positions.  A window is staged
// in shared memory in one round of loads issued together: its tokens with
// the k-1 before it, its scores, and the key.  Warp w, step j tests positions
// 32 (w + 8 j) + lane against the key; the ballot is one 32-bit word of the
// window's match bitmask, and thread i owns word i.  One block scan of the
// word popcounts gives the CTA's match count and every thread's rank, so
// positions are written at their global ascending rank with no sort.
// Matches whose score clears theta_score are appended to a shared buffer and
// each is ranked by counting the buffered matches before it in (score desc,
// position desc) order, which gives the CTA's best top_c in one pass; if more
// match than the buffer holds, per-thread lists merged block-wide are used
// instead.  In the split case every CTA pushes its count
// to all peers and its best top_c to CTA 0 through distributed shared memory
// (once the cluster barrier's entry phase shows every CTA running) before one
// cluster barrier; after it nobody touches another CTA's shared memory.  CTA 0 ranks the (at most 64) listed matches the same way and
// gathers the selected continuations (from the staged window when it alone
// scanned the buffer).  A slice that
// spans several windows stages them in turn, and again for the position pass.
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
constexpr int kHalo = RS_MAX_L - 1;      // tokens staged before the window
constexpr int kScanCand = 256;           // matches ranked from the shared buffer

// (s, p) before (s2, p2): higher score first, then the more recent position
__device__ __forceinline__ bool sp_before(float s, int p, float s2, int p2) {
    return s > s2 || (s == s2 && p > p2);
}

struct ScanShared {
    int tok[kHalo + kWin];   // X[w0 - kHalo, w0 + kWin) (unwritten outside [0, t))
    float sc[kWin];          // S[w0, w0 + kWin)
    uint32_t bits[kWin / 32];
    float cs[kScanCand];     // matches with S >= theta_score (first kScanCand)
    int cp[kScanCand];
    int ccnt;
    int warp_sums[kScanWarps + 1];
    float wv[kScanWarps];
    int wp[kScanWarps];
    int key[RS_MAX_L];
    long long peer_cnt[kScanCluster];           // match count of each CTA (pushed by its owner)
    float peer_s[kScanCluster][RS_MAX_TOPC];    // CTA 0: each CTA's best top_c
    int peer_p[kScanCluster][RS_MAX_TOPC];
    int peer_n[kScanCluster];
    float top_s[RS_MAX_TOPC];                   // this CTA's best top_c
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
    int before = 0, sum = 0;
#pragma unroll
    for (int w = 0; w < kScanWarps; ++w) {
        const int y = sh.warp_sums[w];
        before += w < warp ? y : 0;
        sum += y;
    }
    __syncthreads();  // warp_sums reusable
    *total = sum;
    return before + x - v;
}

// Stage window [w0, w0 + kWin): tokens from w0 - kHalo that lie in
// [0, tok_hi), scores of the positions below `hi`, as asynchronous 4-byte
// copies (all in flight at once; the caller waits and synchronises).  Slots
// outside those ranges are left unwritten: the key test reads only tokens of
// candidate positions p - i, 0 <= p - i < hi, and a gathered span only
// tokens below t.
__device__ __forceinline__ void cp_async4(void *smem, const void *gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem)
                 : "memory");
}

__device__ __forceinline__ void stage_window(const int32_t *__restrict__ X, const float *__restrict__ S,
                                             long long tok_hi, long long hi, long long w0, ScanShared &sh) {
    const long long a = w0 - kHalo;
    const int j0 = (int)(a < 0 ? -a : 0);
    const int j1 = (int)(tok_hi - a < kHalo + kWin ? tok_hi - a : kHalo + kWin);
    for (int j = j0 + threadIdx.x; j < j1; j += kScanThreads) cp_async4(&sh.tok[j], X + a + j);
    const int n = (int)(hi - w0 < kWin ? hi - w0 : kWin);
    for (int j = threadIdx.x; j < n; j += kScanThreads) cp_async4(&sh.sc[j], S + w0 + j);
    asm volatile("cp.async.commit_group;" ::: "memory");
}

__device__ __forceinline__ void stage_wait() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// The match bitmask of the staged window restricted to [lo, hi).  The key is
// in registers (key[i] = X[t - k + i]).  Thread (warp, lane) tests positions
// w0 + 256 j + 32 warp + lane, j = 0..31.  Pass 1 has no branches: one
// shared load and compare of the last token per position and a ballot per
// word, kept by lane j.  Pass 2 visits only the words with a hit and
// compares the other k - 1 tokens.  The bitmask is written with one store per
// thread.
__device__ __forceinline__ void window_bits(const int (&key)[RS_MAX_L], int k, long long w0, long long lo,
                                            long long hi, ScanShared &sh) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int klast = key[k - 1];
    const int r0 = warp * 32 + lane;  // offset of this thread's j = 0 position in the window
    // valid j: lo <= w0 + r0 + 256 j < hi
    const long long dlo = lo - w0 - r0, dhi = hi - w0 - r0;
    const int jlo = dlo <= 0 ? 0 : (int)((dlo + kScanThreads - 1) / kScanThreads);
    const int jhi = dhi <= 0 ? 0 : (int)((dhi + kScanThreads - 1) / kScanThreads);
    const int *tk = sh.tok + kHalo + r0;
    uint32_t mine = 0;
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
        const bool m = (j >= jlo) & (j < jhi) & (tk[j * kScanThreads] == klast);
        const uint32_t bal = __ballot_sync(0xffffffffu, m);
        mine = lane == j ? bal : mine;
    }
    if (k > 1) {
        uint32_t words = __ballot_sync(0xffffffffu, mine != 0u);
        while (words) {
            const int j = __ffs(words) - 1;
            words &= words - 1;
            bool m = (j >= jlo) & (j < jhi) & (tk[j * kScanThreads] == klast);
            for (int i = 1; i < k; ++i) m = m && (tk[j * kScanThreads - i] == key[k - 1 - i]);
            const uint32_t bal = __ballot_sync(0xffffffffu, m);
            mine = lane == j ? bal : mine;
        }
    }
    sh.bits[warp + kScanWarps * lane] = mine;
}

// Rank of (s, p) among n distinct (score, position) pairs in shared memory:
// the number of pairs before it in (score desc, position desc) order.
__device__ __forceinline__ int sp_rank(float s, int p, const float *cs, const int *cp, int n) {
    int r = 0;
    for (int q = 0; q < n; ++q) r += sp_before(cs[q], cp[q], s, p);
    return r;
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
    pdl_enter();
    cg::cluster_group cluster = cg::this_cluster();
    const int crank = (int)cluster.block_rank();
    const int b = blockIdx.y;
    const int tid = threadIdx.x;
    extern __shared__ __align__(16) unsigned char scan_smem[];
    ScanShared &sh = *reinterpret_cast<ScanShared *>(scan_smem);
    const long long t0 = tok_off[b];
    const long long t = tok_off[b + 1] - t0;
    // the buffers hold tok_off[B] tokens: a range outside them is not read
    const bool off_ok = t0 >= 0 && t >= 0 && t0 + t <= tok_off[gridDim.y];
    const int32_t *X = tokens + (off_ok ? t0 : 0);
    const float *S = scores + (off_ok ? t0 : 0);
    const int k = k_star[b];

    int st = off_ok ? 0 : RS_ST_BAD_OFFSET;
    bool run = off_ok && k > 0 && (gate_ok == nullptr || gate_ok[b] != 0);
    if (run && k > RS_MAX_L) {
        st = RS_ST_TOO_LARGE;
        run = false;
    }
    if (run && (long long)k > t) run = false;

    // this CTA's slice [lo, hi) of the positions [0, t-2]; matches need p >= k-1
    // t <= kWin: the tokens [0, t) all fit the staged window (after the halo)
    const bool solo = !run || t <= kWin;  // CTA 0 alone, no cluster barrier
    if (solo && crank != 0) return;
    if (!solo) cluster_arrive_relaxed();  // this CTA runs; the wait sits before the first push
    long long lo = 0, hi = 0;
    if (run) {
        const long long n = t - 1;
        long long per = solo ? n : (n + kScanCluster - 1) / kScanCluster;
        per = (per + 31) / 32 * 32;
        lo = (long long)crank * per;
        hi = lo + per < n ? lo + per : n;
        if (lo > hi) lo = hi;
    }
    const long long plo = lo > k - 1 ? lo : (long long)(k - 1);
    const bool single = hi - lo <= kWin;
    if (tid == 0) sh.ccnt = 0;
    if (run && tid < k) sh.key[tid] = X[t - k + tid];
    if (run && lo < hi) stage_window(X, S, solo ? t : hi, hi, lo, sh);
    stage_wait();
    __syncthreads();
    int key[RS_MAX_L];
#pragma unroll
    for (int i = 0; i < RS_MAX_L; ++i) key[i] = (run && i < k) ? sh.key[i] : -1;

    // ---- pass 1: match bits, count, candidates ----
    float ls[RS_MAX_TOPC];
    int lp[RS_MAX_TOPC];
#pragma unroll
    for (int i = 0; i < RS_MAX_TOPC; ++i) {
        ls[i] = -INFINITY;
        lp[i] = -1;
    }
    int cnt = 0, rank = 0;
    for (long long w0 = lo; w0 < hi; w0 += kWin) {
        if (w0 != lo) {
            __syncthreads();  // the previous window is consumed
            stage_window(X, S, hi, hi, w0, sh);
            stage_wait();
            __syncthreads();
        }
        window_bits(key, k, w0, plo, hi, sh);
        __syncthreads();
        uint32_t rem = sh.bits[tid];
        cnt += __popc(rem);
        while (rem) {
            const int bit = __ffs(rem) - 1;
            rem &= rem - 1;
            const int off = tid * 32 + bit;
            const float s = sh.sc[off];
            if (!(s >= theta_score)) continue;
            const int p = (int)(w0 + off);
            const int q = atomicAdd(&sh.ccnt, 1);
            if (q < kScanCand) {
                sh.cs[q] = s;
                sh.cp[q] = p;
            }
            if (sp_before(s, p, ls[RS_MAX_TOPC - 1], lp[RS_MAX_TOPC - 1])) {
                float cs = s;
                int cp = p;
#pragma unroll
                for (int i = 0; i < RS_MAX_TOPC; ++i) {
                    if (sp_before(cs, cp, ls[i], lp[i])) {
                        const float ts = ls[i];
                        const int tp = lp[i];
                        ls[i] = cs;
                        lp[i] = cp;
                        cs = ts;
                        cp = tp;
                    }
                }
            }
        }
    }
    // the CTA's count; in a single window also every thread's position rank
    int cta_total = 0;
    rank = block_excl_scan(cnt, sh, &cta_total);  // single window: cnt = popc(bits[tid])
    // the CTA's best top_c: rank every buffered candidate by counting
    const int ncand = sh.ccnt;
    if (ncand <= kScanCand) {
        for (int e = tid; e < ncand; e += kScanThreads) {
            const float sv = sh.cs[e];
            const int pv = sh.cp[e];
            const int r = sp_rank(sv, pv, sh.cs, sh.cp, ncand);
            if (r < top_c) {
                sh.top_s[r] = sv;
                sh.top_p[r] = pv;
            }
        }
        if (tid == 0) sh.ntop = ncand < top_c ? ncand : top_c;
    } else {
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
                for (int i = 0; i < RS_MAX_TOPC - 1; ++i) {
                    ls[i] = ls[i + 1];
                    lp[i] = lp[i + 1];
                }
                ls[RS_MAX_TOPC - 1] = -INFINITY;
                lp[RS_MAX_TOPC - 1] = -1;
            }
        }
        if (tid == 0) sh.ntop = ntop;
    }

    // ---- the slice's global rank (pushed counts); positions in ascending order ----
    long long offset = 0, total = cta_total;
    if (!solo) {
        __syncthreads();  // this CTA's top list is complete
        cluster_wait();   // every CTA of the cluster is running
        if (tid < kScanCluster) *cluster.map_shared_rank(&sh.peer_cnt[crank], tid) = cta_total;
        if (tid < RS_MAX_TOPC) {
            *cluster.map_shared_rank(&sh.peer_s[crank][tid], 0) = sh.top_s[tid];
            *cluster.map_shared_rank(&sh.peer_p[crank][tid], 0) = sh.top_p[tid];
        }
        if (tid == 0) *cluster.map_shared_rank(&sh.peer_n[crank], 0) = sh.ntop;
        cluster_arrive_release();  // every push is visible after the wait
        cluster_wait();
        total = 0;
        for (int r = 0; r < kScanCluster; ++r) {
            const long long c = sh.peer_cnt[r];
            if (r < crank) offset += c;
            total += c;
        }
    } else {
        __syncthreads();
    }
    if (run && offset < pos_cap) {
        if (single) {
            uint32_t rem = lo < hi ? sh.bits[tid] : 0u;
            int i = 0;
            while (rem) {
                const int bit = __ffs(rem) - 1;
                rem &= rem - 1;
                const long long idx = offset + rank + i++;
                if (idx < pos_cap) pos[(long long)b * pos_cap + idx] = (int32_t)(lo + (long long)tid * 32 + bit);
            }
        } else {
            long long base = offset;
            for (long long w0 = lo; w0 < hi && base < pos_cap; w0 += kWin) {
                __syncthreads();  // the previous window is consumed
                stage_window(X, S, hi, hi, w0, sh);
                stage_wait();
                __syncthreads();
                window_bits(key, k, w0, plo, hi, sh);
                __syncthreads();
                uint32_t rem = sh.bits[tid];
                int wtotal = 0;
                const int r0 = block_excl_scan(__popc(rem), sh, &wtotal);
                int i = 0;
                while (rem) {
                    const int bit = __ffs(rem) - 1;
                    rem &= rem - 1;
                    const long long idx = base + r0 + i++;
                    if (idx < pos_cap) pos[(long long)b * pos_cap + idx] = (int32_t)(w0 + (long long)tid * 32 + bit);
                }
                base += wtotal;
            }
        }
    }

    // ---- CTA 0: merge the per-CTA lists, selection outputs ----
    if (crank == 0) {
        const long long stored = total < pos_cap ? total : pos_cap;
        for (long long i = stored + tid; i < pos_cap; i += kScanThreads) pos[(long long)b * pos_cap + i] = -1;
        if (total > pos_cap) st |= RS_ST_TRUNCATED;
        // the cluster's candidates (up to kScanCluster * RS_MAX_TOPC), ranked by counting
        float *ms = sh.cs;  // reused: the CTA's own buffer is no longer needed
        int *mp = sh.cp;
        int nm = 0;
        if (solo) {
            nm = sh.ntop;
            for (int q = tid; q < nm; q += kScanThreads) {
                ms[q] = sh.top_s[q];
                mp[q] = sh.top_p[q];
            }
        } else {
            for (int r = 0; r < kScanCluster; ++r) {
                const int n = sh.peer_n[r];
                if (tid < n) {
                    ms[nm + tid] = sh.peer_s[r][tid];
                    mp[nm + tid] = sh.peer_p[r][tid];
                }
                nm += n;
            }
        }
        __syncthreads();
        if (tid < nm) {
            const int r = sp_rank(ms[tid], mp[tid], ms, mp, nm);
            if (r < top_c) sh.sel[r] = mp[tid];
        }
        if (tid == 0) sh.ntop = nm < top_c ? nm : top_c;
        __syncthreads();
        const int nsel = sh.ntop;
        for (int i = tid; i < top_c * span_len; i += kScanThreads) {
            const int c = i / span_len, j = i - c * span_len;
            int v = -1;
            if (c < nsel) {
                const long long p = sh.sel[c];
                long long len = t - 1 - p;
                if (len > span_len) len = span_len;
                // solo: X[p + 1 + j], p + 1 + j <= t - 1, is staged at tok[kHalo + p + 1 + j]
                if (j < len) v = solo ? sh.tok[kHalo + p + 1 + j] : __ldg(X + p + 1 + j);
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
    static int attr_done[64] = {0};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_done[dev]) {
        cudaError_t e = cudaFuncSetAttribute(match_scan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)sizeof(ScanShared));
        if (e != cudaSuccess) {
            set_error("rs_match_scan: cudaFuncSetAttribute: %s", cudaGetErrorString(e));
            return RS_ERR_CUDA;
        }
        attr_done[dev] = 1;
    }
    launch_pdl(match_scan_kernel, dim3(kScanCluster, B), dim3(kScanThreads), sizeof(ScanShared),
        (cudaStream_t)stream, tokens, tok_off, k_star, gate_ok, scores, p.theta_score, p.top_c, p.span_len,
        pos_cap, count, pos, sel_pos, sel_len, spans, n_sel, status);
    RS_CHECK_LAUNCH("rs_match_scan");
    return RS_OK;
}
