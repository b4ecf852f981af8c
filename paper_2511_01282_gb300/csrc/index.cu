// index.cu -- an inverted index over the committed token buffers, and the
// retrieval of Section 3.3 answered from it (rs_match_index_build,
// rs_match_scan_indexed).  The two queries Algorithm 1 asks of its suffix
// automaton -- Contains(key) and RetrievePositions(key), key = the buffer's
// last k <= RS_MAX_L tokens -- are answered exactly from the ascending list
// of positions holding the key's last token: each is a candidate, verified
// against the other k - 1 key tokens.  A query touches O(occurrences of one
// token) instead of O(t).
//
// Layout of the index (per request b, sizes from rs_match_index_bytes):
//   start[b][0 .. V+1]  bucket offsets: positions holding token v are
//                       list[b][start[v] .. start[v+1]); ids outside [0, V)
//                       share bucket V (verification compares real tokens);
//   fill[b][0 .. V]     build scratch (per-bucket fill counters);
//   list[b][...]        positions relative to the request's first token,
//                       ascending within a bucket (request b's lists start
//                       at base[b], its first token's offset at build time);
//   built[b]            how many of the request's tokens the index covers.
// Positions at or after built[b] (tokens appended since the build) are
// tested one by one (a linear tail).
//
// Build: (1) bucket counts by atomic increments, (2) one CTA per request
// turns them into offsets with a block scan, (3) one CTA per request fills
// the buckets in position order, 1024 positions per round: the round's
// (token, position) pairs are sorted in shared memory, so each token's run is
// contiguous and ascending, and the run's base slot is its bucket offset plus
// the bucket's fill so far.
// Query: one CTA per request walks the candidates in rounds of 1024 (bucket,
// then tail), verifies them, writes matches at their ascending rank (block
// scan of the round's hits) and ranks the matches that clear theta_score by
// counting, as the scan does.
#include <math.h>

#include "common.cuh"

namespace rs {
namespace {

constexpr int kIdxThreads = 1024;
constexpr int kQryThreads = 256;
constexpr int kQryRound = 1024;          // candidates per query round (4 per thread)
constexpr int kQryCand = 256;            // matches ranked from the shared buffer

struct IndexView {
    int32_t *start, *fill, *list;
    int64_t *built, *base;  // per request: tokens covered, first list slot
};

inline IndexView carve_index(void *base, int B, int V, long long t_total) {
    Carve cv(base);
    IndexView v;
    v.built = cv.take<int64_t>((size_t)B);
    v.base = cv.take<int64_t>((size_t)B);
    v.start = cv.take<int32_t>((size_t)B * (V + 2));
    v.fill = cv.take<int32_t>((size_t)B * (V + 1));
    v.list = cv.take<int32_t>((size_t)t_total);
    return v;
}
inline size_t index_bytes(int B, int V, long long t_total) {
    Carve cv(nullptr);
    cv.take<int64_t>((size_t)B);
    cv.take<int64_t>((size_t)B);
    cv.take<int32_t>((size_t)B * (V + 2));
    cv.take<int32_t>((size_t)B * (V + 1));
    cv.take<int32_t>((size_t)t_total);
    return cv.used();
}

__device__ __forceinline__ int bucket_of(int tok, int V) { return (tok >= 0 && tok < V) ? tok : V; }

// (1) zero the counters of request blockIdx.y, then count its tokens
__global__ void __launch_bounds__(256)
index_count(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off, int V, IndexView ix) {
    pdl_enter();
    const int b = blockIdx.y;
    int32_t *cnt = ix.start + (long long)b * (V + 2);
    const long long t0 = tok_off[b], t = tok_off[b + 1] - t0;
    // counts live at cnt[v + 1]; cnt[0] stays 0 (exclusive scan in place later)
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < t; i += stride)
        atomicAdd(&cnt[bucket_of(tokens[t0 + i], V) + 1], 1);
}

__global__ void __launch_bounds__(256)
index_zero(const int64_t *__restrict__ tok_off, int V, IndexView ix) {
    pdl_enter();
    const int b = blockIdx.y;
    const long long n = V + 2;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += stride) {
        ix.start[(long long)b * (V + 2) + i] = 0;
        if (i < V + 1) ix.fill[(long long)b * (V + 1) + i] = 0;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        ix.built[b] = tok_off[b + 1] - tok_off[b];
        ix.base[b] = tok_off[b];
    }
}

// (2) inclusive scan of cnt[1 .. V+1] in place: start[v] = sum of counts below v
__global__ void __launch_bounds__(kIdxThreads)
index_offsets(int V, IndexView ix) {
    pdl_enter();
    __shared__ int s_w[kIdxThreads / 32];
    __shared__ int s_carry;
    const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int32_t *cnt = ix.start + (long long)b * (V + 2);
    if (threadIdx.x == 0) s_carry = 0;
    __syncthreads();
    for (int base = 1; base < V + 2; base += kIdxThreads) {
        const int i = base + threadIdx.x;
        const int v = i < V + 2 ? cnt[i] : 0;
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) s_w[warp] = x;
        __syncthreads();
        int before = 0, sum = 0;
        for (int w = 0; w < kIdxThreads / 32; ++w) {
            const int y = s_w[w];
            before += w < warp ? y : 0;
            sum += y;
        }
        const int incl = s_carry + before + x;
        if (i < V + 2) cnt[i] = incl;
        __syncthreads();
        if (threadIdx.x == 0) s_carry += sum;
        __syncthreads();
    }
}

// (3) fill the buckets in position order, one round of kIdxThreads positions at
// a time: sort the round's (bucket, position) keys, then each run of a bucket
// takes consecutive slots after the bucket's fill so far.
__global__ void __launch_bounds__(kIdxThreads)
index_fill(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off, int V, IndexView ix) {
    pdl_enter();
    __shared__ unsigned long long s_key[kIdxThreads];
    __shared__ int s_base[kIdxThreads];
    __shared__ int s_w[kIdxThreads / 32];
    const int b = blockIdx.x, tid = threadIdx.x;
    const long long t0 = tok_off[b], t = tok_off[b + 1] - t0;
    const int32_t *start = ix.start + (long long)b * (V + 2);
    int32_t *fill = ix.fill + (long long)b * (V + 1);
    int32_t *list = ix.list + t0;
    const int lane = tid & 31, warp = tid >> 5;
    for (long long r0 = 0; r0 < t; r0 += kIdxThreads) {
        const long long p = r0 + tid;
        // key = bucket (high 32 bits) : position within the round (low bits); padding sorts last
        s_key[tid] = p < t ? ((unsigned long long)(unsigned)bucket_of(tokens[t0 + p], V) << 32) | (unsigned)tid
                           : ~0ull;
        __syncthreads();
        for (int k = 2; k <= kIdxThreads; k <<= 1) {  // bitonic sort, ascending
            for (int j = k >> 1; j > 0; j >>= 1) {
                const int partner = tid ^ j;
                if (partner > tid) {
                    const unsigned long long a = s_key[tid], c = s_key[partner];
                    const bool up = (tid & k) == 0;
                    if ((a > c) == up) {
                        s_key[tid] = c;
                        s_key[partner] = a;
                    }
                }
                __syncthreads();
            }
        }
        const unsigned long long key = s_key[tid];
        const bool real = key != ~0ull;
        const int bk = (int)(key >> 32);
        const bool head = real && (tid == 0 || (int)(s_key[tid - 1] >> 32) != bk);
        // a run's head reads the bucket's slot base; the run's members follow it
        if (head) s_base[tid] = start[bk] + fill[bk];
        // each element's run head: the largest head index at or before it (max scan)
        int h = head ? tid : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, h, o);
            if (lane >= o) h = max(h, y);
        }
        if (lane == 31) s_w[warp] = h;
        __syncthreads();
        for (int w = 0; w < warp; ++w) h = max(h, s_w[w]);
        if (real) {
            list[s_base[h] + (tid - h)] = (int32_t)(r0 + (long long)(key & 0xffffffffu));
            // the run's last member advances the bucket's fill
            if (tid == kIdxThreads - 1 || (int)(s_key[tid + 1] >> 32) != bk || s_key[tid + 1] == ~0ull)
                fill[bk] += tid - h + 1;
        }
        __syncthreads();
    }
}

// (s, p) before (s2, p2): higher score first, then the more recent position
__device__ __forceinline__ bool sp_before(float s, int p, float s2, int p2) {
    return s > s2 || (s == s2 && p > p2);
}

__global__ void __launch_bounds__(kQryThreads)
index_query(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off, int V,
            const int32_t *__restrict__ k_star, const uint8_t *__restrict__ gate_ok,
            const float *__restrict__ scores, float theta_score, int top_c, int span_len, int pos_cap,
            IndexView ix, int32_t *__restrict__ count, int32_t *__restrict__ pos, int32_t *__restrict__ sel_pos,
            int32_t *__restrict__ sel_len, int32_t *__restrict__ spans, int32_t *__restrict__ n_sel,
            int32_t *__restrict__ status) {
    pdl_enter();
    constexpr int kPer = kQryRound / kQryThreads;
    __shared__ int s_key[RS_MAX_L];
    __shared__ int s_w[kQryThreads / 32];
    __shared__ float s_cs[kQryCand];
    __shared__ int s_cp[kQryCand];
    __shared__ int s_ccnt;
    __shared__ float s_bv[kQryThreads / 32];
    __shared__ int s_bp[kQryThreads / 32];
    __shared__ int s_sel[RS_MAX_TOPC];
    __shared__ int s_nsel;
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const long long t0 = tok_off[b];
    const long long t = tok_off[b + 1] - t0;
    const int32_t *X = tokens + t0;
    const float *S = scores + t0;
    const int k = k_star[b];
    int st = 0;
    bool run = k > 0 && (gate_ok == nullptr || gate_ok[b] != 0);
    if (run && k > RS_MAX_L) {
        st = RS_ST_TOO_LARGE;
        run = false;
    }
    if (run && (long long)k > t) run = false;
    if (run && tid < k) s_key[tid] = X[t - k + tid];
    if (tid == 0) s_ccnt = 0;
    __syncthreads();
    int key[RS_MAX_L];
#pragma unroll
    for (int i = 0; i < RS_MAX_L; ++i) key[i] = (run && i < k) ? s_key[i] : 0;
    // candidates: the bucket of the key's last token (positions < built), then the tail
    long long bs = 0, be = 0, tail0 = t;
    if (run) {
        const int bk = bucket_of(key[k - 1], V);
        const int32_t *start = ix.start + (long long)b * (V + 2);
        bs = start[bk];
        be = start[bk + 1];
        const long long built = ix.built[b];
        tail0 = built < t ? built : t;
    }
    const int32_t *blist = ix.list + (run ? ix.base[b] : 0);
    const long long nb = be - bs, nt = run ? (t - 1) - tail0 : 0;  // tail: positions tail0 .. t-2
    const long long ncand = nb + (nt > 0 ? nt : 0);

    float ls[RS_MAX_TOPC];
    int lp[RS_MAX_TOPC];
#pragma unroll
    for (int i = 0; i < RS_MAX_TOPC; ++i) {
        ls[i] = -INFINITY;
        lp[i] = -1;
    }
    long long total = 0;  // matches so far (the next match's rank)
    for (long long c0 = 0; c0 < ncand; c0 += kQryRound) {
        int cp[kPer];
        bool hit[kPer];
        int nh = 0;
#pragma unroll
        for (int q = 0; q < kPer; ++q) {  // candidate c0 + kPer * tid + q, in order
            const long long c = c0 + (long long)kPer * tid + q;
            cp[q] = -1;
            if (c < nb) cp[q] = blist[bs + c];
            else if (c < ncand) cp[q] = (int)(tail0 + (c - nb));
        }
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int p = cp[q];
            bool m = p >= k - 1 && (long long)p <= t - 2;
            if (m) {
                for (int i = 0; i < k; ++i) m = m && (X[p - i] == key[k - 1 - i]);
            }
            hit[q] = m;
            nh += m;
        }
        // ascending rank of this thread's hits in the round
        int x = nh;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) s_w[warp] = x;
        __syncthreads();
        int before = 0, sum = 0;
#pragma unroll
        for (int w = 0; w < kQryThreads / 32; ++w) {
            const int y = s_w[w];
            before += w < warp ? y : 0;
            sum += y;
        }
        __syncthreads();
        long long r = total + before + x - nh;
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            if (!hit[q]) continue;
            const int p = cp[q];
            if (r < pos_cap) pos[(long long)b * pos_cap + r] = p;
            ++r;
            const float s = S[p];
            if (!(s >= theta_score)) continue;
            const int slot = atomicAdd(&s_ccnt, 1);
            if (slot < kQryCand) {
                s_cs[slot] = s;
                s_cp[slot] = p;
            }
            if (sp_before(s, p, ls[RS_MAX_TOPC - 1], lp[RS_MAX_TOPC - 1])) {
                float cs = s;
                int cq = p;
#pragma unroll
                for (int i = 0; i < RS_MAX_TOPC; ++i)
                    if (sp_before(cs, cq, ls[i], lp[i])) {
                        const float ts = ls[i];
                        const int tq = lp[i];
                        ls[i] = cs;
                        lp[i] = cq;
                        cs = ts;
                        cq = tq;
                    }
            }
        }
        total += sum;
    }
    __syncthreads();
    // the best top_c: rank the buffered matches by counting, else merge the per-thread lists
    const int nc = s_ccnt;
    if (nc <= kQryCand) {
        for (int e = tid; e < nc; e += kQryThreads) {
            int rk = 0;
            for (int q = 0; q < nc; ++q) rk += sp_before(s_cs[q], s_cp[q], s_cs[e], s_cp[e]);
            if (rk < top_c) s_sel[rk] = s_cp[e];
        }
        if (tid == 0) s_nsel = nc < top_c ? nc : top_c;
    } else {
        int nsel = 0;
        for (int c = 0; c < top_c; ++c) {
            float hv = ls[0];
            int hp = lp[0];
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
                s_bv[warp] = hv;
                s_bp[warp] = hp;
            }
            __syncthreads();
            hv = s_bv[0];
            hp = s_bp[0];
            for (int w = 1; w < kQryThreads / 32; ++w)
                if (sp_before(s_bv[w], s_bp[w], hv, hp)) {
                    hv = s_bv[w];
                    hp = s_bp[w];
                }
            __syncthreads();
            if (hp < 0) break;
            if (tid == 0) s_sel[c] = hp;
            nsel = c + 1;
            if (lp[0] == hp) {  // the owner pops its head
#pragma unroll
                for (int i = 0; i < RS_MAX_TOPC - 1; ++i) {
                    ls[i] = ls[i + 1];
                    lp[i] = lp[i + 1];
                }
                ls[RS_MAX_TOPC - 1] = -INFINITY;
                lp[RS_MAX_TOPC - 1] = -1;
            }
        }
        if (tid == 0) s_nsel = nsel;
    }
    const long long stored = total < pos_cap ? total : pos_cap;
    for (long long i = stored + tid; i < pos_cap; i += kQryThreads) pos[(long long)b * pos_cap + i] = -1;
    __syncthreads();
    const int nsel = s_nsel;
    for (int i = tid; i < top_c * span_len; i += kQryThreads) {
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
        int sp = -1, sl = 0;
        if (tid < nsel) {
            sp = s_sel[tid];
            const long long len = t - 1 - sp;
            sl = (int)(len > span_len ? span_len : len);
        }
        sel_pos[(long long)b * top_c + tid] = sp;
        sel_len[(long long)b * top_c + tid] = sl;
    }
    if (tid == 0) {
        count[b] = (int32_t)total;
        n_sel[b] = nsel;
        status[b] = st | (total > pos_cap ? RS_ST_TRUNCATED : 0);
    }
}

}  // namespace
}  // namespace rs

using namespace rs;

extern "C" size_t rs_match_index_bytes(int B, int V, int64_t t_total) {
    if (B < 0 || V < 1 || t_total < 0) return 0;
    return index_bytes(B, V, t_total);
}

extern "C" rs_status rs_match_index_build(const int32_t *tokens, const int64_t *tok_off, int B, int V,
                                          int64_t t_total, void *index, size_t index_bytes_avail, void *stream) {
    clear_error();
    RS_CHECK_ARG(B >= 0 && B <= 65535, "rs_match_index_build: B=%d outside [0, 65535]", B);
    RS_CHECK_ARG(V >= 1 && V < (1 << 30), "rs_match_index_build: V=%d outside [1, 2^30)", V);
    RS_CHECK_ARG(t_total >= 0 && t_total < (1ll << 31), "rs_match_index_build: t_total outside [0, 2^31)");
    RS_CHECK_ARG(B == 0 || (tokens && tok_off) || t_total == 0, "rs_match_index_build: null pointer");
    const size_t need = index_bytes(B, V, t_total);
    if (index_bytes_avail < need || !index) {
        set_error("rs_match_index_build: index %zu bytes < %zu required", index_bytes_avail, need);
        return RS_ERR_CAPACITY;
    }
    if (B == 0) return RS_OK;
    cudaStream_t st = (cudaStream_t)stream;
    IndexView ix = carve_index(index, B, V, t_total);
    const unsigned zx = (unsigned)std::min<long long>((V + 2 + 255) / 256, 64);
    launch_pdl(index_zero, dim3(zx, B), dim3(256), 0, st, tok_off, V, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/zero");
    launch_pdl(index_count, dim3(16, B), dim3(256), 0, st, tokens, tok_off, V, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/count");
    launch_pdl(index_offsets, dim3(B), dim3(kIdxThreads), 0, st, V, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/offsets");
    launch_pdl(index_fill, dim3(B), dim3(kIdxThreads), 0, st, tokens, tok_off, V, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/fill");
    return RS_OK;
}

extern "C" rs_status rs_match_scan_indexed(const int32_t *tokens, const int64_t *tok_off, int B,
                                           const int32_t *k_star, const uint8_t *gate_ok, const float *scores,
                                           rs_params p, int pos_cap, int32_t *count, int32_t *pos,
                                           int32_t *sel_pos, int32_t *sel_len, int32_t *spans, int32_t *n_sel,
                                           int32_t *status, int V, int64_t t_total, const void *index,
                                           size_t index_bytes_avail, void *stream) {
    clear_error();
    RS_CHECK_ARG(B >= 0 && B <= 65535, "rs_match_scan_indexed: B=%d outside [0, 65535]", B);
    RS_CHECK_ARG(pos_cap >= 0, "rs_match_scan_indexed: negative pos_cap");
    RS_CHECK_ARG(p.top_c >= 1 && p.top_c <= RS_MAX_TOPC, "rs_match_scan_indexed: top_c=%d outside [1, %d]",
                 p.top_c, RS_MAX_TOPC);
    RS_CHECK_ARG(p.span_len >= 1 && p.span_len <= RS_MAX_SPAN, "rs_match_scan_indexed: span_len=%d outside [1, %d]",
                 p.span_len, RS_MAX_SPAN);
    RS_CHECK_ARG(V >= 1, "rs_match_scan_indexed: V must be >= 1");
    RS_CHECK_ARG(B == 0 || (tokens && tok_off && k_star && scores && count && sel_pos && sel_len && spans &&
                            n_sel && status && (pos || pos_cap == 0)),
                 "rs_match_scan_indexed: null pointer");
    const size_t need = index_bytes(B, V, t_total);
    if (index_bytes_avail < need || !index) {
        set_error("rs_match_scan_indexed: index %zu bytes < %zu required", index_bytes_avail, need);
        return RS_ERR_CAPACITY;
    }
    if (B == 0) return RS_OK;
    IndexView ix = carve_index(const_cast<void *>(index), B, V, t_total);
    launch_pdl(index_query, dim3(B), dim3(kQryThreads), 0, (cudaStream_t)stream, tokens, tok_off, V, k_star,
        gate_ok, scores, p.theta_score, p.top_c, p.span_len, pos_cap, ix, count, pos, sel_pos, sel_len, spans, n_sel,
        status);
    RS_CHECK_LAUNCH("rs_match_scan_indexed");
    return RS_OK;
}
