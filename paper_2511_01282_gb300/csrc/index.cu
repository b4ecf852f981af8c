// index.cu -- an inverted index over the committed token buffers, kept up to
// date step by step, and the retrieval of Section 3.3 answered from it
// (rs_match_index_build, rs_match_index_append, rs_match_scan_indexed).  The
// two queries Algorithm 1 asks of its suffix automaton -- Contains(key) and
// RetrievePositions(key), key = the buffer's last k <= RS_MAX_L tokens -- are
// answered exactly from the ascending list of positions holding the key's
// last token: each is a candidate, verified against the other k - 1 key
// tokens.  Algorithm 1's Update (the step's committed tokens join the index)
// is rs_match_index_append.  A query touches O(occurrences of one token)
// instead of O(t); an append touches O(appended tokens).
//
// Layout of the index (per request b, sizes from rs_match_index_bytes):
//   start[b][0 .. V+1]  bucket offsets: the positions holding token v are
//                       bucket[start[v] .. start[v] + len[v]) in ascending
//                       order; ids outside [0, V) share bucket V
//                       (verification compares the real tokens).  Bucket v
//                       has room for count_v + count_v / 4 + 2 entries
//                       (count_v: occurrences at build time);
//   len[b][0 .. V]      entries in each bucket;
//   list (per request, at base[b]): kOvf overflow slots, then the buckets.
//                       A position whose bucket is full goes to the overflow
//                       list (ascending; all of a token's overflow entries
//                       are newer than its bucket entries);
//   built[b]            positions 0 .. built[b] - 1 are in the index;
//                       later ones (tokens appended and not yet indexed, or
//                       left out when the overflow list was full) are tested
//                       one by one (a linear tail).
// base[b] = tok_off[b] + tok_off[b] / 4 + b (2 (V + 1) + kOvf) at build time:
// request b's share is at least t_b + t_b / 4 + 2 (V + 1) + kOvf slots, which
// holds every bucket's room (sum of count_v / 4 <= t_b / 4).
//
// Build: every token's key (request, bucket) is sorted with a stable LSD
// radix sort (8-bit digits; per 4096-key tile a histogram, a two-level scan
// of the digit x tile counts, then a stable scatter that ranks each key within
// its tile by warp match and per-warp digit counters), so every bucket's
// positions come out ascending; a last pass places each sorted position at
// its bucket's start plus its rank.  All of it is parallel over the tokens
// of all requests.
// Append: one CTA per request takes the new positions in rounds of 256; each
// position's rank among the round's positions of its bucket gives its slot
// after the bucket's entries; full buckets spill to the overflow list in
// position order; if that is full too, indexing stops at the first such
// position (it and every later one stay in the linear tail, and the status
// word says so).
// Query: one CTA per request walks the candidates in rounds of 1024 (bucket,
// overflow list, then tail), verifies them, writes matches at their ascending
// rank (block scan of the round's hits) and ranks the matches that clear
// theta_score by counting, as the scan does.
#include <math.h>

#include <algorithm>

#include "common.cuh"

namespace rs {
namespace {

constexpr int kIdxThreads = 1024;
constexpr int kQryThreads = 256;
constexpr int kQryRound = 1024;          // candidates per query round (4 per thread)
constexpr int kQryCand = 256;            // matches ranked from the shared buffer
constexpr int kOvf = 4096;               // overflow slots per request
constexpr int kRadixBins = 256;          // 8-bit digits
constexpr int kTile = 4096;              // keys per radix tile
constexpr int kRadixThreads = 256;       // 8 warps x 512 keys per tile
constexpr int kAppThreads = 256;         // positions per append round

struct IndexView {
    int32_t *valid;         // 1 when the build's offsets were consistent (else the index holds nothing)
    int64_t *built, *base;  // per request: positions indexed, first list slot
    int32_t *ovf_n;         // per request: overflow entries
    int32_t *start;         // [B][V + 2]
    int32_t *len;           // [B][V + 1]
    int32_t *list;
    // build scratch
    int32_t *sstart;        // [B][V + 1]: exclusive prefix of the bucket counts
    uint32_t *key[2];
    int32_t *val[2];
    int32_t *hist;          // [kRadixBins][ntiles]
    int32_t *dtot;          // [kRadixBins]
};

inline long long list_slots(int B, int V, long long t_total) {
    return t_total + t_total / 4 + (long long)B * (2ll * (V + 1) + kOvf);
}
inline long long n_tiles(long long t_total) { return (t_total + kTile - 1) / kTile; }

// Carves the index (and its build scratch) out of `base`; returns the bytes used.
inline size_t carve_index(void *base, int B, int V, long long t_total, IndexView *v) {
    Carve cv(base);
    v->valid = cv.take<int32_t>(1);
    v->built = cv.take<int64_t>((size_t)B);
    v->base = cv.take<int64_t>((size_t)B);
    v->ovf_n = cv.take<int32_t>((size_t)B);
    v->start = cv.take<int32_t>((size_t)B * (V + 2));
    v->len = cv.take<int32_t>((size_t)B * (V + 1));
    v->list = cv.take<int32_t>((size_t)list_slots(B, V, t_total));
    v->sstart = cv.take<int32_t>((size_t)B * (V + 1));
    v->key[0] = cv.take<uint32_t>((size_t)t_total);
    v->key[1] = cv.take<uint32_t>((size_t)t_total);
    v->val[0] = cv.take<int32_t>((size_t)t_total);
    v->val[1] = cv.take<int32_t>((size_t)t_total);
    v->hist = cv.take<int32_t>((size_t)kRadixBins * n_tiles(t_total));
    v->dtot = cv.take<int32_t>((size_t)kRadixBins);
    return cv.used();
}
inline size_t index_bytes(int B, int V, long long t_total) {
    IndexView v;
    return carve_index(nullptr, B, V, t_total, &v);
}
// bits of a sort key (request, bucket): buckets 0 .. V, requests 0 .. B - 1
inline int bits_for(long long n) {  // smallest b with n < 2^b
    int b = 0;
    while (b < 63 && (1ll << b) <= n) ++b;
    return b;
}

__device__ __forceinline__ int bucket_of(int tok, int V) { return (tok >= 0 && tok < V) ? tok : V; }
__device__ __forceinline__ int room_of(int count) { return count + count / 4 + 2; }

// (0) the build's offsets: tok_off[0] = 0, ascending, tok_off[B] = t_total;
// every later build kernel does nothing unless they are
__global__ void __launch_bounds__(256)
index_check(const int64_t *__restrict__ tok_off, int B, long long t_total, IndexView ix) {
    pdl_enter();
    __shared__ int s_bad;
    if (threadIdx.x == 0) s_bad = tok_off[0] != 0 || tok_off[B] != t_total;
    __syncthreads();
    for (int b = threadIdx.x; b < B; b += blockDim.x)
        if (tok_off[b + 1] < tok_off[b]) s_bad = 1;
    __syncthreads();
    if (threadIdx.x == 0) *ix.valid = s_bad ? 0 : 1;
}

// (1) per request: zero the bucket counts, record the request's extent
__global__ void __launch_bounds__(256)
index_init(const int64_t *__restrict__ tok_off, int V, IndexView ix) {
    pdl_enter();
    if (!*ix.valid) return;
    const int b = blockIdx.y;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < V + 1; i += stride)
        ix.len[(long long)b * (V + 1) + i] = 0;
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        const long long o = tok_off[b];
        ix.built[b] = tok_off[b + 1] - o;
        ix.base[b] = o + o / 4 + (long long)b * (2ll * (V + 1) + kOvf);
        ix.ovf_n[b] = 0;
    }
}

// (2) count every bucket and write each token's sort key (request, bucket)
// and its global position
__global__ void __launch_bounds__(256)
index_count(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off, int V, int vbits,
            IndexView ix) {
    pdl_enter();
    if (!*ix.valid) return;
    const int b = blockIdx.y;
    int32_t *cnt = ix.len + (long long)b * (V + 1);
    const long long t0 = tok_off[b], t = tok_off[b + 1] - t0;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < t; i += stride) {
        const int bk = bucket_of(tokens[t0 + i], V);
        atomicAdd(&cnt[bk], 1);
        ix.key[0][t0 + i] = ((uint32_t)b << vbits) | (uint32_t)bk;
        ix.val[0][t0 + i] = (int32_t)(t0 + i);
    }
}

// (3) per request: bucket starts (prefix of the rooms) and the sorted starts
// (prefix of the counts); len keeps the counts.  Each thread takes kOffPer
// consecutive buckets, so one round of the block covers 8192 of them.
constexpr int kOffPer = 8;
__global__ void __launch_bounds__(kIdxThreads)
index_offsets(int V, IndexView ix) {
    pdl_enter();
    if (!*ix.valid) return;
    __shared__ int s_w[2][kIdxThreads / 32];
    __shared__ int s_carry[2];
    const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int32_t *cnt = ix.len + (long long)b * (V + 1);
    int32_t *start = ix.start + (long long)b * (V + 2);
    int32_t *sstart = ix.sstart + (long long)b * (V + 1);
    if (threadIdx.x < 2) s_carry[threadIdx.x] = 0;
    __syncthreads();
    for (int base = 0; base < V + 1; base += kIdxThreads * kOffPer) {
        const int i0 = base + threadIdx.x * kOffPer;
        int c[kOffPer];
        int r0 = 0, r1 = 0;  // this thread's rooms and counts
#pragma unroll
        for (int q = 0; q < kOffPer; ++q) {
            c[q] = i0 + q < V + 1 ? cnt[i0 + q] : 0;
            r0 += i0 + q < V + 1 ? room_of(c[q]) : 0;
            r1 += c[q];
        }
        int x0 = r0, x1 = r1;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y0 = __shfl_up_sync(0xffffffffu, x0, o), y1 = __shfl_up_sync(0xffffffffu, x1, o);
            if (lane >= o) {
                x0 += y0;
                x1 += y1;
            }
        }
        if (lane == 31) {
            s_w[0][warp] = x0;
            s_w[1][warp] = x1;
        }
        __syncthreads();
        int b0 = 0, b1 = 0, t0s = 0, t1s = 0;
        for (int w = 0; w < kIdxThreads / 32; ++w) {
            b0 += w < warp ? s_w[0][w] : 0;
            b1 += w < warp ? s_w[1][w] : 0;
            t0s += s_w[0][w];
            t1s += s_w[1][w];
        }
        int e0 = s_carry[0] + b0 + x0 - r0, e1 = s_carry[1] + b1 + x1 - r1;
#pragma unroll
        for (int q = 0; q < kOffPer; ++q) {
            if (i0 + q < V + 1) {
                start[i0 + q] = e0;
                sstart[i0 + q] = e1;
                e0 += room_of(c[q]);
                e1 += c[q];
            }
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            s_carry[0] += t0s;
            s_carry[1] += t1s;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) start[V + 1] = s_carry[0];
}

// (4) radix sort passes: tile histograms ...
__global__ void __launch_bounds__(kRadixThreads)
radix_hist(const uint32_t *__restrict__ key, long long N, int shift, long long ntiles, int32_t *__restrict__ hist,
           const int32_t *__restrict__ valid) {
    pdl_enter();
    if (!*valid) return;
    __shared__ int cnt[kRadixBins];
    const long long tile = blockIdx.x;
    cnt[threadIdx.x] = 0;
    __syncthreads();
    for (int e = threadIdx.x; e < kTile; e += kRadixThreads) {
        const long long i = tile * kTile + e;
        if (i < N) atomicAdd(&cnt[(key[i] >> shift) & (kRadixBins - 1)], 1);
    }
    __syncthreads();
    hist[(long long)threadIdx.x * ntiles + tile] = cnt[threadIdx.x];
}

// ... each digit's total over the tiles ...
__global__ void __launch_bounds__(kRadixThreads)
radix_total(const int32_t *__restrict__ hist, long long ntiles, int32_t *__restrict__ dtot,
            const int32_t *__restrict__ valid) {
    pdl_enter();
    if (!*valid) return;
    __shared__ int s_w[kRadixThreads / 32];
    const int d = blockIdx.x;
    int sum = 0;
    for (long long t = threadIdx.x; t < ntiles; t += kRadixThreads) sum += hist[(long long)d * ntiles + t];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if ((threadIdx.x & 31) == 0) s_w[threadIdx.x >> 5] = sum;
    __syncthreads();
    if (threadIdx.x == 0) {
        int tot = 0;
        for (int w = 0; w < kRadixThreads / 32; ++w) tot += s_w[w];
        dtot[d] = tot;
    }
}

// ... (digit, tile) offsets: the digits below d, then the tiles before t ...
__global__ void __launch_bounds__(kRadixThreads)
radix_offsets(int32_t *__restrict__ hist, long long ntiles, const int32_t *__restrict__ dtot,
              const int32_t *__restrict__ valid) {
    pdl_enter();
    if (!*valid) return;
    __shared__ int s_w[kRadixThreads / 32];
    __shared__ int s_carry;
    const int d = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        int c = 0;
        for (int e = 0; e < d; ++e) c += dtot[e];
        s_carry = c;
    }
    __syncthreads();
    for (long long base = 0; base < ntiles; base += kRadixThreads) {
        const long long t = base + threadIdx.x;
        const int v = t < ntiles ? hist[(long long)d * ntiles + t] : 0;
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) s_w[warp] = x;
        __syncthreads();
        int before = 0, sum = 0;
        for (int w = 0; w < kRadixThreads / 32; ++w) {
            before += w < warp ? s_w[w] : 0;
            sum += s_w[w];
        }
        if (t < ntiles) hist[(long long)d * ntiles + t] = s_carry + before + x - v;
        __syncthreads();
        if (threadIdx.x == 0) s_carry += sum;
        __syncthreads();
    }
}

// ... and the stable scatter: warp w takes keys w*512 .. w*512 + 511 of the
// tile, 32 at a time; a key's rank is the count of equal digits before it in
// the tile (earlier warps, earlier rounds of its warp, lower lanes of its round)
__global__ void __launch_bounds__(kRadixThreads)
radix_scatter(const uint32_t *__restrict__ kin, const int32_t *__restrict__ vin, uint32_t *__restrict__ kout,
              int32_t *__restrict__ vout, long long N, int shift, long long ntiles, const int32_t *__restrict__ hist,
              const int32_t *__restrict__ valid) {
    pdl_enter();
    if (!*valid) return;
    constexpr int kWarps = kRadixThreads / 32;
    constexpr int kRounds = kTile / kRadixThreads;
    __shared__ int wcnt[kWarps][kRadixBins];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const long long tile = blockIdx.x;
    for (int i = threadIdx.x; i < kWarps * kRadixBins; i += kRadixThreads) (&wcnt[0][0])[i] = 0;
    __syncthreads();
    uint32_t k[kRounds];
    int v[kRounds], rk[kRounds], dg[kRounds];
    const unsigned lt = (1u << lane) - 1u;
#pragma unroll
    for (int q = 0; q < kRounds; ++q) {
        const long long i = tile * kTile + warp * (kTile / kWarps) + q * 32 + lane;
        const bool ok = i < N;
        k[q] = ok ? kin[i] : 0u;
        v[q] = ok ? vin[i] : 0;
        dg[q] = ok ? (int)((k[q] >> shift) & (kRadixBins - 1)) : kRadixBins + lane;  // padding: a digit of its own
        const unsigned peers = __match_any_sync(0xffffffffu, dg[q]);
        const int base = ok ? wcnt[warp][dg[q]] : 0;
        __syncwarp();
        if (ok && (peers & lt) == 0) wcnt[warp][dg[q]] = base + __popc(peers);
        __syncwarp();
        rk[q] = ok ? base + __popc(peers & lt) : -1;
    }
    __syncthreads();
    {  // exclusive prefix of each digit's counts over the warps
        const int d = threadIdx.x;
        int run = 0;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const int c = wcnt[w][d];
            wcnt[w][d] = run;
            run += c;
        }
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kRounds; ++q) {
        if (rk[q] < 0) continue;
        const long long dst = (long long)hist[(long long)dg[q] * ntiles + tile] + wcnt[warp][dg[q]] + rk[q];
        kout[dst] = k[q];
        vout[dst] = v[q];
    }
}

// (5) each sorted position into its bucket: its rank among the request's
// positions of that bucket is its sorted index minus the bucket's sorted start
__global__ void __launch_bounds__(256)
index_place(const uint32_t *__restrict__ key, const int32_t *__restrict__ val, long long N,
            const int64_t *__restrict__ tok_off, int V, int vbits, IndexView ix) {
    pdl_enter();
    if (!*ix.valid) return;
    const long long stride = (long long)gridDim.x * blockDim.x;
    const uint32_t vmask = (vbits >= 32) ? 0xffffffffu : ((1u << vbits) - 1u);
    for (long long j = blockIdx.x * (long long)blockDim.x + threadIdx.x; j < N; j += stride) {
        const uint32_t kk = key[j];
        const int b = (int)(vbits >= 32 ? 0 : (kk >> vbits));
        const int bk = (int)(kk & vmask);
        const long long t0 = tok_off[b];
        const long long rank = j - t0 - ix.sstart[(long long)b * (V + 1) + bk];
        ix.list[ix.base[b] + kOvf + ix.start[(long long)b * (V + 2) + bk] + rank] = (int32_t)(val[j] - t0);
    }
}

// Append: the positions built[b] .. t_b - 1 of every request, in rounds of
// kAppThreads; see the file comment.
__global__ void __launch_bounds__(kAppThreads)
index_append(const int32_t *__restrict__ tokens, const int64_t *__restrict__ tok_off, int V, IndexView ix,
             int32_t *__restrict__ status) {
    pdl_enter();
    constexpr int kW = kAppThreads / 32;
    __shared__ int s_bk[kAppThreads];
    __shared__ unsigned char s_ok[kAppThreads];  // in the index (p < cut) and in its bucket
    __shared__ int s_w[kW];
    __shared__ long long s_cut;
    __shared__ int s_novf;
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const long long t0 = tok_off[b], t = tok_off[b + 1] - t0;
    // an index whose build saw inconsistent offsets holds nothing, and the
    // buffers hold tok_off[B] tokens: otherwise nothing is read or written
    if (!*ix.valid || t0 < 0 || t < 0 || t0 + t > tok_off[gridDim.x]) {
        if (tid == 0 && status) status[b] = RS_ST_BAD_OFFSET;
        return;
    }
    const int32_t *X = tokens + t0;
    int32_t *start = ix.start + (long long)b * (V + 2);
    int32_t *len = ix.len + (long long)b * (V + 1);
    int32_t *ovf = ix.list + ix.base[b];
    int32_t *buckets = ovf + kOvf;
    long long built = ix.built[b];
    int novf = ix.ovf_n[b];
    bool full = false;
    for (long long r0 = built; r0 < t && !full; r0 += kAppThreads) {
        const long long p = r0 + tid;
        const bool valid = p < t;
        const int bk = valid ? bucket_of(X[p], V) : -1;
        s_bk[tid] = bk;
        if (tid == 0) s_cut = t;
        __syncthreads();
        int rank = 0;
        for (int j = 0; j < tid; ++j) rank += s_bk[j] == bk;
        const int lo = valid ? len[bk] : 0;
        const int room = valid ? start[bk + 1] - start[bk] : 0;
        const int slot = lo + rank;
        const bool inb = valid && slot < room;
        const bool ov = valid && !inb;
        // overflow ranks in position order
        int x = ov ? 1 : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) s_w[warp] = x;
        __syncthreads();
        int before = 0, nov = 0;
        for (int w = 0; w < kW; ++w) {
            before += w < warp ? s_w[w] : 0;
            nov += s_w[w];
        }
        const int oslot = novf + before + x - (ov ? 1 : 0);
        if (ov && oslot >= kOvf) atomicMin(&s_cut, p);  // the first position with no room anywhere
        __syncthreads();
        const long long cut = s_cut;
        const bool in = valid && p < cut;
        s_ok[tid] = (unsigned char)(in && inb);
        if (in && inb) buckets[start[bk] + slot] = (int32_t)p;
        if (in && ov) ovf[oslot] = (int32_t)p;
        if (tid == 0) s_novf = 0;
        __syncthreads();
        // the last indexed position of a bucket in this round sets its length
        if (in && inb) {
            bool last = true;
            for (int j = tid + 1; j < kAppThreads; ++j)
                if (s_bk[j] == bk && s_ok[j]) last = false;
            if (last) len[bk] = slot + 1;
        }
        if (in && ov) atomicAdd(&s_novf, 1);
        __syncthreads();
        novf += s_novf;
        if (cut < t) {
            built = cut;
            full = true;
        } else {
            built = r0 + kAppThreads < t ? r0 + kAppThreads : t;
        }
        __syncthreads();  // s_bk, s_ok, s_cut reused by the next round
    }
    if (tid == 0) {
        ix.built[b] = built;
        ix.ovf_n[b] = novf;
        if (status) status[b] = built < t ? RS_ST_TRUNCATED : 0;
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
    // an index whose build saw inconsistent offsets holds nothing, and the
    // buffers hold tok_off[B] tokens: otherwise the request is not read
    const bool off_ok = *ix.valid && t0 >= 0 && t >= 0 && t0 + t <= tok_off[gridDim.x];
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
    if (run && tid < k) s_key[tid] = X[t - k + tid];
    if (tid == 0) s_ccnt = 0;
    __syncthreads();
    int key[RS_MAX_L];
#pragma unroll
    for (int i = 0; i < RS_MAX_L; ++i) key[i] = (run && i < k) ? s_key[i] : 0;
    // candidates, ascending: the bucket of the key's last token, the overflow
    // list (every token's overflow entries are newer than its bucket's), then
    // the positions not indexed (built .. t - 2)
    long long nb = 0, no = 0, tail0 = t;
    const int32_t *blist = nullptr, *olist = nullptr;
    if (run) {
        const int bk = bucket_of(key[k - 1], V);
        olist = ix.list + ix.base[b];
        blist = olist + kOvf + ix.start[(long long)b * (V + 2) + bk];
        nb = ix.len[(long long)b * (V + 1) + bk];
        no = ix.ovf_n[b];
        const long long built = ix.built[b];
        tail0 = built < t ? built : t;
    }
    const long long nt = run ? (t - 1) - tail0 : 0;  // tail: positions tail0 .. t-2
    const long long ncand = nb + no + (nt > 0 ? nt : 0);

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
            if (c < nb) cp[q] = blist[c];
            else if (c < nb + no) cp[q] = olist[c - nb];
            else if (c < ncand) cp[q] = (int)(tail0 + (c - nb - no));
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

static rs_status check_index(const char *who, int B, int V, int64_t t_total, const void *index,
                             size_t index_bytes_avail) {
    RS_CHECK_ARG(B >= 0 && B <= 65535, "%s: B=%d outside [0, 65535]", who, B);
    RS_CHECK_ARG(V >= 1 && V < (1 << 30), "%s: V=%d outside [1, 2^30)", who, V);
    RS_CHECK_ARG(t_total >= 0 && t_total < (1ll << 31), "%s: t_total outside [0, 2^31)", who);
    if (bits_for(V) + bits_for(B > 0 ? B - 1 : 0) > 32) {
        set_error("%s: B=%d requests with V=%d need more than 32 key bits", who, B, V);
        return RS_ERR_UNSUPPORTED;
    }
    const size_t need = index_bytes(B, V, t_total);
    if (index_bytes_avail < need || !index) {
        set_error("%s: index %zu bytes < %zu required", who, index_bytes_avail, need);
        return RS_ERR_CAPACITY;
    }
    return RS_OK;
}

extern "C" rs_status rs_match_index_build(const int32_t *tokens, const int64_t *tok_off, int B, int V,
                                          int64_t t_total, void *index, size_t index_bytes_avail, void *stream) {
    clear_error();
    const rs_status e = check_index("rs_match_index_build", B, V, t_total, index, index_bytes_avail);
    if (e != RS_OK) return e;
    RS_CHECK_ARG(B == 0 || (tokens && tok_off) || t_total == 0, "rs_match_index_build: null pointer");
    if (B == 0) return RS_OK;
    cudaStream_t st = (cudaStream_t)stream;
    IndexView ix;
    carve_index(index, B, V, t_total, &ix);
    const int vbits = bits_for(V);
    const int keybits = vbits + bits_for(B - 1);
    launch_pdl(index_check, dim3(1), dim3(256), 0, st, tok_off, B, (long long)t_total, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/check");
    const unsigned zx = (unsigned)std::min<long long>((V + 1 + 255) / 256, 64);
    launch_pdl(index_init, dim3(zx, B), dim3(256), 0, st, tok_off, V, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/init");
    const unsigned cx = (unsigned)std::max<long long>(1, std::min<long long>((t_total / B + 1023) / 1024, 256));
    launch_pdl(index_count, dim3(cx, B), dim3(256), 0, st, tokens, tok_off, V, vbits, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/count");
    launch_pdl(index_offsets, dim3(B), dim3(kIdxThreads), 0, st, V, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/offsets");
    if (t_total == 0) return RS_OK;
    // stable LSD radix sort of the (request, bucket) keys, 8 bits per pass
    const long long N = t_total, nt = n_tiles(t_total);
    int cur = 0;
    for (int shift = 0; shift < keybits; shift += 8, cur ^= 1) {
        launch_pdl(radix_hist, dim3((unsigned)nt), dim3(kRadixThreads), 0, st, ix.key[cur], N, shift, nt, ix.hist,
                   ix.valid);
        RS_CHECK_LAUNCH("rs_match_index_build/radix_hist");
        launch_pdl(radix_total, dim3(kRadixBins), dim3(kRadixThreads), 0, st, ix.hist, nt, ix.dtot, ix.valid);
        RS_CHECK_LAUNCH("rs_match_index_build/radix_total");
        launch_pdl(radix_offsets, dim3(kRadixBins), dim3(kRadixThreads), 0, st, ix.hist, nt, ix.dtot, ix.valid);
        RS_CHECK_LAUNCH("rs_match_index_build/radix_offsets");
        launch_pdl(radix_scatter, dim3((unsigned)nt), dim3(kRadixThreads), 0, st, ix.key[cur], ix.val[cur],
                   ix.key[cur ^ 1], ix.val[cur ^ 1], N, shift, nt, ix.hist, ix.valid);
        RS_CHECK_LAUNCH("rs_match_index_build/radix_scatter");
    }
    const unsigned px = (unsigned)std::min<long long>((N + 255) / 256, 148ll * 16);
    launch_pdl(index_place, dim3(px), dim3(256), 0, st, ix.key[cur], ix.val[cur], N, tok_off, V, vbits, ix);
    RS_CHECK_LAUNCH("rs_match_index_build/place");
    return RS_OK;
}

extern "C" rs_status rs_match_index_append(const int32_t *tokens, const int64_t *tok_off, int B, int V,
                                           int64_t t_total, void *index, size_t index_bytes_avail, int32_t *status,
                                           void *stream) {
    clear_error();
    const rs_status e = check_index("rs_match_index_append", B, V, t_total, index, index_bytes_avail);
    if (e != RS_OK) return e;
    RS_CHECK_ARG(B == 0 || (tokens && tok_off), "rs_match_index_append: null pointer");
    if (B == 0) return RS_OK;
    IndexView ix;
    carve_index(index, B, V, t_total, &ix);
    launch_pdl(index_append, dim3(B), dim3(kAppThreads), 0, (cudaStream_t)stream, tokens, tok_off, V, ix, status);
    RS_CHECK_LAUNCH("rs_match_index_append");
    return RS_OK;
}

extern "C" rs_status rs_match_scan_indexed(const int32_t *tokens, const int64_t *tok_off, int B,
                                           const int32_t *k_star, const uint8_t *gate_ok, const float *scores,
                                           rs_params p, int pos_cap, int32_t *count, int32_t *pos,
                                           int32_t *sel_pos, int32_t *sel_len, int32_t *spans, int32_t *n_sel,
                                           int32_t *status, int V, int64_t t_total, const void *index,
                                           size_t index_bytes_avail, void *stream) {
    clear_error();
    const rs_status e = check_index("rs_match_scan_indexed", B, V, t_total, index, index_bytes_avail);
    if (e != RS_OK) return e;
    RS_CHECK_ARG(pos_cap >= 0, "rs_match_scan_indexed: negative pos_cap");
    RS_CHECK_ARG(p.top_c >= 1 && p.top_c <= RS_MAX_TOPC, "rs_match_scan_indexed: top_c=%d outside [1, %d]",
                 p.top_c, RS_MAX_TOPC);
    RS_CHECK_ARG(p.span_len >= 1 && p.span_len <= RS_MAX_SPAN, "rs_match_scan_indexed: span_len=%d outside [1, %d]",
                 p.span_len, RS_MAX_SPAN);
    RS_CHECK_ARG(B == 0 || (tokens && tok_off && k_star && scores && count && sel_pos && sel_len && spans &&
                            n_sel && status && (pos || pos_cap == 0)),
                 "rs_match_scan_indexed: null pointer");
    if (B == 0) return RS_OK;
    IndexView ix;
    carve_index(const_cast<void *>(index), B, V, t_total, &ix);
    launch_pdl(index_query, dim3(B), dim3(kQryThreads), 0, (cudaStream_t)stream, tokens, tok_off, V, k_star,
        gate_ok, scores, p.theta_score, p.top_c, p.span_len, pos_cap, ix, count, pos, sel_pos, sel_len, spans, n_sel,
        status);
    RS_CHECK_LAUNCH("rs_match_scan_indexed");
    return RS_OK;
}
