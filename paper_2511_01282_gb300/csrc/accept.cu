// accept.cu -- rs_accept: source-aware verification (Section 3.4, Eq. 6-7
// and the look-ahead tolerance procedure), longest accepted path and winner
// (Algorithm 1 l.13), EMA feedback (Eq. 4-5, Algorithm 1 l.15-22).
//
// Kernel 1 (accept_rows): three persistent CTAs per SM walk the (row,
// 8192-logit chunk) work items; each thread copies the next item's 32
// logits into a second shared-memory stage (cp.async) while it works on the
// current item from registers.  Per item the CTA produces the chunk's (max,
// sum e^(z - max)[, sum e^(z - max) (z - max)]) triple and its beta best
// (logit, id) pairs in the total order (logit desc, id asc).  The beta-th largest of a warp's 32 lane maxima (warp
// bitonic sort) bounds the chunk's beta-th largest logit from below, and so
// does the largest such bound over the warps; the few logits at or above it
// are appended to shared memory and one warp (rotating over items) ranks them
// by beta rounds of a "best after the previous winner" warp reduction (exact;
// with many ties at the bound every warp ranks its own logits and that warp
// merges the lists).
// No dynamic register indexing.
// Kernel 2 (accept_merge): one warp per row merges the chunk results into
// argmax, top-beta, log-sum-exp, the row's largest logit (workspace, for
// kernel 3) and (optionally) the row entropy.
// Kernel 3 (accept_decide): one CTA per request checks the tree, verifies
// model nodes (each thread walks its own root path over per-node match
// flags), runs the look-ahead procedure per chain (one thread per chain),
// picks the winner and updates the scores (one thread per selection).
#include <math.h>

#include <algorithm>

#include "common.cuh"
#include "sm100.cuh"

namespace rs {
namespace {

constexpr int kAccThreads = 256;
constexpr int kAccVpt = 32;
constexpr int kAccChunk = kAccThreads * kAccVpt;
constexpr int kNoId = 0x7fffffff;  // "no candidate": after every real (v, id)
constexpr int kCandCap = 64;        // per-warp candidate buffer (logits at or above the threshold)

struct VI {
    float v;
    int i;
};

__device__ __forceinline__ VI vi_best(VI a, VI b) { return vi_before(b.v, b.i, a.v, a.i) ? b : a; }

__device__ __forceinline__ VI vi_shfl(VI a, int o) {
    VI b;
    b.v = __shfl_xor_sync(0xffffffffu, a.v, o);
    b.i = __shfl_xor_sync(0xffffffffu, a.i, o);
    return b;
}

__device__ __forceinline__ VI warp_vi_best(VI a) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) a = vi_best(a, vi_shfl(a, o));
    return a;
}

// (max m, sum e^(z-m), sum e^(z-m) (z-m)) of a set of logits: the row's
// log-sum-exp is m + ln s and its entropy ln s - w / s.
struct MS {
    float m, s, w;
};

__device__ __forceinline__ MS ms_merge(MS a, MS b) {
    if (a.s == 0.f) return b;
    if (b.s == 0.f) return a;
    const float M = fmaxf(a.m, b.m);
    const float ca = __expf(a.m - M), cb = __expf(b.m - M);
    return MS{M, a.s * ca + b.s * cb, ca * (a.w + a.s * (a.m - M)) + cb * (b.w + b.s * (b.m - M))};
}

__device__ __forceinline__ MS ms_shfl(MS a, int o) {
    return MS{__shfl_xor_sync(0xffffffffu, a.m, o), __shfl_xor_sync(0xffffffffu, a.s, o),
              __shfl_xor_sync(0xffffffffu, a.w, o)};
}

// Bitonic sort of one float per lane within aligned groups of G lanes (a
// power of two <= 32), every group ending in descending order: lane g G + i
// holds the group's (i + 1)-th largest value.
template <int G>
__device__ __forceinline__ float group_sort_desc(float x, int lane) {
#pragma unroll
    for (int k = 2; k <= G; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
            const float y = __shfl_xor_sync(0xffffffffu, x, j);
            const bool desc = (k == G) || ((lane & k) == 0);
            const bool keep_max = ((lane & j) == 0) == desc;
            x = keep_max ? fmaxf(x, y) : fminf(x, y);
        }
    }
    return x;
}

// The warp maximum and the largest over the warp's G-lane groups of the
// group's beta-th largest lane value (beta <= G).
template <int G>
__device__ __forceinline__ void warp_max_and_bound(float mx, int lane, int beta, float *wmax, float *bound) {
    const float sorted = group_sort_desc<G>(mx, lane);
    float m = -INFINITY, t = -INFINITY;
#pragma unroll
    for (int g = 0; g < 32; g += G) {
        m = fmaxf(m, __shfl_sync(0xffffffffu, sorted, g));
        t = fmaxf(t, __shfl_sync(0xffffffffu, sorted, g + beta - 1));
    }
    *wmax = m;
    *bound = t;
}

// cp.async: per-thread asynchronous global -> shared copies.  A thread's
// wait_group only waits for its own copies, so no wait depends on another
// thread.
__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(sm100::smem_u32(smem)), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async4(void *smem, const void *gmem) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(sm100::smem_u32(smem)), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }

// Start copying the logits this thread will hold of work item `item` = (row,
// chunk) into `stage` (the same slots it later reads; ids >= V are skipped).
template <bool kVec>
__device__ __forceinline__ void fetch_item(const float *__restrict__ logits, int V, int nchunks, int item,
                                           float *stage) {
    const int r = item / nchunks;
    const int c0 = (item - r * nchunks) * kAccChunk;
    const float *row = logits + (long long)r * V;
    const int tid = threadIdx.x;
    if (kVec) {
#pragma unroll
        for (int j = 0; j < kAccVpt / 4; ++j) {
            const int off = (j * kAccThreads + tid) * 4;
            if (c0 + off < V) cp_async16(stage + off, row + c0 + off);  // V % 4 == 0: whole float4
        }
    } else {
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) {
            const int off = j * kAccThreads + tid;
            if (c0 + off < V) cp_async4(stage + off, row + c0 + off);
        }
    }
}

template <bool kVec>
__device__ __forceinline__ void read_item(const float *stage, int V, int c0, float (&v)[kAccVpt]) {
    const int tid = threadIdx.x;
    if (kVec) {
#pragma unroll
        for (int j = 0; j < kAccVpt / 4; ++j) {
            const int off = (j * kAccThreads + tid) * 4;
            float4 x = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
            if (c0 + off < V) x = *reinterpret_cast<const float4 *>(stage + off);
            v[4 * j + 0] = x.x;
            v[4 * j + 1] = x.y;
            v[4 * j + 2] = x.z;
            v[4 * j + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) {
            const int off = j * kAccThreads + tid;
            v[j] = c0 + off < V ? stage[off] : -INFINITY;
        }
    }
}

struct RowsShared {
    MS sms[kAccThreads / 32];
    float thr[kAccThreads / 32];
    VI wtop[kAccThreads / 32][RS_MAX_BETA];  // per-warp lists (tie fallback)
    VI cbuf[kCandCap];                       // the chunk's candidates
    int cnt;
};

// One work item on the logits in registers: the chunk's (max, sum e, sum e
// (z - max)) triple and its best beta candidates.
// `rw` is the warp that ranks the candidates and writes the item's results
// (rotated over items).  `sh` alternates between two copies over items, so no
// barrier is needed at the end: a copy is next written two items later, after
// every thread has passed the first barrier of the item in between.
template <bool kVec, bool kEnt>
__device__ __forceinline__ void rows_item(const float (&v)[kAccVpt], int V, int c0, int beta, int blk,
                                          VI *__restrict__ cand, MS *__restrict__ part, RowsShared &sh, int rw) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr float kL2E = 1.4426950408889634f;
    if (tid == 0) sh.cnt = 0;

    // logit id of register j (padding slots have ids >= V)
    auto id_of = [&](int j) -> int {
        if (kVec) return c0 + ((j >> 2) * kAccThreads + tid) * 4 + (j & 3);
        return c0 + j * kAccThreads + tid;
    };

    // lane maximum; the warp maximum and a lower bound on the chunk's beta-th
    // largest logit from the sorted lane maxima: the warp holds beta lane
    // maxima >= its beta-th largest, and each is a logit of the chunk.  Every lane exponentiates against the warp
    // maximum, so the warp's (max, sum e, sum e (z - max)) is a plain sum.
    float m8[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) m8[q] = fmaxf(fmaxf(v[q], v[q + 8]), fmaxf(v[q + 16], v[q + 24]));
    const float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                           fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
    float wmax, thr_w;
    warp_max_and_bound<32>(mx, lane, beta, &wmax, &thr_w);
    MS t{wmax, 0.f, 0.f};
    if (wmax != -INFINITY) {
        // base 2: u = (z - max) log2(e), e = 2^u; sum e (z - max) = ln 2 sum e u
        const float nb = -wmax * kL2E;
        float s4[4] = {0.f, 0.f, 0.f, 0.f};
        float w4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) {
            if (kEnt) {
                const float u = fmaxf(fmaf(v[j], kL2E, nb), -1e30f);  // -inf -> -1e30: e = 0, e u = 0
                const float e = sm100::ex2(u);
                s4[j & 3] += e;
                w4[j & 3] = fmaf(e, u, w4[j & 3]);
            } else {
                s4[j & 3] += sm100::ex2(fmaf(v[j], kL2E, nb));
            }
        }
        float ss = (s4[0] + s4[1]) + (s4[2] + s4[3]);
        float ww = (w4[0] + w4[1]) + (w4[2] + w4[3]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            ss += __shfl_xor_sync(0xffffffffu, ss, o);
            if (kEnt) ww += __shfl_xor_sync(0xffffffffu, ww, o);
        }
        t.s = ss;
        t.w = ww * 0.6931471805599453f;
    }
    if (lane == 0) {
        sh.sms[warp] = t;
        sh.thr[warp] = thr_w;
    }

    // ---- the chunk's best beta, exactly, in (logit desc, id asc) order ----
    // Only logits >= T = max over warps of the bounds can be in the chunk's
    // best beta; they are appended to one shared buffer and ranked by one
    // warp (each candidate's rank = the number of candidates before it).  If
    // ties overflow the buffer, every warp ranks its own logits and that warp
    // merges the eight lists instead.
    __syncthreads();
    float thr = sh.thr[0];
#pragma unroll
    for (int w = 1; w < kAccThreads / 32; ++w) thr = fmaxf(thr, sh.thr[w]);
    if (mx >= thr) {
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) {
            if (v[j] >= thr) {
                const int id = id_of(j);
                if (id < V) {
                    const int p = atomicAdd(&sh.cnt, 1);
                    if (p < kCandCap) sh.cbuf[p] = VI{v[j], id};
                }
            }
        }
    }
    __syncthreads();
    const int total = sh.cnt;
    if (total <= kCandCap) {
        if (warp == rw) {
            VI x0 = lane < total ? sh.cbuf[lane] : VI{-INFINITY, kNoId};
            VI x1 = lane + 32 < total ? sh.cbuf[lane + 32] : VI{-INFINITY, kNoId};
            int r0 = 0, r1 = 0;
            for (int q = 0; q < total; ++q) {
                const VI y = sh.cbuf[q];
                r0 += vi_before(y.v, y.i, x0.v, x0.i);
                r1 += vi_before(y.v, y.i, x1.v, x1.i);
            }
            if (lane < total && r0 < beta) cand[(long long)blk * beta + r0] = x0;
            if (lane + 32 < total && r1 < beta) cand[(long long)blk * beta + r1] = x1;
            if (lane >= total && lane < beta) cand[(long long)blk * beta + lane] = VI{-INFINITY, kNoId};
        }
    } else {
        VI prev{INFINITY, -1};
        for (int k = 0; k < beta; ++k) {
            VI best{-INFINITY, kNoId};
#pragma unroll
            for (int j = 0; j < kAccVpt; ++j) {
                const int id = id_of(j);
                if (id < V && vi_before(prev.v, prev.i, v[j], id) && vi_before(v[j], id, best.v, best.i))
                    best = VI{v[j], id};
            }
            best = warp_vi_best(best);
            prev = best;
            if (lane == 0) sh.wtop[warp][k] = best;
        }
        __syncthreads();
        if (warp == rw) {
            constexpr int kW = kAccThreads / 32;
            VI prevb{INFINITY, -1};
            for (int k = 0; k < beta; ++k) {
                VI best{-INFINITY, kNoId};
                for (int q = lane; q < kW * beta; q += 32) {
                    const VI x = sh.wtop[q / beta][q % beta];
                    if (x.i != kNoId && vi_before(prevb.v, prevb.i, x.v, x.i) &&
                        vi_before(x.v, x.i, best.v, best.i))
                        best = x;
                }
                best = warp_vi_best(best);
                prevb = best;
                if (lane == 0) cand[(long long)blk * beta + k] = best;
            }
        }
    }
    if (warp == rw) {  // the eight warp triples, merged as a 3-level tree
        MS a = lane < kAccThreads / 32 ? sh.sms[lane] : MS{-INFINITY, 0.f, 0.f};
#pragma unroll
        for (int o = 4; o > 0; o >>= 1) a = ms_merge(a, ms_shfl(a, o));
        if (lane == 0) part[blk] = a;
    }
}

// Persistent over work items: while a CTA works on item i, the copies of
// item i + gridDim.x into the other shared-memory stage are in flight.
constexpr int kRowsStages = 2;
constexpr size_t kRowsSmem = (size_t)kRowsStages * kAccChunk * sizeof(float);

template <bool kVec, bool kEnt>
__global__ void __launch_bounds__(kAccThreads, 3)
accept_rows(const float *__restrict__ logits, int V, int nchunks, int beta, int n_items,
            VI *__restrict__ cand, MS *__restrict__ part) {
    pdl_enter();
    __shared__ RowsShared sh[2];
    extern __shared__ __align__(16) float s_stage[];  // kRowsStages x kAccChunk
    const int step = gridDim.x;
    int item = blockIdx.x;
    if (item < n_items) fetch_item<kVec>(logits, V, nchunks, item, s_stage);
    cp_async_commit();
    for (int k = 0; item < n_items; ++k, item += step) {
        float *cur = s_stage + (k & 1) * kAccChunk;
        float *nxt = s_stage + ((k + 1) & 1) * kAccChunk;
        if (item < n_items - step) fetch_item<kVec>(logits, V, nchunks, item + step, nxt);
        cp_async_commit();
        cp_async_wait_1();  // this thread's copies of `item` have landed
        const int c0 = (item % nchunks) * kAccChunk;
        float v[kAccVpt];
        read_item<kVec>(cur, V, c0, v);
        rows_item<kVec, kEnt>(v, V, c0, beta, item, cand, part, sh[k & 1], k % (kAccThreads / 32));
    }
}

// Row statistics: one warp per row merges the chunk candidates (loaded
// once into registers, <= 32 * kCandPerLane) by beta rounds of a warp-wide
// "best after the previous winner" reduction, and the chunk (m, s, w)
// triples into the log-sum-exp (and the entropy when asked).
constexpr int kMergeThreads = 256;
constexpr int kCandPerLane = 8;

__global__ void __launch_bounds__(kMergeThreads)
accept_merge(const VI *__restrict__ cand, const MS *__restrict__ part, int nchunks, int beta, int R,
             int32_t *__restrict__ argmax, int32_t *__restrict__ topk, float *__restrict__ lse,
             float *__restrict__ entropy, float *__restrict__ rowmax) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const long long r = (long long)blockIdx.x * (kMergeThreads / 32) + (threadIdx.x >> 5);
    if (r >= R) return;
    MS ms{-INFINITY, 0.f, 0.f};
    for (int c = lane; c < nchunks; c += 32) ms = ms_merge(ms, part[r * nchunks + c]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) ms = ms_merge(ms, ms_shfl(ms, o));
    const int ncand = nchunks * beta;
    VI cv[kCandPerLane];
#pragma unroll
    for (int q = 0; q < kCandPerLane; ++q) {
        const int c = lane + 32 * q;
        cv[q] = c < ncand ? cand[r * ncand + c] : VI{-INFINITY, kNoId};
    }
    VI prev{INFINITY, -1};
    for (int k = 0; k < beta; ++k) {
        VI best{-INFINITY, kNoId};
#pragma unroll
        for (int q = 0; q < kCandPerLane; ++q) {
            const VI x = cv[q];
            if (x.i != kNoId && vi_before(prev.v, prev.i, x.v, x.i) && vi_before(x.v, x.i, best.v, best.i))
                best = x;
        }
        best = warp_vi_best(best);
        prev = best;
        if (lane == 0) {
            const int id = best.i == kNoId ? -1 : best.i;
            topk[r * beta + k] = id;
            if (k == 0) {
                argmax[r] = id;
                rowmax[r] = best.v;
            }
        }
    }
    if (lane == 0) {
        lse[r] = ms.s > 0.f ? ms.m + __logf(ms.s) : -INFINITY;
        if (entropy) entropy[r] = ms.s > 0.f ? (__logf(ms.s) - ms.w / ms.s) : 0.f;
    }
}

constexpr int kDecThreads = 512;
constexpr int kNodeWords = RS_MAX_NODES / 32;

// One CTA per request.  Every global read happens in two dependent rounds
// at the start (the tree, the row statistics and the selected positions'
// scores; then the logit of each node's token in its parent's row); the rest
// works on shared memory.  Per node it precomputes the greedy match
// (token == argmax of the parent row) and the relaxed check of Eq. 6-7
// (token among the parent row's top beta and max logit - token logit <= tau
// in fp64), so each chain's look-ahead walk and each model node's path check
// read only flags.  Chain c's nodes are ranked by popcounts of per-chain
// membership masks (one warp ballot per 32 nodes).
__global__ void __launch_bounds__(kDecThreads)
accept_decide(const float *__restrict__ logits, int V, const int32_t *__restrict__ node_off,
              const int32_t *__restrict__ tokens, const int32_t *__restrict__ parents,
              const uint8_t *__restrict__ source, const int8_t *__restrict__ chain,
              const int32_t *__restrict__ sel_pos, const int64_t *__restrict__ tok_off, rs_params p,
              int acc_cap, const int32_t *__restrict__ argmax, const int32_t *__restrict__ topk,
              const float *__restrict__ lse, const float *__restrict__ rowmax, float *__restrict__ p_tok,
              int32_t *__restrict__ acc_len, int32_t *__restrict__ acc_nodes, int32_t *__restrict__ bonus,
              int32_t *__restrict__ winner, uint8_t *__restrict__ commit, float *__restrict__ scores,
              int32_t *__restrict__ status) {
    pdl_enter();
    const int b = blockIdx.x;
    const int n0 = node_off[b];
    const int N = node_off[b + 1] - n0;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int beta = p.beta, top_c = p.top_c;

    __shared__ int s_arg[RS_MAX_NODES];
    __shared__ int s_top[RS_MAX_NODES * RS_MAX_BETA];
    __shared__ int s_par[RS_MAX_NODES];
    __shared__ int s_tok[RS_MAX_NODES];
    __shared__ float s_zmax[RS_MAX_NODES];  // each row's largest logit
    __shared__ float s_ztok[RS_MAX_NODES];  // node i: logit of its token in its parent's row
    __shared__ uint8_t s_src[RS_MAX_NODES];
    __shared__ int8_t s_chn[RS_MAX_NODES];
    __shared__ uint8_t s_g[RS_MAX_NODES];   // greedy match
    __shared__ uint8_t s_rx[RS_MAX_NODES];  // relaxed check (Eq. 6 and Eq. 7)
    __shared__ uint32_t s_cmask[RS_MAX_TOPC][kNodeWords];
    __shared__ int s_cnodes[RS_MAX_TOPC][RS_MAX_NODES];
    __shared__ int s_clen[RS_MAX_TOPC];
    __shared__ int s_cacc[RS_MAX_TOPC];
    __shared__ int s_selp[RS_MAX_TOPC];
    __shared__ float s_selS[RS_MAX_TOPC];
    __shared__ int s_bad, s_stt, s_win, s_dup;
    __shared__ int s_best;  // (depth << 16) | (0xffff - node)

    int st = 0;
    if (N > RS_MAX_NODES) st = RS_ST_TOO_LARGE;
    else if (N < 1) st = RS_ST_BAD_TREE;
    if (tid == 0) {
        s_bad = 0;
        s_best = 0;
        s_stt = 0;
    }
    const long long t0 = tok_off[b];
    const long long t = tok_off[b + 1] - t0;
    if (tid < top_c) {  // the selected positions and their scores (Eq. 4-5 inputs)
        const int pos = sel_pos[(long long)b * top_c + tid];
        s_selp[tid] = pos;
        s_selS[tid] = (pos >= 0 && (long long)pos < t) ? scores[t0 + pos] : 0.f;
    }
    __syncthreads();

    // ---- round 1 + 2: tree, row statistics, token logits ----
    if (st == 0) {
        for (int i = tid; i < N; i += kDecThreads) {
            const int pa = parents[n0 + i];
            const int sr = source[n0 + i];
            const int ch = chain[n0 + i];
            const int tk = tokens[n0 + i];
            s_arg[i] = argmax[n0 + i];
            s_zmax[i] = rowmax[n0 + i];
            s_par[i] = pa;
            s_tok[i] = tk;
            s_src[i] = (uint8_t)sr;
            s_chn[i] = (int8_t)ch;
            commit[n0 + i] = 0;
            bool bad;
            if (i == 0) bad = (pa != -1 || sr != 0 || ch != -1);
            else bad = (pa < 0 || pa >= i || sr < 1 || sr > 2 || (sr == 2 && (ch < 0 || ch >= top_c)) ||
                        (sr == 1 && ch != -1) || tk < 0 || tk >= V);
            if (bad) {
                atomicOr(&s_bad, 1);
            } else if (i == 0) {
                p_tok[n0] = 1.f;
            } else {
                const float z = logits[(long long)(n0 + pa) * V + tk];
                s_ztok[i] = z;
                p_tok[n0 + i] = __expf(z - lse[n0 + pa]);
            }
        }
        for (int x = tid; x < N * beta; x += kDecThreads)
            s_top[(x / beta) * RS_MAX_BETA + (x % beta)] = topk[(long long)n0 * beta + x];
    }
    __syncthreads();
    const bool ok1 = st == 0 && s_bad == 0;

    // ---- model nodes hang from the root or from model nodes; chain
    // membership masks; per-node greedy and relaxed flags ----
    if (ok1) {
        for (int i = 1 + tid; i < N; i += kDecThreads) {
            const int pa = s_par[i], x = s_tok[i];
            if (s_src[i] == 1 && s_src[pa] > 1) atomicOr(&s_bad, 1);
            s_g[i] = (uint8_t)(x == s_arg[pa]);
            bool in_top = false;
            for (int j = 0; j < beta; ++j) in_top |= (s_top[pa * RS_MAX_BETA + j] == x);
            const double gap = (double)s_zmax[pa] - (double)s_ztok[i];
            s_rx[i] = (uint8_t)(in_top && gap <= (double)p.tau);
        }
        if (warp < kNodeWords) {
            const int i = warp * 32 + lane;
            const int ch = (i > 0 && i < N && s_src[i] == 2) ? s_chn[i] : -1;
            for (int c = 0; c < top_c; ++c) {
                const uint32_t m = __ballot_sync(0xffffffffu, ch == c);
                if (lane == 0) s_cmask[c][warp] = m;
            }
        }
    }
    __syncthreads();
    const bool ok2 = ok1 && s_bad == 0;
    // ---- chain c in index order: node of rank r ----
    if (ok2) {
        for (int i = 1 + tid; i < N; i += kDecThreads) {
            if (s_src[i] != 2) continue;
            const int c = s_chn[i], w = i >> 5;
            int rank = __popc(s_cmask[c][w] & ((1u << (i & 31)) - 1u));
            for (int q = 0; q < w; ++q) rank += __popc(s_cmask[c][q]);
            s_cnodes[c][rank] = i;
        }
        if (tid < top_c) {
            int L = 0;
#pragma unroll
            for (int q = 0; q < kNodeWords; ++q) L += __popc(s_cmask[tid][q]);
            s_clen[tid] = L;
        }
    }
    __syncthreads();
    // ---- each chain is a path from the root: rank r hangs from rank r - 1 ----
    if (ok2) {
        for (int x = tid; x < top_c * RS_MAX_NODES; x += kDecThreads) {
            const int c = x / RS_MAX_NODES, r = x - c * RS_MAX_NODES;
            if (r >= s_clen[c]) continue;
            if (s_par[s_cnodes[c][r]] != (r == 0 ? 0 : s_cnodes[c][r - 1])) atomicOr(&s_bad, 1);
        }
    }
    __syncthreads();
    if (st == 0 && s_bad) st = RS_ST_BAD_TREE;

    // ---- outputs of a rejected request ----
    if (st != 0) {
        for (int i = tid; i < N; i += kDecThreads) {
            p_tok[n0 + i] = 0.f;
            commit[n0 + i] = 0;
        }
        for (int j = tid; j < acc_cap; j += kDecThreads) acc_nodes[(long long)b * acc_cap + j] = -1;
        if (tid == 0) {
            acc_len[b] = 0;
            winner[b] = -2;
            bonus[b] = -1;
            status[b] = st;
        }
        return;
    }

    // ---- strict verification of model nodes: every node on the root path matches ----
    for (int i = 1 + tid; i < N; i += kDecThreads) {
        if (s_src[i] != 1) continue;
        bool ok = true;
        int depth = 0;
        for (int a = i; a > 0; a = s_par[a]) {
            ok = ok && s_g[a];
            ++depth;
        }
        if (ok) atomicMax(&s_best, (depth << 16) | (0xffff - i));
    }

    // ---- relaxed verification with look-ahead, one thread per chain ----
    if (tid < top_c) {
        const int c = tid, L = s_clen[c];
        const int *d = s_cnodes[c];
        int l0 = 0;
        while (l0 < L && s_g[d[l0]]) ++l0;
        int cur = l0, last = l0;
        for (int att = 0; att < p.phi; ++att) {
            if (cur >= L || !s_rx[d[cur]]) break;
            int xi = 0;
            while (cur + 1 + xi < L && s_g[d[cur + 1 + xi]]) ++xi;
            if (xi >= p.m) {
                last = cur + 1 + xi;
                cur = last;
            } else {
                cur = cur + 1;
            }
        }
        s_cacc[c] = last;
    }
    __syncthreads();

    // ---- winner, accepted path, bonus, commit ----
    if (tid == 0) {
        const int model_len = s_best >> 16;
        const int best_node = model_len > 0 ? 0xffff - (s_best & 0xffff) : 0;
        int best_len = model_len, win = model_len > 0 ? -1 : -2;
        for (int c = 0; c < top_c; ++c)
            if (s_cacc[c] > best_len) {
                best_len = s_cacc[c];
                win = c;
            }
        if (best_len == 0) win = -2;
        int last_node = 0;
        if (win == -1) {
            int a = best_node;
            last_node = a;
            for (int j = best_len - 1; j >= 0; --j) {
                if (j < acc_cap) acc_nodes[(long long)b * acc_cap + j] = a;
                commit[n0 + a] = 1;
                a = s_par[a];
            }
        } else if (win >= 0) {
            for (int j = 0; j < best_len; ++j) {
                const int a = s_cnodes[win][j];
                if (j < acc_cap) acc_nodes[(long long)b * acc_cap + j] = a;
                commit[n0 + a] = 1;
                last_node = a;
            }
        }
        for (int j = best_len; j < acc_cap; ++j) acc_nodes[(long long)b * acc_cap + j] = -1;
        commit[n0] = 1;
        acc_len[b] = best_len;
        winner[b] = win;
        bonus[b] = s_arg[last_node];
        s_win = win;
        s_stt = best_len > acc_cap ? RS_ST_TRUNCATED : 0;
        // a position selected twice is updated twice, in selection order
        int dup = 0;
        for (int c = 0; c < top_c; ++c)
            for (int c2 = 0; c2 < c; ++c2)
                dup |= (s_selp[c] >= 0 && s_selp[c] == s_selp[c2]);
        s_dup = dup;
    }
    __syncthreads();

    // ---- Eq. 4-5 in fp64, rounded once to the fp32 table ----
    const double a = (double)p.alpha;
    auto ema = [&](int c, double S) -> double {
        const double R = (s_win == c) ? __ddiv_rn((double)s_cacc[c], (double)s_clen[c]) : 0.0;
        return __dadd_rn(__dmul_rn(__dsub_rn(1.0, a), S), __dmul_rn(a, R));
    };
    if (!s_dup) {
        if (tid < top_c) {
            const int c = tid, pos = s_selp[c];
            if (pos >= 0 && s_clen[c] != 0) {
                if ((long long)pos >= t) atomicOr(&s_stt, RS_ST_BAD_POS);
                else scores[t0 + pos] = __double2float_rn(ema(c, (double)s_selS[c]));
            }
        }
    } else if (tid == 0) {
        for (int c = 0; c < top_c; ++c) {
            const int pos = s_selp[c];
            if (pos < 0 || s_clen[c] == 0) continue;
            if ((long long)pos >= t) {
                s_stt |= RS_ST_BAD_POS;
                continue;
            }
            float *S = scores + t0 + pos;
            *S = __double2float_rn(ema(c, (double)(*S)));
        }
    }
    __syncthreads();
    if (tid == 0) status[b] = s_stt;
}

}  // namespace
}  // namespace rs

using namespace rs;

extern "C" size_t rs_accept_workspace_size(int R, int V, int beta) {
    if (R < 0 || V < 1 || beta < 1) return 0;
    int nchunks = (V + kAccChunk - 1) / kAccChunk;
    Carve cv(nullptr);
    cv.take<VI>((size_t)R * nchunks * beta);
    cv.take<MS>((size_t)R * nchunks);
    cv.take<float>((size_t)R);
    return cv.used();
}

extern "C" rs_status rs_accept(const float *logits, int R, int V, const int32_t *node_off, int B,
                               const int32_t *tokens, const int32_t *parents, const uint8_t *source,
                               const int8_t *chain, const int32_t *sel_pos, const int64_t *tok_off,
                               rs_params p, int acc_cap, int32_t *argmax, int32_t *topk, float *lse,
                               float *p_tok, float *entropy, int32_t *acc_len, int32_t *acc_nodes,
                               int32_t *bonus, int32_t *winner, uint8_t *commit, float *scores, int32_t *status,
                               void *workspace, size_t workspace_bytes, void *stream) {
    clear_error();
    RS_CHECK_ARG(R >= 0 && B >= 0, "rs_accept: negative size (R=%d, B=%d)", R, B);
    RS_CHECK_ARG(V >= 1, "rs_accept: V must be >= 1 (got %d)", V);
    RS_CHECK_ARG(p.beta >= 1 && p.beta <= RS_MAX_BETA && p.beta <= V,
                 "rs_accept: beta=%d outside [1, min(%d, V)]", p.beta, RS_MAX_BETA);
    RS_CHECK_ARG(p.top_c >= 1 && p.top_c <= RS_MAX_TOPC, "rs_accept: top_c=%d outside [1, %d]", p.top_c,
                 RS_MAX_TOPC);
    RS_CHECK_ARG(p.tau >= 0.f, "rs_accept: tau must be >= 0");
    RS_CHECK_ARG(p.phi >= 0 && p.m >= 0, "rs_accept: phi and m must be >= 0");
    RS_CHECK_ARG(p.alpha >= 0.f && p.alpha <= 1.f, "rs_accept: alpha outside [0, 1]");
    RS_CHECK_ARG(acc_cap >= 1, "rs_accept: acc_cap must be >= 1");
    RS_CHECK_ARG(R == 0 || (logits && tokens && parents && source && chain && argmax && topk && lse &&
                            p_tok && commit),
                 "rs_accept: null row pointer");
    RS_CHECK_ARG(B == 0 || (node_off && sel_pos && tok_off && acc_len && acc_nodes && bonus && winner &&
                            scores && status),
                 "rs_accept: null request pointer");
    const int nchunks = (V + kAccChunk - 1) / kAccChunk;
    if (nchunks * p.beta > 32 * kCandPerLane) {
        set_error("rs_accept: V=%d with beta=%d exceeds the %d top-k candidates a row merge holds", V, p.beta,
                  32 * kCandPerLane);
        return RS_ERR_UNSUPPORTED;
    }
    const size_t need = rs_accept_workspace_size(R, V, p.beta);
    if (workspace_bytes < need || (need && !workspace)) {
        set_error("rs_accept: workspace %zu bytes < %zu required", workspace_bytes, need);
        return RS_ERR_CAPACITY;
    }
    cudaStream_t st = (cudaStream_t)stream;
    Carve cv(workspace);
    VI *cand = cv.take<VI>((size_t)R * nchunks * p.beta);
    MS *part = cv.take<MS>((size_t)R * nchunks);
    float *rowmax = cv.take<float>((size_t)R);
    if (R > 0) {
        const long long blocks = (long long)R * nchunks;
        RS_CHECK_ARG(blocks < (1ll << 30), "rs_accept: R*chunks too large");
        const int n_items = (int)blocks;
        const bool vec = (V % 4 == 0) && (((uintptr_t)logits & 15) == 0);
        const bool ent = entropy != nullptr;
        const unsigned grid = (unsigned)std::min<long long>(blocks, 3ll * num_sms());
        static int attr_done[64] = {0};
        int dev = 0;
        cudaGetDevice(&dev);
        if (dev >= 0 && dev < 64 && !attr_done[dev]) {
            cudaError_t e = cudaSuccess;
            const int bytes = (int)kRowsSmem;
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(accept_rows<true, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(accept_rows<true, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(accept_rows<false, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(accept_rows<false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
            if (e != cudaSuccess) {
                set_error("rs_accept: cudaFuncSetAttribute: %s", cudaGetErrorString(e));
                return RS_ERR_CUDA;
            }
            attr_done[dev] = 1;
        }
        if (vec && ent)
            launch_full(accept_rows<true, true>, dim3(grid), dim3(kAccThreads), kRowsSmem, st, logits, V, nchunks,
                p.beta, n_items, cand, part);
        else if (vec)
            launch_full(accept_rows<true, false>, dim3(grid), dim3(kAccThreads), kRowsSmem, st, logits, V,
                nchunks, p.beta, n_items, cand, part);
        else if (ent)
            launch_full(accept_rows<false, true>, dim3(grid), dim3(kAccThreads), kRowsSmem, st, logits, V,
                nchunks, p.beta, n_items, cand, part);
        else
            launch_full(accept_rows<false, false>, dim3(grid), dim3(kAccThreads), kRowsSmem, st, logits, V,
                nchunks, p.beta, n_items, cand, part);
        RS_CHECK_LAUNCH("rs_accept/accept_rows");
        launch_pdl(accept_merge, dim3((R + kMergeThreads / 32 - 1) / (kMergeThreads / 32)), dim3(kMergeThreads),
            0, st, cand, part, nchunks, p.beta, R, argmax, topk, lse, entropy, rowmax);
        RS_CHECK_LAUNCH("rs_accept/accept_merge");
    }
    if (B > 0) {
        launch_pdl(accept_decide, dim3(B), dim3(kDecThreads), 0, st, logits, V, node_off, tokens, parents,
            source, chain, sel_pos, tok_off, p, acc_cap, argmax, topk, lse, rowmax, p_tok, acc_len, acc_nodes,
            bonus, winner, commit, scores, status);
        RS_CHECK_LAUNCH("rs_accept/accept_decide");
    }
    return RS_OK;
}
