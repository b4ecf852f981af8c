// accept.cu -- rs_accept: source-aware verification (Section 3.4, Eq. 6-7
// and the look-ahead tolerance procedure), longest accepted path and winner
// (Algorithm 1), EMA feedback (Eq. 4-5 and Algorithm 1's score update).
//
// Kernel 1 (accept_rows): one CTA per (row, 8192-logit chunk) streams the
// chunk once and produces its (max, sum e^(z - max)[, sum e^(z - max)
// (z - max)]) triple and its beta best (logit, id) pairs in the total order
// (logit desc, id asc); the top-beta is exact and sort-free apart from one
// 16-lane sort that sets the candidate threshold.  No dynamic register
// indexing.
// Row merge: one warp per row merges the chunk results into argmax,
// top-beta, log-sum-exp, the row's largest logit (workspace, for kernel 3)
// and (optionally) the row entropy.  When a row has at most 8 chunks the
// row's chunk CTAs form one cluster: each pushes its results into CTA 0's
// shared memory and CTA 0 merges them after the cluster barrier, so the row
// statistics need no second kernel.  Longer rows write their chunk results
// to the workspace and kernel 2 (accept_merge) merges them.
// Kernel 3 (accept_decide): one CTA per request checks the tree, verifies
// model nodes (each thread walks its own root path over per-node match
// flags), runs the look-ahead procedure per chain (one thread per chain),
// picks the winner and updates the scores (one thread per selection).
#include <math.h>

#include <cooperative_groups.h>

#include <algorithm>

#include "common.cuh"
#include "sm100.cuh"

namespace rs {
namespace {

namespace cg = cooperative_groups;

constexpr int kAccThreads = 256;
constexpr int kAccVpt = 32;
constexpr int kAccChunk = kAccThreads * kAccVpt;
constexpr int kNoId = 0x7fffffff;  // "no candidate": after every real (v, id)
constexpr int kCandCap = 64;        // per-warp candidate buffer (logits at or above the threshold)
constexpr int kFuseMax = 8;         // rows of at most this many chunks merge inside their cluster

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

constexpr int kHalves = 2 * kAccThreads / 32;  // half-warps per CTA (16 >= RS_MAX_BETA)
static_assert(kHalves >= RS_MAX_BETA, "the bound needs beta half-warp maxima");

struct RowsShared {
    MS sms[kAccThreads / 32];
    float hmax[kHalves];
    VI wtop[kAccThreads / 32][RS_MAX_BETA];  // per-warp lists (tie fallback)
    VI cbuf[kCandCap];                       // the chunk's candidates
    VI rx_cand[kFuseMax * RS_MAX_BETA];      // CTA 0 of a row: every chunk's beta best
    MS rx_ms[kFuseMax];                      // and every chunk's triple
    int cnt;
};

// Per-row outputs of the row statistics.
struct RowOut {
    int32_t *argmax, *topk;
    float *lse, *entropy, *rowmax;  // entropy may be null
};

// One warp merges row r's chunk results: the chunk (m, s, w) triples into
// the log-sum-exp (and the entropy), the chunk candidate lists (ncand <=
// 32 kPer pairs, loaded once into registers) into argmax and top-beta by
// beta rounds of a warp-wide "best after the previous winner" reduction.
template <int kPer>
__device__ __forceinline__ void merge_row(const VI *cand, int ncand, const MS *part, int nchunks, int beta,
                                          long long r, const RowOut &o, int lane) {
    MS ms{-INFINITY, 0.f, 0.f};
    for (int c = lane; c < nchunks; c += 32) ms = ms_merge(ms, part[c]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ms = ms_merge(ms, ms_shfl(ms, off));
    VI cv[kPer];
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
        const int c = lane + 32 * q;
        cv[q] = c < ncand ? cand[c] : VI{-INFINITY, kNoId};
    }
    VI prev{INFINITY, -1};
    for (int k = 0; k < beta; ++k) {
        VI best{-INFINITY, kNoId};
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const VI x = cv[q];
            if (x.i != kNoId && vi_before(prev.v, prev.i, x.v, x.i) && vi_before(x.v, x.i, best.v, best.i))
                best = x;
        }
        best = warp_vi_best(best);
        prev = best;
        if (lane == 0) {
            const int id = best.i == kNoId ? -1 : best.i;
            o.topk[r * beta + k] = id;
            if (k == 0) {
                o.argmax[r] = id;
                o.rowmax[r] = best.v;
            }
        }
    }
    if (lane == 0) {
        o.lse[r] = ms.s > 0.f ? ms.m + __logf(ms.s) : -INFINITY;
        if (o.entropy) o.entropy[r] = ms.s > 0.f ? (__logf(ms.s) - ms.w / ms.s) : 0.f;
    }
}

// One CTA per (row, 8192-logit chunk) item: the chunk's (max, sum e^(z -
// max)[, sum e^(z - max) (z - max)]) triple and its beta best (logit, id)
// pairs in the order (logit desc, id asc).
//   * Each thread streams 32 logits into registers (eight 128-bit loads; the
//     in-range test is dropped for chunks that lie inside the row).
//   * Every lane exponentiates against its warp's maximum, so a warp's
//     triple is a plain shuffle sum.
//   * Top-beta: the sixteen half-warp maxima are logits of sixteen disjoint
//     parts of the chunk, so the beta-th largest of them (one 16-lane sort)
//     is a lower bound T on the chunk's beta-th largest logit.  Only logits
//     >= T can be among the best beta; a lane looks at a group of four only
//     if the group's maximum clears T, appends the survivors to shared
//     memory, and warp 0 ranks them by counting (rank = the number of
//     candidates before it in the total order).  If ties at T overflow the
//     buffer, every warp ranks its own logits by beta "best after the
//     previous winner" rounds and warp 0 merges the eight lists (exact too).
//   * kFuse: the chunk's results go to CTA 0 of the row (the CTAs of a row
//     are one cluster, chunk = rank), which merges the row after the
//     cluster barrier; otherwise they go to the workspace for accept_merge.
template <bool kVec, bool kEnt, bool kFuse>
__global__ void __launch_bounds__(kAccThreads, 4)
accept_rows(const float *__restrict__ logits, int V, int nchunks, int beta, VI *__restrict__ cand,
            MS *__restrict__ part, RowOut o) {
    pdl_enter();
    __shared__ RowsShared sh;
    const long long blk = blockIdx.x;
    const long long r = blockIdx.x / (unsigned)nchunks;  // 32-bit division
    const int chunk = (int)(blk - r * nchunks);
    const int c0 = chunk * kAccChunk;
    const float *row = logits + r * (long long)V;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr float kL2E = 1.4426950408889634f;
    const bool clustered = kFuse && nchunks > 1;
    if (clustered) cluster_arrive_relaxed();
    if (tid == 0) sh.cnt = 0;
    VI *dcand = cand + blk * beta;  // where this chunk's beta best and triple go
    MS *dms = part + blk;
    if (kFuse) {
        dcand = &sh.rx_cand[chunk * beta];
        dms = &sh.rx_ms[chunk];
        if (clustered) {
            cg::cluster_group cl = cg::this_cluster();
            dcand = cl.map_shared_rank(dcand, 0);
            dms = cl.map_shared_rank(dms, 0);
        }
    }

    // logit id of register j (ids >= V are padding, held as -inf)
    auto id_of = [&](int j) -> int {
        if (kVec) return c0 + ((j >> 2) * kAccThreads + tid) * 4 + (j & 3);
        return c0 + j * kAccThreads + tid;
    };
    float v[kAccVpt];
    if (kVec) {
        const bool inside = c0 + kAccChunk <= V;
#pragma unroll
        for (int j = 0; j < kAccVpt / 4; ++j) {
            const int off = c0 + (j * kAccThreads + tid) * 4;
            float4 x = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
            if (inside || off < V) x = ldg_stream4(reinterpret_cast<const float4 *>(row + off));  // V % 4 == 0
            v[4 * j + 0] = x.x;
            v[4 * j + 1] = x.y;
            v[4 * j + 2] = x.z;
            v[4 * j + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) {
            const int off = c0 + j * kAccThreads + tid;
            v[j] = off < V ? ldg_stream(row + off) : -INFINITY;
        }
    }

    // group, lane, half-warp and warp maxima
    float g[kAccVpt / 4];
#pragma unroll
    for (int q = 0; q < kAccVpt / 4; ++q) g[q] = fmaxf(fmaxf(v[4 * q], v[4 * q + 1]), fmaxf(v[4 * q + 2], v[4 * q + 3]));
    const float mx = fmaxf(fmaxf(fmaxf(g[0], g[1]), fmaxf(g[2], g[3])), fmaxf(fmaxf(g[4], g[5]), fmaxf(g[6], g[7])));
    float hm = mx;
#pragma unroll
    for (int off = 1; off < 16; off <<= 1) hm = fmaxf(hm, __shfl_xor_sync(0xffffffffu, hm, off));
    const float wmax = fmaxf(hm, __shfl_xor_sync(0xffffffffu, hm, 16));
    if ((lane & 15) == 0) sh.hmax[2 * warp + (lane >> 4)] = hm;

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
        for (int off = 16; off > 0; off >>= 1) {
            ss += __shfl_xor_sync(0xffffffffu, ss, off);
            if (kEnt) ww += __shfl_xor_sync(0xffffffffu, ww, off);
        }
        t.s = ss;
        t.w = ww * 0.6931471805599453f;
    }
    if (lane == 0) sh.sms[warp] = t;
    __syncthreads();

    // T = the beta-th largest half-warp maximum (both half-warps sort the same 16)
    const float thr = __shfl_sync(0xffffffffu, group_sort_desc<16>(sh.hmax[lane & 15], lane), beta - 1);
    if (mx >= thr) {
#pragma unroll
        for (int q = 0; q < kAccVpt / 4; ++q) {
            if (g[q] >= thr) {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = 4 * q + e;
                    const int id = id_of(j);
                    if (v[j] >= thr && id < V) {
                        const int p = atomicAdd(&sh.cnt, 1);
                        if (p < kCandCap) sh.cbuf[p] = VI{v[j], id};
                    }
                }
            }
        }
    }
    __syncthreads();
    const int total = sh.cnt;
    if (clustered) cluster_wait();  // every CTA of the row runs: CTA 0's shared memory is live
    if (total <= kCandCap) {
        if (warp == 0) {
            VI x0 = lane < total ? sh.cbuf[lane] : VI{-INFINITY, kNoId};
            VI x1 = lane + 32 < total ? sh.cbuf[lane + 32] : VI{-INFINITY, kNoId};
            int r0 = 0, r1 = 0;
            for (int q = 0; q < total; ++q) {
                const VI y = sh.cbuf[q];
                r0 += vi_before(y.v, y.i, x0.v, x0.i);
                r1 += vi_before(y.v, y.i, x1.v, x1.i);
            }
            if (lane < total && r0 < beta) dcand[r0] = x0;
            if (lane + 32 < total && r1 < beta) dcand[r1] = x1;
            if (lane >= total && lane < beta) dcand[lane] = VI{-INFINITY, kNoId};
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
        if (warp == 0) {
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
                if (lane == 0) dcand[k] = best;
            }
        }
    }
    if (warp == 0) {  // the eight warp triples, merged as a 3-level tree
        MS a = lane < kAccThreads / 32 ? sh.sms[lane] : MS{-INFINITY, 0.f, 0.f};
#pragma unroll
        for (int off = 4; off > 0; off >>= 1) a = ms_merge(a, ms_shfl(a, off));
        if (lane == 0) *dms = a;
    }
    if (kFuse) {
        if (clustered) {
            cluster_arrive_release();  // the pushes above are visible in CTA 0 after the wait
            cluster_wait();
        } else {
            __syncthreads();
        }
        if (chunk == 0 && warp == 0)
            merge_row<kFuseMax * RS_MAX_BETA / 32>(sh.rx_cand, nchunks * beta, sh.rx_ms, nchunks, beta, r, o, lane);
    }
}

// Row statistics of rows longer than kFuseMax chunks: one warp per row
// merges the chunk results from the workspace.
constexpr int kMergeThreads = 256;
constexpr int kCandPerLane = 8;

__global__ void __launch_bounds__(kMergeThreads)
accept_merge(const VI *__restrict__ cand, const MS *__restrict__ part, int nchunks, int beta, int R, RowOut o) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const long long r = (long long)blockIdx.x * (kMergeThreads / 32) + (threadIdx.x >> 5);
    if (r >= R) return;
    const int ncand = nchunks * beta;
    merge_row<kCandPerLane>(cand + r * ncand, ncand, part + r * nchunks, nchunks, beta, r, o, lane);
}

constexpr int kDecThreads = 512;
static_assert(kDecThreads >= RS_MAX_NODES + RS_MAX_TOPC, "one thread per node plus one per selection");
constexpr int kNodeWords = RS_MAX_NODES / 32;

// One CTA per request.  Every global read happens in two dependent rounds
// at the start (the tree and the row statistics, then the logit of each
// node's token in its parent's row; the selected positions and their scores
// are read by other threads at the same time); the rest works on shared
// memory.  Per node it precomputes the greedy match
// (token == argmax of the parent row) and the relaxed check of Eq. 6-7
// (token among the parent row's top beta and max logit - token logit <= tau
// in fp64), so each chain's look-ahead walk and each model node's path check
// read only flags.  Chain c's nodes are ranked by popcounts of per-chain
// membership masks (one warp ballot per 32 nodes).
__global__ void __launch_bounds__(kDecThreads)
accept_decide(const float *__restrict__ logits, int R, int V, const int32_t *__restrict__ node_off,
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

    // the request's rows must lie in [0, R) and its buffer in the score table
    // (tok_off[B] entries); outside them nothing is read or written
    const bool rows_ok = n0 >= 0 && N >= 0 && (long long)n0 + N <= R;
    const long long t0 = tok_off[b];
    const long long t = tok_off[b + 1] - t0;
    const bool tok_ok = t0 >= 0 && t >= 0 && t0 + t <= tok_off[gridDim.x];
    int st = 0;
    if (!rows_ok || !tok_ok) st = RS_ST_BAD_OFFSET;
    else if (N > RS_MAX_NODES) st = RS_ST_TOO_LARGE;
    else if (N < 1) st = RS_ST_BAD_TREE;
    if (tid == 0) {
        s_bad = 0;
        s_best = 0;
        s_stt = 0;
    }

    // ---- every global read up front.  Node = tid (N <= RS_MAX_NODES, one
    // per thread): its tree entries and row statistics, then its token's
    // logit in the parent's row (two dependent rounds); meanwhile threads
    // RS_MAX_NODES .. read the selected positions and their scores (Eq. 4-5
    // inputs) and every thread reads top-beta ids ----
    const int node = tid;
    int r_pa = 0, r_sr = 0, r_ch = 0, r_tk = 0, r_am = 0;
    float r_zmax = 0.f, r_z = 0.f, r_lp = 0.f;
    bool r_bad = false;
    if (st == 0 && node < N) {
        r_pa = parents[n0 + node];
        r_sr = source[n0 + node];
        r_ch = chain[n0 + node];
        r_tk = tokens[n0 + node];
        r_am = argmax[n0 + node];
        r_zmax = rowmax[n0 + node];
        if (node == 0) r_bad = (r_pa != -1 || r_sr != 0 || r_ch != -1);
        else r_bad = (r_pa < 0 || r_pa >= node || r_sr < 1 || r_sr > 2 || (r_sr == 2 && (r_ch < 0 || r_ch >= top_c)) ||
                    (r_sr == 1 && r_ch != -1) || r_tk < 0 || r_tk >= V);
        if (!r_bad && node > 0) {
            r_z = logits[(long long)(n0 + r_pa) * V + r_tk];
            r_lp = lse[n0 + r_pa];
        }
    }
    const int js = tid - RS_MAX_NODES;
    int selp = -1;
    float selS = 0.f;
    if (js >= 0 && js < top_c) {
        selp = sel_pos[(long long)b * top_c + js];
        selS = (tok_ok && selp >= 0 && (long long)selp < t) ? scores[t0 + selp] : 0.f;
    }
    if (st == 0)
        for (int x = tid; x < N * beta; x += kDecThreads)
            s_top[(x / beta) * RS_MAX_BETA + (x % beta)] = topk[(long long)n0 * beta + x];
    __syncthreads();  // s_bad, s_best and s_stt are initialised
    if (js >= 0 && js < top_c) {
        s_selp[js] = selp;
        s_selS[js] = selS;
    }
    if (st == 0 && node < N) {
        s_arg[node] = r_am;
        s_zmax[node] = r_zmax;
        s_par[node] = r_pa;
        s_tok[node] = r_tk;
        s_src[node] = (uint8_t)r_sr;
        s_chn[node] = (int8_t)r_ch;
        commit[n0 + node] = 0;
        if (r_bad) {
            atomicOr(&s_bad, 1);
        } else if (node == 0) {
            p_tok[n0] = 1.f;
        } else {
            s_ztok[node] = r_z;
            p_tok[n0 + node] = __expf(r_z - r_lp);
        }
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
        for (int i = tid; rows_ok && i < N; i += kDecThreads) {
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

namespace {
using RowsFn = void (*)(const float *, int, int, int, VI *, MS *, RowOut);
template <bool kFuse>
RowsFn rows_fn(bool vec, bool ent) {
    if (vec) return ent ? accept_rows<true, true, kFuse> : accept_rows<true, false, kFuse>;
    return ent ? accept_rows<false, true, kFuse> : accept_rows<false, false, kFuse>;
}
}  // namespace

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
        const bool vec = (V % 4 == 0) && (((uintptr_t)logits & 15) == 0);
        const bool ent = entropy != nullptr;
        const bool fuse = nchunks <= kFuseMax;
        const RowOut ro{argmax, topk, lse, entropy, rowmax};
        const RowsFn fn = fuse ? rows_fn<true>(vec, ent) : rows_fn<false>(vec, ent);
        const dim3 grid((unsigned)blocks);
        if (fuse && nchunks > 1)
            launch_pdl_cluster(fn, grid, dim3(kAccThreads), 0, st, nchunks, logits, V, nchunks, p.beta, cand, part, ro);
        else
            launch_pdl(fn, grid, dim3(kAccThreads), 0, st, logits, V, nchunks, p.beta, cand, part, ro);
        RS_CHECK_LAUNCH("rs_accept/accept_rows");
        if (!fuse) {
            launch_pdl(accept_merge, dim3((R + kMergeThreads / 32 - 1) / (kMergeThreads / 32)), dim3(kMergeThreads),
                0, st, cand, part, nchunks, p.beta, R, ro);
            RS_CHECK_LAUNCH("rs_accept/accept_merge");
        }
    }
    if (B > 0) {
        launch_pdl(accept_decide, dim3(B), dim3(kDecThreads), 0, st, logits, R, V, node_off, tokens, parents,
            source, chain, sel_pos, tok_off, p, acc_cap, argmax, topk, lse, rowmax, p_tok, acc_len, acc_nodes,
            bonus, winner, commit, scores, status);
        RS_CHECK_LAUNCH("rs_accept/accept_decide");
    }
    return RS_OK;
}
