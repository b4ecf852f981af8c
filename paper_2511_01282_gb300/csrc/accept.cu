// accept.cu -- rs_accept: source-aware verification (Section 3.4, Eq. 6-7
// and the look-ahead tolerance procedure), longest accepted path and winner
// (Algorithm 1 l.13), EMA feedback (Eq. 4-5, Algorithm 1 l.15-22).
//
// Kernel 1 (accept_rows): one CTA per (row, 8192-logit chunk).  Each thread
// holds 32 logits in registers; the CTA produces the chunk's (max, sum e^(z -
// max)) pair and its beta best (logit, id) pairs in the total order (logit
// desc, id asc).  Each warp first bounds its beta-th largest logit from below
// by the beta-th largest of its 32 lane maxima (a warp bitonic sort), appends
// the few logits at or above that bound to shared memory and ranks only those
// by beta rounds of a "best after the previous winner" warp reduction (exact;
// with many ties at the bound it ranks all of the warp's logits instead);
// warp 0 merges the eight lists.  No dynamic register indexing.
// Kernel 2 (accept_decide): one CTA per request.  Warps merge the chunk
// candidates of each row (argmax, top-beta, lse); then the block checks the
// tree, verifies model nodes (each thread walks its own root path), runs the
// look-ahead procedure per chain (one thread per chain), picks the winner and
// updates the scores.
#include <math.h>

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

struct MS {
    float m, s;
};

__device__ __forceinline__ MS ms_merge(MS a, MS b) {
    if (a.s == 0.f) return b;
    if (b.s == 0.f) return a;
    float M = fmaxf(a.m, b.m);
    return MS{M, a.s * __expf(a.m - M) + b.s * __expf(b.m - M)};
}

// Descending bitonic sort of one float per lane across the warp.
__device__ __forceinline__ float warp_sort_desc(float x, int lane) {
#pragma unroll
    for (int k = 2; k <= 32; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
            const float y = __shfl_xor_sync(0xffffffffu, x, j);
            const bool keep_max = ((lane & j) == 0) == ((lane & k) == 0);
            x = keep_max ? fmaxf(x, y) : fminf(x, y);
        }
    }
    return x;
}

template <bool kVec>
__global__ void __launch_bounds__(kAccThreads, 3)
accept_rows(const float *__restrict__ logits, int V, int nchunks, int beta, VI *__restrict__ cand,
            MS *__restrict__ part) {
    const long long blk = blockIdx.x;
    const long long r = blk / nchunks;
    const int chunk = (int)(blk - r * nchunks);
    const float *row = logits + r * (long long)V;
    const int c0 = chunk * kAccChunk;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    constexpr float kL2E = 1.4426950408889634f;

    __shared__ MS sms[kAccThreads / 32];
    __shared__ VI s_wtop[kAccThreads / 32][RS_MAX_BETA];  // each warp's best beta
    __shared__ VI s_cbuf[kAccThreads / 32][kCandCap];     // each warp's candidates
    __shared__ int s_cnt[kAccThreads / 32];
    if (lane == 0) s_cnt[warp] = 0;

    float v[kAccVpt];
    if (kVec) {
#pragma unroll
        for (int j = 0; j < kAccVpt / 4; ++j) {
            const int idx = c0 + (j * kAccThreads + tid) * 4;
            float4 x;
            if (idx + 3 < V) {
                x = ldg_stream4(reinterpret_cast<const float4 *>(row + idx));
            } else {
                x.x = idx + 0 < V ? row[idx + 0] : -INFINITY;
                x.y = idx + 1 < V ? row[idx + 1] : -INFINITY;
                x.z = idx + 2 < V ? row[idx + 2] : -INFINITY;
                x.w = -INFINITY;
            }
            v[4 * j + 0] = x.x;
            v[4 * j + 1] = x.y;
            v[4 * j + 2] = x.z;
            v[4 * j + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) {
            const int idx = c0 + j * kAccThreads + tid;
            v[j] = idx < V ? ldg_stream(row + idx) : -INFINITY;
        }
    }
    // logit id of register j (padding slots have ids >= V)
    auto id_of = [&](int j) -> int {
        if (kVec) return c0 + ((j >> 2) * kAccThreads + tid) * 4 + (j & 3);
        return c0 + j * kAccThreads + tid;
    };

    // lane maximum (pairwise) and (max, sum e^(z - max)) for the log-sum-exp
    float m8[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) m8[q] = fmaxf(fmaxf(v[q], v[q + 8]), fmaxf(v[q + 16], v[q + 24]));
    const float mx = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                           fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
    MS t{mx, 0.f};
    if (mx != -INFINITY) {
        const float nb = -mx * kL2E;
        float s4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int j = 0; j < kAccVpt; ++j) s4[j & 3] += sm100::ex2(fmaf(v[j], kL2E, nb));
        t.s = (s4[0] + s4[1]) + (s4[2] + s4[3]);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        MS u{__shfl_xor_sync(0xffffffffu, t.m, o), __shfl_xor_sync(0xffffffffu, t.s, o)};
        t = ms_merge(t, u);
    }
    if (lane == 0) sms[warp] = t;

    // ---- the warp's best beta, exactly, in (logit desc, id asc) order ----
    // The beta-th largest lane maximum is a lower bound on the warp's beta-th
    // largest logit (the beta lanes it ranks each hold a logit >= it), so
    // only logits >= it can be in the warp's best beta.  Those few are
    // appended to a shared buffer and ranked; if ties overflow the buffer,
    // every logit of the warp is ranked instead.
    const float thr = __shfl_sync(0xffffffffu, warp_sort_desc(mx, lane), beta - 1);
    __syncwarp();
#pragma unroll
    for (int j = 0; j < kAccVpt; ++j) {
        if (v[j] >= thr) {
            const int id = id_of(j);
            if (id < V) {
                const int p = atomicAdd(&s_cnt[warp], 1);
                if (p < kCandCap) s_cbuf[warp][p] = VI{v[j], id};
            }
        }
    }
    __syncwarp();
    const int total = s_cnt[warp];
    VI prev{INFINITY, -1};
    if (total <= kCandCap) {
        for (int k = 0; k < beta; ++k) {
            VI best{-INFINITY, kNoId};
            for (int q = lane; q < total; q += 32) {
                const VI x = s_cbuf[warp][q];
                if (vi_before(prev.v, prev.i, x.v, x.i) && vi_before(x.v, x.i, best.v, best.i)) best = x;
            }
            best = warp_vi_best(best);
            prev = best;
            if (lane == 0) s_wtop[warp][k] = best;
        }
    } else {
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
            if (lane == 0) s_wtop[warp][k] = best;
        }
    }
    __syncthreads();

    // ---- warp 0 merges the warps' lists into the chunk's best beta ----
    if (warp == 0) {
        constexpr int kW = kAccThreads / 32;
        VI prevb{INFINITY, -1};
        for (int k = 0; k < beta; ++k) {
            VI best{-INFINITY, kNoId};
            for (int q = lane; q < kW * beta; q += 32) {
                const VI x = s_wtop[q / beta][q % beta];
                if (x.i != kNoId && vi_before(prevb.v, prevb.i, x.v, x.i) && vi_before(x.v, x.i, best.v, best.i))
                    best = x;
            }
            best = warp_vi_best(best);
            prevb = best;
            if (lane == 0) cand[blk * beta + k] = best;
        }
        if (lane == 0) {
            MS a = sms[0];
            for (int w = 1; w < kW; ++w) a = ms_merge(a, sms[w]);
            part[blk] = a;
        }
    }
}

constexpr int kDecThreads = 512;
// candidates per lane when a warp merges one row: nchunks * beta <= 32 * 8
constexpr int kCandPerLane = 8;

__global__ void __launch_bounds__(kDecThreads)
accept_decide(const float *__restrict__ logits, int V, int nchunks, const VI *__restrict__ cand,
              const MS *__restrict__ part, const int32_t *__restrict__ node_off,
              const int32_t *__restrict__ tokens, const int32_t *__restrict__ parents,
              const uint8_t *__restrict__ source, const int8_t *__restrict__ chain,
              const int32_t *__restrict__ sel_pos, const int64_t *__restrict__ tok_off, rs_params p,
              int acc_cap, int32_t *__restrict__ argmax, int32_t *__restrict__ topk,
              float *__restrict__ lse, float *__restrict__ p_tok, int32_t *__restrict__ acc_len,
              int32_t *__restrict__ acc_nodes, int32_t *__restrict__ bonus, int32_t *__restrict__ winner,
              uint8_t *__restrict__ commit, float *__restrict__ scores, int32_t *__restrict__ status) {
    const int b = blockIdx.x;
    const int n0 = node_off[b];
    const int N = node_off[b + 1] - n0;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int beta = p.beta, top_c = p.top_c;

    __shared__ int s_arg[RS_MAX_NODES];
    __shared__ float s_lse[RS_MAX_NODES];
    __shared__ int s_top[RS_MAX_NODES * RS_MAX_BETA];
    __shared__ int s_par[RS_MAX_NODES];
    __shared__ int s_tok[RS_MAX_NODES];
    __shared__ uint8_t s_src[RS_MAX_NODES];
    __shared__ int8_t s_chn[RS_MAX_NODES];
    __shared__ int s_cnodes[RS_MAX_TOPC][RS_MAX_NODES];
    __shared__ int s_clen[RS_MAX_TOPC];
    __shared__ int s_cacc[RS_MAX_TOPC];
    __shared__ int s_bad;
    __shared__ int s_best;  // (depth << 16) | (0xffff - node)

    // ---- row statistics (every row of the request): one warp per row ----
    // the row's chunk candidates (<= 32 * kCandPerLane) are loaded once into
    // registers, then beta rounds of a warp-wide "best after the previous
    // winner" reduction run on them
    const int ncand = nchunks * beta;
    for (int lr = warp; lr < N; lr += kDecThreads / 32) {
        const long long r = n0 + lr;
        MS ms{-INFINITY, 0.f};
        for (int c = lane; c < nchunks; c += 32) ms = ms_merge(ms, part[r * nchunks + c]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            MS u{__shfl_xor_sync(0xffffffffu, ms.m, o), __shfl_xor_sync(0xffffffffu, ms.s, o)};
            ms = ms_merge(ms, u);
        }
        const float l = ms.s > 0.f ? ms.m + __logf(ms.s) : -INFINITY;
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
                if (lr < RS_MAX_NODES) s_top[lr * RS_MAX_BETA + k] = id;
                if (k == 0) {
                    argmax[r] = id;
                    lse[r] = l;
                    if (lr < RS_MAX_NODES) {
                        s_arg[lr] = id;
                        s_lse[lr] = l;
                    }
                }
            }
        }
    }

    // ---- tree layout check ----
    if (tid == 0) {
        s_bad = 0;
        s_best = 0;
    }
    __syncthreads();
    int st = 0;
    if (N > RS_MAX_NODES) st = RS_ST_TOO_LARGE;
    else if (N < 1) st = RS_ST_BAD_TREE;
    if (st == 0) {
        for (int i = tid; i < N; i += kDecThreads) {
            int pa = parents[n0 + i];
            int sr = source[n0 + i];
            int ch = chain[n0 + i];
            s_par[i] = pa;
            s_tok[i] = tokens[n0 + i];
            s_src[i] = (uint8_t)sr;
            s_chn[i] = (int8_t)ch;
            bool bad;
            if (i == 0) bad = (pa != -1 || sr != 0 || ch != -1);
            else bad = (pa < 0 || pa >= i || sr < 1 || sr > 2 || (sr == 2 && (ch < 0 || ch >= top_c)) ||
                        (sr == 1 && ch != -1) || s_tok[i] < 0 || s_tok[i] >= V);
            if (bad) atomicOr(&s_bad, 1);
        }
        __syncthreads();
        if (!s_bad) {
            // model nodes hang from the root or from model nodes
            for (int i = 1 + tid; i < N; i += kDecThreads)
                if (s_src[i] == 1 && s_src[s_par[i]] > 1) atomicOr(&s_bad, 1);
            // chain c: its nodes in index order form a path from the root
            if (tid < top_c) {
                int c = tid, L = 0, last = 0;
                for (int i = 1; i < N; ++i) {
                    if (s_src[i] != 2 || s_chn[i] != c) continue;
                    if (s_par[i] != last) atomicOr(&s_bad, 1);
                    s_cnodes[c][L++] = i;
                    last = i;
                }
                s_clen[c] = L;
            }
        }
        __syncthreads();
        if (s_bad) st = RS_ST_BAD_TREE;
    }

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

    // ---- p_tok and strict verification of model nodes ----
    for (int i = tid; i < N; i += kDecThreads) {
        commit[n0 + i] = 0;
        if (i == 0) {
            p_tok[n0] = 1.f;
            continue;
        }
        int pa = s_par[i];
        float z = logits[(long long)(n0 + pa) * V + s_tok[i]];
        p_tok[n0 + i] = __expf(z - s_lse[pa]);
        if (s_src[i] == 1) {
            bool ok = true;
            int depth = 0, a = i;
            while (a > 0) {
                ok = ok && (s_tok[a] == s_arg[s_par[a]]);
                ++depth;
                a = s_par[a];
            }
            if (ok) atomicMax(&s_best, (depth << 16) | (0xffff - i));
        }
    }

    // ---- relaxed verification with look-ahead, one thread per chain ----
    if (tid < top_c) {
        const int c = tid, L = s_clen[c];
        const int *d = s_cnodes[c];
        auto greedy = [&](int j) { return s_tok[d[j]] == s_arg[s_par[d[j]]]; };
        int l0 = 0;
        while (l0 < L && greedy(l0)) ++l0;
        int cur = l0, last = l0;
        for (int att = 0; att < p.phi; ++att) {
            if (cur >= L) break;
            const int row = s_par[d[cur]];
            const int x = s_tok[d[cur]];
            bool in_top = false;
            for (int j = 0; j < beta; ++j) in_top |= (s_top[row * RS_MAX_BETA + j] == x);
            const float *zr = logits + (long long)(n0 + row) * V;
            double gap = (double)zr[s_arg[row]] - (double)zr[x];
            if (!(in_top && gap <= (double)p.tau)) break;
            int xi = 0;
            while (cur + 1 + xi < L && greedy(cur + 1 + xi)) ++xi;
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

    // ---- winner, accepted path, bonus, commit, EMA ----
    if (tid == 0) {
        int model_len = s_best >> 16;
        int best_node = model_len > 0 ? 0xffff - (s_best & 0xffff) : 0;
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
                int a = s_cnodes[win][j];
                if (j < acc_cap) acc_nodes[(long long)b * acc_cap + j] = a;
                commit[n0 + a] = 1;
                last_node = a;
            }
        }
        for (int j = best_len; j < acc_cap; ++j) acc_nodes[(long long)b * acc_cap + j] = -1;
        commit[n0] = 1;
        int stt = best_len > acc_cap ? RS_ST_TRUNCATED : 0;
        acc_len[b] = best_len;
        winner[b] = win;
        bonus[b] = s_arg[last_node];

        // Eq. 4-5 in fp64, rounded once to the fp32 table
        const long long t0 = tok_off[b];
        const long long t = tok_off[b + 1] - t0;
        const double a = (double)p.alpha;
        for (int c = 0; c < top_c; ++c) {
            int pos = sel_pos[(long long)b * top_c + c];
            if (pos < 0 || s_clen[c] == 0) continue;
            if ((long long)pos >= t) {
                stt |= RS_ST_BAD_POS;
                continue;
            }
            double R = (win == c) ? __ddiv_rn((double)s_cacc[c], (double)s_clen[c]) : 0.0;
            float *S = scores + t0 + pos;
            double upd = __dadd_rn(__dmul_rn(__dsub_rn(1.0, a), (double)(*S)), __dmul_rn(a, R));
            *S = __double2float_rn(upd);
        }
        status[b] = stt;
    }
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
    return cv.used();
}

extern "C" rs_status rs_accept(const float *logits, int R, int V, const int32_t *node_off, int B,
                               const int32_t *tokens, const int32_t *parents, const uint8_t *source,
                               const int8_t *chain, const int32_t *sel_pos, const int64_t *tok_off,
                               rs_params p, int acc_cap, int32_t *argmax, int32_t *topk, float *lse,
                               float *p_tok, int32_t *acc_len, int32_t *acc_nodes, int32_t *bonus,
                               int32_t *winner, uint8_t *commit, float *scores, int32_t *status,
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
    if (R > 0) {
        long long blocks = (long long)R * nchunks;
        RS_CHECK_ARG(blocks < (1ll << 31), "rs_accept: R*chunks too large");
        bool vec = (V % 4 == 0) && (((uintptr_t)logits & 15) == 0);
        if (vec)
            accept_rows<true><<<(unsigned)blocks, kAccThreads, 0, st>>>(logits, V, nchunks, p.beta, cand, part);
        else
            accept_rows<false><<<(unsigned)blocks, kAccThreads, 0, st>>>(logits, V, nchunks, p.beta, cand, part);
        RS_CHECK_LAUNCH("rs_accept/accept_rows");
    }
    if (B > 0) {
        accept_decide<<<B, kDecThreads, 0, st>>>(logits, V, nchunks, cand, part, node_off, tokens, parents,
                                                 source, chain, sel_pos, tok_off, p, acc_cap, argmax, topk,
                                                 lse, p_tok, acc_len, acc_nodes, bonus, winner, commit,
                                                 scores, status);
        RS_CHECK_LAUNCH("rs_accept/accept_decide");
    }
    return RS_OK;
}
