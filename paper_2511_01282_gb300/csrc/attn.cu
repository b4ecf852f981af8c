// attn.cu -- rs_tree_verify_attn: attention of the verify pass over the
// packed draft tree (the verify forward of Algorithm 1; "parallel verification" of
// Section 3.3).  Node i of request b attends to b's committed prefix and to
// the tree slots of its ancestors and itself.
//
// Work decomposition:
//   segment = (request b, KV head, row tile of 128 (node, q-head-in-group)
//             rows); unit = one 128-key KV tile of a segment.
//   The units of all segments are laid end to end and cut into one equal
//   range per SM, so every SM streams the same number of KV tiles whatever
//   the mix of context lengths (a stream-K split).  A segment that lies
//   inside one CTA's range is finished by that CTA; a segment cut by range
//   boundaries leaves one partial (unnormalised O, running max, running sum)
//   per piece, in one of two slots per CTA, and attn_combine merges them.
//   Nothing spins or waits across CTAs.
//   attn_prep validates each tree and builds a 256-bit ancestor set per
//   node; the tree part of the mask is a bit test on it.
// Launches: attn_prep (B CTAs) -> attn_tc_kernel (one CTA per SM; see
// attn_core.cuh) -> attn_combine (three CTAs per SM over the split segments' rows).
#include <cudaTypedefs.h>
#include <math.h>

#include <algorithm>
#include <cstdlib>
#include <cstring>

#include <mutex>

#include "attn_core.cuh"
#include "attn_pair.cuh"
#include "common.cuh"

namespace rs {
namespace {

__global__ void __launch_bounds__(256)
attn_prep(const int32_t *__restrict__ node_off, const int32_t *__restrict__ ctx_len,
          const int64_t *__restrict__ kv_off, const int32_t *__restrict__ parents, int R, long long kv_rows,
          int Hq, int Hkv, int D, int seg_rows, ReqInfo *__restrict__ info, uint32_t *__restrict__ anc,
          float *__restrict__ out, float *__restrict__ lse, int32_t *__restrict__ status) {
    pdl_enter();
    const int b = blockIdx.x, tid = threadIdx.x;
    const int n0 = node_off[b];
    const int N = node_off[b + 1] - n0;
    const int S = ctx_len[b];
    const long long kv0 = kv_off[b];
    const int G = Hq / Hkv;
    __shared__ int s_par[RS_MAX_NODES];
    __shared__ int s_bad;

    // the request's rows must lie in [0, R) and its keys (prefix, then one
    // slot per node) in [0, kv_rows); outside them nothing is read or written
    const bool rows_ok = n0 >= 0 && N >= 0 && (long long)n0 + N <= R;
    int st = 0;
    if (!rows_ok || kv0 < 0 || (S >= 0 && kv0 + S + N > kv_rows)) st = RS_ST_BAD_OFFSET;
    else if (S < 0) st = RS_ST_BAD_TREE;
    else if (N > RS_MAX_NODES) st = RS_ST_TOO_LARGE;
    if (tid == 0) s_bad = 0;
    __syncthreads();
    if (st == 0) {
        for (int i = tid; i < N; i += blockDim.x) {
            int pa = parents[n0 + i];
            s_par[i] = pa;
            if (i == 0 ? pa != -1 : (pa < 0 || pa >= i)) atomicOr(&s_bad, 1);
        }
        __syncthreads();
        if (s_bad) st = RS_ST_BAD_TREE;
    }
    if (st == 0) {
        for (int i = tid; i < N; i += blockDim.x) {
            uint32_t bits[kAncWords];
#pragma unroll
            for (int w = 0; w < kAncWords; ++w) bits[w] = 0;
            for (int x = i; x >= 0; x = s_par[x]) bits[x >> 5] |= 1u << (x & 31);
#pragma unroll
            for (int w = 0; w < kAncWords; ++w) anc[(long long)(n0 + i) * kAncWords + w] = bits[w];
        }
        if (tid == 0) {
            int mt = (N * G + seg_rows - 1) / seg_rows;
            int nt = (S + N + kBN - 1) / kBN;
            info[b] = ReqInfo{Hkv * mt * nt, mt, nt, N * G};
        }
    } else {
        if (tid == 0) info[b] = ReqInfo{0, 0, 0, 0};
        if (rows_ok && N > 0) {
            const long long n = (long long)N * Hq;
            for (long long x = tid; x < n * D; x += blockDim.x) out[(long long)n0 * Hq * D + x] = 0.f;
            for (long long x = tid; x < n; x += blockDim.x) lse[(long long)n0 * Hq + x] = 0.f;
        }
    }
    if (tid == 0) status[b] = st;
}

// attn_combine: every block first reads all job records (one per attention
// CTA; a record names the split segment that CTA started) and cuts each job
// into items of rows by a block scan, then takes items blockIdx.x,
// blockIdx.x + gridDim.x, ...  A lane merges one column quad of rpw
// consecutive rows, rpw = 4, 2 or 1 for segments of <= 2, <= 4 or more
// pieces, so that it issues the loads of up to kCombPairs (row, piece)
// partials (o, m, l) at once: an item costs one memory round trip for
// segments of up to eight pieces whatever their number.  The pieces of a
// row are folded in piece order with a running maximum (deterministic):
// M = max_p m_p, L = sum_p e^(m_p - M) l_p, O = sum_p e^(m_p - M) O_p / L.
// The pieces of a segment are the partial of CTA c (slot first_slot) and
// slot 0 of every later CTA up to c1 with a non-empty unit range (the CTAs'
// ranges are read from the records the attention kernel leaves beside the
// jobs, so the combine does not depend on how the work was split).
constexpr int kCombThreads = 256;
constexpr int kCombPairs = 8;  // (row, piece) loads in flight per lane

// Exclusive prefix of one int per thread of the block, in thread order.
__device__ __forceinline__ int block_excl_scan(int v, int *s_w, int *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    int before = 0, sum = 0;
#pragma unroll
    for (int w = 0; w < kCombThreads / 32; ++w) {
        before += w < warp ? s_w[w] : 0;
        sum += s_w[w];
    }
    __syncthreads();
    *total = sum;
    return before + x - v;
}

template <int D>
__device__ __forceinline__ void combine_item(const AttnArgs &a, const CombJob &job, int np, const int *nonempty,
                                             int row0, int rpw) {
    constexpr int kLpr = D / 4;        // lanes per row, one column quad each
    constexpr int kSub = 32 / kLpr;    // row groups per warp
    const int lane = threadIdx.x & 31;
    const int q = lane % kLpr;
    const int grp = (int)(threadIdx.x >> 5) * kSub + lane / kLpr;
    const int G = a.Hq / a.Hkv;
    const int rows = min(a.seg_rows, job.N * G - job.mtile * a.seg_rows);
    const int rbase = row0 + grp * rpw;                 // this lane's first row in the segment
    const int npairs = max(0, min(rpw, rows - rbase)) * np;
    // piece p > 0: slot 0 of the p-th CTA with a non-empty range after CTA c
    auto slot_of = [&](int p) -> long long { return p == 0 ? job.first_slot : 2ll * nonempty[p]; };
    float M = -INFINITY, L = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    int k = 0, p = 0;  // row and piece the fold is at
    for (int x0 = 0; x0 < npairs; x0 += kCombPairs) {
        float m[kCombPairs], l[kCombPairs];
        float4 o[kCombPairs];
        {
            int kk = x0 / np, pp = x0 - kk * np;
#pragma unroll
            for (int s = 0; s < kCombPairs; ++s) {
                m[s] = -INFINITY;
                l[s] = 0.f;
                o[s] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (x0 + s < npairs) {
                    const long long prow = slot_of(pp) * a.seg_rows + rbase + kk;
                    m[s] = a.part_m[prow];
                    l[s] = a.part_l[prow];
                    o[s] = *reinterpret_cast<const float4 *>(a.part_o + prow * D + q * 4);
                    if (++pp == np) {
                        pp = 0;
                        ++kk;
                    }
                }
            }
        }
#pragma unroll
        for (int s = 0; s < kCombPairs; ++s) {
            if (x0 + s >= npairs) break;
            const float mp = m[s];
            if (mp != -INFINITY) {
                if (mp > M) {
                    const float sc = __expf(M - mp);  // M = -inf: 0
                    acc = make_float4(fmaf(acc.x, sc, o[s].x), fmaf(acc.y, sc, o[s].y), fmaf(acc.z, sc, o[s].z),
                                      fmaf(acc.w, sc, o[s].w));
                    L = fmaf(L, sc, l[s]);
                    M = mp;
                } else {
                    const float w = __expf(mp - M);
                    acc = make_float4(fmaf(w, o[s].x, acc.x), fmaf(w, o[s].y, acc.y), fmaf(w, o[s].z, acc.z),
                                      fmaf(w, o[s].w, acc.w));
                    L = fmaf(w, l[s], L);
                }
            }
            if (++p == np) {  // row rbase + k complete
                const int rr = job.mtile * a.seg_rows + rbase + k;
                const int i = rr / G, h = job.kvh * G + (rr - i * G);
                const long long orow = (long long)(job.n0 + i) * a.Hq + h;
                const float f = L > 0.f ? 1.f / L : 0.f;
                *reinterpret_cast<float4 *>(a.out + orow * D + q * 4) =
                    make_float4(acc.x * f, acc.y * f, acc.z * f, acc.w * f);
                if (q == 0) a.lse[orow] = M + __logf(L);
                M = -INFINITY;
                L = 0.f;
                acc = make_float4(0.f, 0.f, 0.f, 0.f);
                p = 0;
                ++k;
            }
        }
    }
}

template <int D>
__global__ void __launch_bounds__(kCombThreads, 3)
attn_combine(AttnArgs a, int Gc) {
    pdl_enter();
    __shared__ CombJob s_job[kAttnMaxGrid];
    __shared__ int s_np[kAttnMaxGrid], s_rpw[kAttnMaxGrid], s_rank[kAttnMaxGrid];
    __shared__ int s_ne[kAttnMaxGrid];  // the CTAs with a non-empty range, in order
    __shared__ int s_pre[kAttnMaxGrid + 1];
    __shared__ int s_w[kCombThreads / 32];
    const int t = threadIdx.x;
    const int G = a.Hq / a.Hkv;
    constexpr int rows_per_group = kCombThreads / (D / 4);  // rows of an item with rpw = 1
    // CTA t's job and whether its range is empty
    CombJob j;
    j.b = -1;
    int ne = 0;
    if (t < Gc) {
        j = a.jobs[t];
        s_job[t] = j;
        const int2 rg = a.ranges[t];
        ne = rg.y > rg.x;
    }
    int rank;
    if (!__syncthreads_or(t < Gc && !ne)) {  // every range non-empty (the usual case): no scan
        rank = t;
        if (t < Gc) {
            s_rank[t] = t;
            s_ne[t] = t;
        }
    } else {
        int n_ne;
        rank = block_excl_scan(ne, s_w, &n_ne);
        if (t < Gc) {
            s_rank[t] = rank;
            if (ne) s_ne[rank] = t;
        }
    }
    __syncthreads();
    // items of the job of CTA t
    int items = 0;
    if (t < Gc && j.b >= 0) {
        const int np = s_rank[j.c1] - rank + 1;  // CTAs t and c1 both hold a piece
        const int rpw = np <= 2 ? 4 : (np <= 4 ? 2 : 1);
        const int rows = min(a.seg_rows, j.N * G - j.mtile * a.seg_rows);
        const int per = rows_per_group * rpw;
        s_np[t] = np;
        s_rpw[t] = rpw;
        items = (rows + per - 1) / per;
    }
    int total;
    const int pre = block_excl_scan(items, s_w, &total);
    if (t < Gc) s_pre[t] = pre;
    if (t == 0) s_pre[Gc] = total;
    __syncthreads();
    for (int it = blockIdx.x; it < total; it += gridDim.x) {
        int lo = 0, hi = Gc - 1;  // last CTA c with s_pre[c] <= it
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (s_pre[mid] <= it) lo = mid;
            else hi = mid - 1;
        }
        const int c = lo;
        const int row0 = (it - s_pre[c]) * rows_per_group * s_rpw[c];
        combine_item<D>(a, s_job[c], s_np[c], s_ne + s_rank[c], row0, s_rpw[c]);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// q [R, Hq, D] bf16 viewed as (D, Hq, R); boxes of 64 head-dim columns x G
// heads x 128 / G nodes: one 128-row tile of (node, q-head-in-group) rows
// in the order of the two-tile form, 128-byte swizzled (the K-major layout
// the S MMA reads), zero fill past R.
bool make_q_map(CUtensorMap *m, const void *base, int R, int Hq, int G, int D) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hq, (cuuint64_t)R};
    cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hq * D * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(kBM / G)};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// [kv_rows, Hkv, D] bf16 viewed as a 3-D tensor (D, Hkv, kv_rows); boxes of
// 64 head-dim columns x 1 head x 128 keys, 128-byte swizzled, zero fill.
bool make_kv_map(CUtensorMap *m, const void *base, long long kv_rows, int Hkv, int D) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hkv, (cuuint64_t)kv_rows};
    cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hkv * D * 2};
    cuuint32_t box[3] = {64, 1, (cuuint32_t)kBN};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int g_attr_done[64][2] = {};       // one-tile form, per device and head dim
int g_pair_attr_done[64][2] = {};  // two-tile form
int g_pair_regs_ok[64][2] = {};    // two-tile form: 1 usable, -1 not (register budget)

// Rows per segment: 256 selects the two-row-tile form (attn_pair.cuh), which
// pays off when requests have more than one 128-row tile per KV head.  The
// host cannot see the trees, so it decides from the average over the call:
// more (node, q-head-in-group) rows per request and KV head than one tile.
// RS_DEBUG_ATTN_FORM=one|pair overrides the choice (a test hook: both forms
// compute the same function).
// The work split keeps its unit and cost prefixes in 32-bit integers.  A
// request of N <= 256 nodes has at most (N G / 128 + 1) <= 2 G + 1 row tiles
// per KV head and (S + N) / 128 + 1 KV tiles, so a call's units are below
// (2 Hq + Hkv) (kv_rows / 128 + B); a unit costs at most 1 + kSegCostMax
// (one-tile form) or kPairWF + kPairWH kSegCostMax (two-tile form) in the
// split, and the costs must stay below 2^31.
double attn_units_bound(int B, long long kv_rows, int Hq, int Hkv) {
    return (2.0 * Hq + Hkv) * ((double)kv_rows / kBN + B);
}
constexpr double kSplitRange = 2.0e9;
constexpr double kOneCost = 1 + kSegCostMax, kPairCost = kPairWF + kPairWH * kSegCostMax;

int attn_seg_rows(int B, int R, int Hq, int Hkv, int D, long long kv_rows) {
    const bool pair_ok = B <= kPairMaxB && attn_units_bound(B, kv_rows, Hq, Hkv) * kPairCost < kSplitRange;
    if (const char *e = getenv("RS_DEBUG_ATTN_FORM")) {
        if (!strcmp(e, "pair")) return pair_ok ? kPairRows : kBM;
        if (!strcmp(e, "one")) return kBM;
    }
    const long long G = Hkv > 0 ? Hq / Hkv : 1;
    return (pair_ok && D == 128 && (long long)R * G > (long long)kBM * B) ? kPairRows : kBM;
}

}  // namespace
}  // namespace rs

using namespace rs;

static int attn_grid() { return std::min(num_sms(), kAttnMaxGrid); }

extern "C" size_t rs_tree_verify_attn_workspace_size(int B, int R, int Hq, int Hkv, int D) {
    if (B < 0 || R < 0 || Hq < 1 || Hkv < 1 || (D != 64 && D != 128)) return 0;
    const size_t Gc = (size_t)attn_grid();
    // sized for the two-tile form whenever the call could take it (the call
    // itself may still fall back to the one-tile form on a huge KV cache)
    const size_t rows = (size_t)attn_seg_rows(B, R, Hq, Hkv, D, 0);
    Carve cv(nullptr);
    cv.take<ReqInfo>((size_t)B);
    cv.take<uint32_t>((size_t)R * kAncWords);
    cv.take<float>(2 * Gc * rows * (size_t)D);
    cv.take<float>(2 * Gc * rows);
    cv.take<float>(2 * Gc * rows);
    cv.take<CombJob>(Gc);
    cv.take<int2>(Gc);
    return cv.used();
}

extern "C" rs_status rs_tree_verify_attn(const uint16_t *q, const uint16_t *k, const uint16_t *v, int64_t kv_rows,
                                         const int64_t *kv_off, const int32_t *ctx_len, const int32_t *node_off,
                                         const int32_t *parents, int B, int R, int Hq, int Hkv, int D, float scale,
                                         float *out, float *lse, int32_t *status, void *workspace,
                                         size_t workspace_bytes, void *stream) {
    clear_error();
    RS_CHECK_ARG(B >= 0 && R >= 0 && kv_rows >= 0, "rs_tree_verify_attn: negative size");
    if (D != 64 && D != 128) {
        set_error("rs_tree_verify_attn: head dim %d unsupported (64 or 128)", D);
        return RS_ERR_UNSUPPORTED;
    }
    if (Hkv < 1 || Hq < 1 || Hq % Hkv != 0) {
        set_error("rs_tree_verify_attn: Hq=%d must be a positive multiple of Hkv=%d", Hq, Hkv);
        return RS_ERR_UNSUPPORTED;
    }
    RS_CHECK_ARG(B <= kAttnMaxB, "rs_tree_verify_attn: B=%d above %d", B, kAttnMaxB);
    RS_CHECK_ARG(kv_rows < (1ll << 31) - kBN, "rs_tree_verify_attn: kv_rows above 2^31");
    RS_CHECK_ARG(isfinite(scale) && scale > 0.f, "rs_tree_verify_attn: scale must be finite and > 0");
    RS_CHECK_ARG(B == 0 || (kv_off && ctx_len && node_off && status), "rs_tree_verify_attn: null request pointer");
    RS_CHECK_ARG(R == 0 || (q && parents && out && lse), "rs_tree_verify_attn: null row pointer");
    RS_CHECK_ARG(kv_rows == 0 || (k && v), "rs_tree_verify_attn: null KV pointer");
    RS_CHECK_ARG((((uintptr_t)k | (uintptr_t)v | (uintptr_t)q) & 15) == 0,
                 "rs_tree_verify_attn: q, k and v must be 16-byte aligned");
    RS_CHECK_ARG((((uintptr_t)out | (uintptr_t)workspace) & 15) == 0,
                 "rs_tree_verify_attn: out and workspace must be 16-byte aligned");
    if (B == 0) return RS_OK;
    if (attn_units_bound(B, kv_rows, Hq, Hkv) * kOneCost >= kSplitRange) {
        set_error("rs_tree_verify_attn: call too large for one launch's 32-bit work split "
                  "((2 Hq + Hkv) (kv_rows / 128 + B) must stay below 2.2e8)");
        return RS_ERR_UNSUPPORTED;
    }
    const size_t need = rs_tree_verify_attn_workspace_size(B, R, Hq, Hkv, D);
    if (workspace_bytes < need || !workspace) {
        set_error("rs_tree_verify_attn: workspace %zu bytes < %zu required", workspace_bytes, need);
        return RS_ERR_CAPACITY;
    }
    const int Gc = attn_grid();
    const int seg_rows = attn_seg_rows(B, R, Hq, Hkv, D, kv_rows);
    Carve cv(workspace);
    ReqInfo *info = cv.take<ReqInfo>((size_t)B);
    uint32_t *anc = cv.take<uint32_t>((size_t)R * kAncWords);
    AttnArgs a;
    a.q = q;
    a.kv_off = kv_off;
    a.ctx_len = ctx_len;
    a.node_off = node_off;
    a.anc = anc;
    a.part_o = cv.take<float>(2 * (size_t)Gc * seg_rows * D);
    a.part_m = cv.take<float>(2 * (size_t)Gc * seg_rows);
    a.part_l = cv.take<float>(2 * (size_t)Gc * seg_rows);
    a.seg_rows = seg_rows;
    a.q_tma = 0;
    a.stage = 0;
    a.jobs = cv.take<CombJob>((size_t)Gc);
    a.ranges = cv.take<int2>((size_t)Gc);
    a.B = B;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.D = D;
    a.scale = scale;
    a.out = out;
    a.lse = lse;
    a.status = status;
    a.kv_stream = 2.0 * (double)kv_rows * Hkv * D * 2 > 0.5 * (double)l2_bytes();
    // staged epilogue stores (one-tile form): a small gain where K/V streams
    // from HBM (13B shape, 2286 -> 2291 steps/s), a small loss on short
    // launches (7B shape, 19.9 k -> 19.7 k steps/s)
    a.stage = seg_rows == kBM && B <= kStageMaxB && a.kv_stream;
    // a test hook: RS_DEBUG_WAIT_LIMIT (clock cycles) shortens every pipeline
    // wait so that the time-out path can be exercised
    a.wait_limit = kWaitLimit;
    if (const char *e = getenv("RS_DEBUG_WAIT_LIMIT")) {
        const long long v = atoll(e);
        if (v > 0) a.wait_limit = v;
    }
    cudaStream_t st = (cudaStream_t)stream;

    // a map over an empty KV cache is never dereferenced: point it at q
    CUtensorMap tmk, tmv;
    const long long rows_map = kv_rows > 0 ? kv_rows : 1;
    if (!make_kv_map(&tmk, kv_rows > 0 ? (const void *)k : (const void *)q, rows_map, Hkv, D) ||
        !make_kv_map(&tmv, kv_rows > 0 ? (const void *)v : (const void *)q, rows_map, Hkv, D)) {
        set_error("rs_tree_verify_attn: cuTensorMapEncodeTiled failed");
        return RS_ERR_CUDA;
    }

    int dev = 0;
    cudaGetDevice(&dev);
    const int di = D == 128 ? 1 : 0;
    const bool pair = seg_rows == kPairRows;
    // the two-tile form copies its Q tiles with TMA when a tile is whole
    // nodes (G divides 128); otherwise its softmax threads write them
    CUtensorMap tmq = tmk;  // never read unless a.q_tma
    const int Gq = Hq / Hkv;
    if (pair && R > 0 && kBM % Gq == 0) {
        if (!make_q_map(&tmq, q, R, Hq, Gq, D)) {
            set_error("rs_tree_verify_attn: cuTensorMapEncodeTiled (q) failed");
            return RS_ERR_CUDA;
        }
        a.q_tma = 1;
    }
    if (const char *e = getenv("RS_DEBUG_ATTN_QCOPY"))  // test hook: force the thread-written Q path
        if (!strcmp(e, "threads")) a.q_tma = 0;
    if (pair && dev >= 0 && dev < 64 && g_pair_regs_ok[dev][di] == 0) {
        // The two-tile kernel moves registers between its warpgroups with
        // setmaxnreg, sized for a launch of 168 registers per thread; with
        // fewer at launch the raise could never be granted.  Checked once.
        cudaFuncAttributes fa;
        const cudaError_t e = D == 128 ? cudaFuncGetAttributes(&fa, attn_pair_kernel<128>)
                                       : cudaFuncGetAttributes(&fa, attn_pair_kernel<64>);
        g_pair_regs_ok[dev][di] = (e == cudaSuccess && fa.numRegs * kPairThreads >=
                                   (int)(2 * 128 * kPairRegsSoft + 128 * kPairRegsProd)) ? 1 : -1;
    }
    if (pair && (dev < 0 || dev >= 64 || g_pair_regs_ok[dev][di] != 1)) {
        set_error("rs_tree_verify_attn: two-tile kernel built with too few registers per thread");
        return RS_ERR_CUDA;
    }
    launch_pdl(attn_prep, dim3(B), dim3(256), 0, st, node_off, ctx_len, kv_off, parents, R, (long long)kv_rows, Hq,
        Hkv, D, seg_rows, info, anc, out, lse,
        status);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/prep");

    int(&attr_done)[64][2] = pair ? g_pair_attr_done : g_attr_done;
    if (dev >= 0 && dev < 64 && !attr_done[dev][di]) {
        cudaError_t e;
        if (pair) {
            const int smem_max = (int)attn_pair_smem_bytes(kPairMaxB);
            e = D == 128 ? cudaFuncSetAttribute(attn_pair_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                smem_max)
                         : cudaFuncSetAttribute(attn_pair_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                smem_max);
        } else {
            const int smem_max = (int)std::max(attn_smem_bytes(kAttnMaxB), attn_smem_bytes_staged(kStageMaxB));
            e = D == 128 ? cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                smem_max)
                         : cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                smem_max);
        }
        if (e != cudaSuccess) {
            set_error("rs_tree_verify_attn: cudaFuncSetAttribute: %s", cudaGetErrorString(e));
            return RS_ERR_CUDA;
        }
        attr_done[dev][di] = 1;
    }
    if (pair) {
        const size_t smem = attn_pair_smem_bytes(B);
        if (D == 128)
            launch_full(attn_pair_kernel<128>, dim3(Gc), dim3(kPairThreads), smem, st, a, info, tmk, tmv, tmq);
        else
            launch_full(attn_pair_kernel<64>, dim3(Gc), dim3(kPairThreads), smem, st, a, info, tmk, tmv, tmq);
    } else {
        const size_t smem = a.stage ? attn_smem_bytes_staged(B) : attn_smem_bytes(B);
        if (D == 128)
            launch_full(attn_tc_kernel<128>, dim3(Gc), dim3(kAttnThreads), smem, st, a, info, tmk, tmv);
        else
            launch_full(attn_tc_kernel<64>, dim3(Gc), dim3(kAttnThreads), smem, st, a, info, tmk, tmv);
    }
    RS_CHECK_LAUNCH("rs_tree_verify_attn/main");
    // a full launch: combine blocks parked early beside the attention CTAs
    // (programmatic launch) measured slower on the batched workload
    if (D == 128) launch_full(attn_combine<128>, dim3(3 * Gc), dim3(kCombThreads), 0, st, a, Gc);
    else launch_full(attn_combine<64>, dim3(3 * Gc), dim3(kCombThreads), 0, st, a, Gc);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/combine");
    return RS_OK;
}
