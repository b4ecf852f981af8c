// attn.cu -- rs_tree_verify_attn: attention of the verify pass over the
// packed draft tree (Algorithm 1 l.13 / l.25; "parallel verification" of
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
// attn_core.cuh) -> attn_combine (four CTAs per range).
#include <cudaTypedefs.h>
#include <math.h>

#include <algorithm>

#include <mutex>

#include "attn_core.cuh"
#include "common.cuh"

namespace rs {
namespace {

__global__ void __launch_bounds__(256)
attn_prep(const int32_t *__restrict__ node_off, const int32_t *__restrict__ ctx_len,
          const int32_t *__restrict__ parents, int Hq, int Hkv, int D, ReqInfo *__restrict__ info,
          uint32_t *__restrict__ anc, float *__restrict__ out, float *__restrict__ lse,
          int32_t *__restrict__ status) {
    pdl_enter();
    const int b = blockIdx.x, tid = threadIdx.x;
    const int n0 = node_off[b];
    const int N = node_off[b + 1] - n0;
    const int S = ctx_len[b];
    const int G = Hq / Hkv;
    __shared__ int s_par[RS_MAX_NODES];
    __shared__ int s_bad;

    int st = 0;
    if (N < 0 || S < 0) st = RS_ST_BAD_TREE;
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
            int mt = (N * G + kBM - 1) / kBM;
            int nt = (S + N + kBN - 1) / kBN;
            info[b] = ReqInfo{Hkv * mt * nt, mt, nt, 1};
        }
    } else {
        if (tid == 0) info[b] = ReqInfo{0, 0, 0, 0};
        if (N > 0) {
            const long long n = (long long)N * Hq;
            for (long long x = tid; x < n * D; x += blockDim.x) out[(long long)n0 * Hq * D + x] = 0.f;
            for (long long x = tid; x < n; x += blockDim.x) lse[(long long)n0 * Hq + x] = 0.f;
        }
    }
    if (tid == 0) status[b] = st;
}

// Block (c, y) merges rows [32 y, 32 y + 32) of the split segment CTA c of
// the attention kernel started (its job record; four blocks per segment).
// The segment's pieces are the partials of CTA c (slot first_slot) and of
// slot 0 of every later CTA up to c1 with a non-empty range.
// Phase 1: thread (row r, lane group j) folds the (m, l) pairs of pieces j,
// j + 8, ... into a running (max, sum); warp 0 merges the eight folds into the
// row's M = max_p m_p and 1 / L, L = sum_p e^(m_p - M) l_p.  Phase 2: each
// thread owns D / 32 (row, 4 head-dim columns) items and sums e^(m_p - M) O_p
// over the pieces, two pieces per round, so a round keeps 2 x D / 32 float4
// partial loads and their m_p loads in flight (the first round is issued
// before phase 1, so the two phases share one memory round trip).  The
// summation order is fixed (piece order), so the result does not depend on
// timing.
constexpr int kCombThreads = 256;
constexpr int kCombRows = 32;                    // rows per block
constexpr int kCombGroups = kBM / kCombRows;     // blocks per split segment
constexpr int kCombFold = kCombThreads / kCombRows;  // lane groups in phase 1
constexpr int kCombBatch = 2;                    // pieces per phase-2 round

__global__ void __launch_bounds__(kCombThreads, 4)  // the 4 x Gc blocks in one wave
attn_combine(AttnArgs a) {
    pdl_enter();
    __shared__ int s_slot[kAttnMaxGrid];
    __shared__ float s_fm[kCombFold][kCombRows], s_fl[kCombFold][kCombRows];
    __shared__ float s_M[kCombRows], s_iL[kCombRows];
    const int c = blockIdx.x;
    const CombJob job = a.jobs[c];
    if (job.b < 0) return;
    const int G = a.Hq / a.Hkv;
    const int n0 = job.n0, N = job.N, kvh = job.kvh, mtile = job.mtile;
    const int r0 = blockIdx.y * kCombRows;
    const int rows = min(kCombRows, N * G - mtile * kBM - r0);
    if (rows <= 0) return;
    const long long Gc = gridDim.x;
    int np;
    if (job.W >= Gc) {  // every range is non-empty: one piece per CTA c .. c1
        np = job.c1 - c + 1;
        for (int x = threadIdx.x; x < np; x += kCombThreads) s_slot[x] = x == 0 ? job.first_slot : 2 * (c + x);
    } else {
        __shared__ int s_np;
        if (threadIdx.x == 0) {
            int n = 0;
            s_slot[n++] = job.first_slot;
            for (long long cc = c + 1; cc <= job.c1 && n < kAttnMaxGrid; ++cc)
                if (range_lo(cc, job.W, Gc) < range_lo(cc + 1, job.W, Gc)) s_slot[n++] = (int)(2 * cc);
            s_np = n;
        }
        __syncthreads();
        np = s_np;
    }
    __syncthreads();
    const int D = a.D;

    // phase-2 items of this thread (row, column quad), and the first batch of
    // their partial loads, issued before phase 1 so both share one round trip
    constexpr int kMaxItems = kCombRows * 128 / 4 / kCombThreads;  // 4 for D = 128
    const int d4 = D / 4;
    const int nitems = rows * d4;
    float4 acc[kMaxItems];
    int irow[kMaxItems];
#pragma unroll
    for (int k = 0; k < kMaxItems; ++k) {
        acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        const int x = threadIdx.x + k * kCombThreads;
        irow[k] = x < nitems ? x / d4 : -1;
    }
    float m[kCombBatch][kMaxItems];
    float4 o[kCombBatch][kMaxItems];
    auto load_batch = [&](int p0) {
#pragma unroll
        for (int q = 0; q < kCombBatch; ++q) {
            const long long base = p0 + q < np ? (long long)s_slot[p0 + q] * kBM + r0 : -1;
#pragma unroll
            for (int k = 0; k < kMaxItems; ++k) {
                m[q][k] = -INFINITY;
                o[q][k] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (base >= 0 && irow[k] >= 0) {
                    const int x = threadIdx.x + k * kCombThreads;
                    const int r = irow[k], cq = x - r * d4;
                    m[q][k] = a.part_m[base + r];
                    o[q][k] = *reinterpret_cast<const float4 *>(a.part_o + (base + r) * D + cq * 4);
                }
            }
        }
    };
    load_batch(0);

    // phase 1: per-row M and 1 / L
    {
        const int r = threadIdx.x & (kCombRows - 1), j = threadIdx.x / kCombRows;
        float fm = -INFINITY, fl = 0.f;
        if (r < rows) {
            for (int p = j; p < np; p += kCombFold) {
                const long long prow = (long long)s_slot[p] * kBM + r0 + r;
                const float mp = a.part_m[prow], lp = a.part_l[prow];
                if (mp == -INFINITY) continue;
                if (mp > fm) {
                    fl = fl * __expf(fm - mp) + lp;  // fm = -inf: fl = 0
                    fm = mp;
                } else {
                    fl += lp * __expf(mp - fm);
                }
            }
        }
        s_fm[j][r] = fm;
        s_fl[j][r] = fl;
        __syncthreads();
        if (threadIdx.x < kCombRows) {
            float M = -INFINITY;
#pragma unroll
            for (int q = 0; q < kCombFold; ++q) M = fmaxf(M, s_fm[q][r]);
            float L = 0.f;
#pragma unroll
            for (int q = 0; q < kCombFold; ++q)
                if (s_fm[q][r] != -INFINITY) L += s_fl[q][r] * __expf(s_fm[q][r] - M);
            s_M[r] = M;
            s_iL[r] = L > 0.f ? 1.f / L : 0.f;
            if (r < rows) {
                const int rr = mtile * kBM + r0 + r;
                const int i = rr / G, h = kvh * G + (rr - i * G);
                a.lse[(long long)(n0 + i) * a.Hq + h] = M + __logf(L);
            }
        }
        __syncthreads();
    }

    // phase 2: the weighted sum of the partial outputs, kCombBatch pieces a round
    for (int p0 = 0; p0 < np; p0 += kCombBatch) {
        if (p0 > 0) load_batch(p0);
#pragma unroll
        for (int q = 0; q < kCombBatch; ++q) {
#pragma unroll
            for (int k = 0; k < kMaxItems; ++k) {
                if (irow[k] < 0 || m[q][k] == -INFINITY) continue;
                const float w = __expf(m[q][k] - s_M[irow[k]]);
                acc[k].x = fmaf(w, o[q][k].x, acc[k].x);
                acc[k].y = fmaf(w, o[q][k].y, acc[k].y);
                acc[k].z = fmaf(w, o[q][k].z, acc[k].z);
                acc[k].w = fmaf(w, o[q][k].w, acc[k].w);
            }
        }
    }
#pragma unroll
    for (int k = 0; k < kMaxItems; ++k) {
        if (irow[k] < 0) continue;
        const int x = threadIdx.x + k * kCombThreads;
        const int r = irow[k], cq = x - r * d4;
        const int rr = mtile * kBM + r0 + r;
        const int i = rr / G, h = kvh * G + (rr - i * G);
        const long long orow = (long long)(n0 + i) * a.Hq + h;
        const float f = s_iL[r];
        *reinterpret_cast<float4 *>(a.out + orow * D + cq * 4) =
            make_float4(acc[k].x * f, acc[k].y * f, acc[k].z * f, acc[k].w * f);
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

int g_attr_done[64][2] = {};

}  // namespace
}  // namespace rs

using namespace rs;

static int attn_grid() { return std::min(num_sms(), kAttnMaxGrid); }

extern "C" size_t rs_tree_verify_attn_workspace_size(int B, int R, int Hq, int Hkv, int D) {
    if (B < 0 || R < 0 || Hq < 1 || Hkv < 1 || (D != 64 && D != 128)) return 0;
    const size_t Gc = (size_t)attn_grid();
    Carve cv(nullptr);
    cv.take<ReqInfo>((size_t)B);
    cv.take<uint32_t>((size_t)R * kAncWords);
    cv.take<float>(2 * Gc * kBM * (size_t)D);
    cv.take<float>(2 * Gc * kBM);
    cv.take<float>(2 * Gc * kBM);
    cv.take<CombJob>(Gc);
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
    if (B == 0) return RS_OK;
    const size_t need = rs_tree_verify_attn_workspace_size(B, R, Hq, Hkv, D);
    if (workspace_bytes < need || !workspace) {
        set_error("rs_tree_verify_attn: workspace %zu bytes < %zu required", workspace_bytes, need);
        return RS_ERR_CAPACITY;
    }
    const int Gc = attn_grid();
    Carve cv(workspace);
    ReqInfo *info = cv.take<ReqInfo>((size_t)B);
    uint32_t *anc = cv.take<uint32_t>((size_t)R * kAncWords);
    AttnArgs a;
    a.q = q;
    a.kv_off = kv_off;
    a.ctx_len = ctx_len;
    a.node_off = node_off;
    a.anc = anc;
    a.part_o = cv.take<float>(2 * (size_t)Gc * kBM * D);
    a.part_m = cv.take<float>(2 * (size_t)Gc * kBM);
    a.part_l = cv.take<float>(2 * (size_t)Gc * kBM);
    a.jobs = cv.take<CombJob>((size_t)Gc);
    a.B = B;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.D = D;
    a.scale = scale;
    a.out = out;
    a.lse = lse;
    a.status = status;
    a.kv_stream = 2.0 * (double)kv_rows * Hkv * D * 2 > 0.5 * (double)l2_bytes();
    cudaStream_t st = (cudaStream_t)stream;

    // a map over an empty KV cache is never dereferenced: point it at q
    CUtensorMap tmk, tmv;
    const long long rows_map = kv_rows > 0 ? kv_rows : 1;
    if (!make_kv_map(&tmk, kv_rows > 0 ? (const void *)k : (const void *)q, rows_map, Hkv, D) ||
        !make_kv_map(&tmv, kv_rows > 0 ? (const void *)v : (const void *)q, rows_map, Hkv, D)) {
        set_error("rs_tree_verify_attn: cuTensorMapEncodeTiled failed");
        return RS_ERR_CUDA;
    }

    launch_pdl(attn_prep, dim3(B), dim3(256), 0, st, node_off, ctx_len, parents, Hq, Hkv, D, info, anc, out, lse,
        status);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/prep");

    int dev = 0;
    cudaGetDevice(&dev);
    const int di = D == 128 ? 1 : 0;
    const size_t smem_max = attn_smem_bytes(kAttnMaxB);
    if (dev >= 0 && dev < 64 && !g_attr_done[dev][di]) {
        cudaError_t e = D == 128 ? cudaFuncSetAttribute(attn_tc_kernel<128>,
                                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_max)
                                 : cudaFuncSetAttribute(attn_tc_kernel<64>,
                                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem_max);
        if (e != cudaSuccess) {
            set_error("rs_tree_verify_attn: cudaFuncSetAttribute: %s", cudaGetErrorString(e));
            return RS_ERR_CUDA;
        }
        g_attr_done[dev][di] = 1;
    }
    const size_t smem = attn_smem_bytes(B);
    if (D == 128)
        launch_full(attn_tc_kernel<128>, dim3(Gc), dim3(kAttnThreads), smem, st, a, info, tmk, tmv);
    else
        launch_full(attn_tc_kernel<64>, dim3(Gc), dim3(kAttnThreads), smem, st, a, info, tmk, tmv);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/main");
    launch_pdl(attn_combine, dim3(Gc, kCombGroups), dim3(kCombThreads), 0, st, a);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/combine");
    return RS_OK;
}
