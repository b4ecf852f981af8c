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
// attn_core.cuh) -> attn_combine (one CTA per SM).
#include <cudaTypedefs.h>
#include <math.h>

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

// Block c merges the split segment whose first piece is c's last piece.
// Phase 1: one thread per row forms M = max_p m_p and the weights
// e^(m_p - M) / sum_p e^(m_p - M) l_p in shared memory.  Phase 2: each thread
// owns 16 (row, 4 head-dim columns) items and, piece by piece, accumulates
// their float4 partials (16 independent loads in flight per thread).
constexpr int kCombThreads = 256;
constexpr int kMaxPieces = 1024;
constexpr int kFastPieces = 16;  // pieces whose weights fit the shared table

__global__ void __launch_bounds__(kCombThreads)
attn_combine(AttnArgs a, const ReqInfo *__restrict__ info) {
    extern __shared__ int s_pref[];
    __shared__ int s_slot[kMaxPieces];
    __shared__ float s_w[kFastPieces][kBM];
    __shared__ float s_M[kBM], s_L[kBM];
    __shared__ int s_np;
    unit_prefix(info, a.B, s_pref);
    const long long W = s_pref[a.B];
    const long long Gc = gridDim.x, c = blockIdx.x;
    const long long u0 = range_lo(c, W, Gc), u1 = range_lo(c + 1, W, Gc);
    if (u0 >= u1) return;
    const int b = find_req(s_pref, a.B, u1 - 1);
    const ReqInfo ri = info[b];
    const long long local = u1 - 1 - s_pref[b];
    const int seg = (int)(local / ri.nt);
    const long long seg_start = s_pref[b] + (long long)seg * ri.nt;
    const long long seg_end = seg_start + ri.nt;
    if (!(seg_start >= u0 && seg_end > u1)) return;  // not the first owner of a split segment
    const long long c1 = owner_of(seg_end - 1, W, Gc);
    if (threadIdx.x == 0) {
        int np = 0;
        for (long long cc = c; cc <= c1 && np < kMaxPieces; ++cc) {
            const long long lo = range_lo(cc, W, Gc);
            if (lo == range_lo(cc + 1, W, Gc)) continue;  // empty range: no piece
            s_slot[np++] = (int)(2 * cc + (seg_start > lo ? 1 : 0));
        }
        s_np = np;
    }
    __syncthreads();
    const int np = s_np;
    const int G = a.Hq / a.Hkv;
    const int n0 = a.node_off[b];
    const int N = a.node_off[b + 1] - n0;
    const int kvh = seg / ri.mt, mtile = seg - kvh * ri.mt;
    const int rows = min(kBM, N * G - mtile * kBM);
    const int D = a.D;
    const bool fast = np <= kFastPieces;
    // phase 1: per-row maximum, normaliser and (fast path) weights
    for (int r = threadIdx.x; r < rows; r += kCombThreads) {
        float M = -INFINITY;
        for (int p = 0; p < np; ++p) M = fmaxf(M, a.part_m[(long long)s_slot[p] * kBM + r]);
        float L = 0.f;
        for (int p = 0; p < np; ++p) {
            const long long prow = (long long)s_slot[p] * kBM + r;
            const float m = a.part_m[prow];
            const float w = m == -INFINITY ? 0.f : __expf(m - M);
            L += w * a.part_l[prow];
            if (fast) s_w[p][r] = w;
        }
        s_M[r] = M;
        s_L[r] = L;
        if (fast)
            for (int p = 0; p < np; ++p) s_w[p][r] /= L;
    }
    __syncthreads();
    // phase 2: outputs, four columns per item; each thread keeps kItems items
    // in flight so the partial loads of different items overlap
    constexpr int kItems = kBM * 32 / kCombThreads;  // 16: all (row, column quad) items of D = 128
    const int d4 = D / 4;
    const int nitems = rows * d4;
    float4 acc[kItems];
#pragma unroll
    for (int k = 0; k < kItems; ++k) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int p = 0; p < np; ++p) {
        const long long base = (long long)s_slot[p] * kBM;
#pragma unroll
        for (int k = 0; k < kItems; ++k) {
            const int x = threadIdx.x + k * kCombThreads;
            if (x >= nitems) continue;
            const int r = x / d4, q = x - r * d4;
            float w;
            if (fast) {
                w = s_w[p][r];
            } else {
                const float m = a.part_m[base + r];
                w = m == -INFINITY ? 0.f : __expf(m - s_M[r]) / s_L[r];
            }
            const float4 o = *reinterpret_cast<const float4 *>(a.part_o + (base + r) * D + q * 4);
            acc[k].x += w * o.x;
            acc[k].y += w * o.y;
            acc[k].z += w * o.z;
            acc[k].w += w * o.w;
        }
    }
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
        const int x = threadIdx.x + k * kCombThreads;
        if (x >= nitems) continue;
        const int r = x / d4, q = x - r * d4;
        const int rr = mtile * kBM + r;
        const int i = rr / G, h = kvh * G + (rr - i * G);
        const long long orow = (long long)(n0 + i) * a.Hq + h;
        *reinterpret_cast<float4 *>(a.out + orow * D + q * 4) = acc[k];
        if (q == 0) a.lse[orow] = s_M[r] + __logf(s_L[r]);
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

static int attn_grid() { return num_sms(); }

extern "C" size_t rs_tree_verify_attn_workspace_size(int B, int R, int Hq, int Hkv, int D) {
    if (B < 0 || R < 0 || Hq < 1 || Hkv < 1 || (D != 64 && D != 128)) return 0;
    const size_t Gc = (size_t)attn_grid();
    Carve cv(nullptr);
    cv.take<ReqInfo>((size_t)B);
    cv.take<uint32_t>((size_t)R * kAncWords);
    cv.take<float>(2 * Gc * kBM * (size_t)D);
    cv.take<float>(2 * Gc * kBM);
    cv.take<float>(2 * Gc * kBM);
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
    a.B = B;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.D = D;
    a.scale = scale;
    a.out = out;
    a.lse = lse;
    a.status = status;
    cudaStream_t st = (cudaStream_t)stream;

    // a map over an empty KV cache is never dereferenced: point it at q
    CUtensorMap tmk, tmv;
    const long long rows_map = kv_rows > 0 ? kv_rows : 1;
    if (!make_kv_map(&tmk, kv_rows > 0 ? (const void *)k : (const void *)q, rows_map, Hkv, D) ||
        !make_kv_map(&tmv, kv_rows > 0 ? (const void *)v : (const void *)q, rows_map, Hkv, D)) {
        set_error("rs_tree_verify_attn: cuTensorMapEncodeTiled failed");
        return RS_ERR_CUDA;
    }

    attn_prep<<<B, 256, 0, st>>>(node_off, ctx_len, parents, Hq, Hkv, D, info, anc, out, lse, status);
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
        attn_tc_kernel<128><<<Gc, kAttnThreads, smem, st>>>(a, info, tmk, tmv);
    else
        attn_tc_kernel<64><<<Gc, kAttnThreads, smem, st>>>(a, info, tmk, tmv);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/main");
    attn_combine<<<Gc, kCombThreads, (size_t)(B + 1) * sizeof(int), st>>>(a, info);
    RS_CHECK_LAUNCH("rs_tree_verify_attn/combine");
    return RS_OK;
}
