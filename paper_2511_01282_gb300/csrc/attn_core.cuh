// attn_core.cuh -- per-piece compute of rs_tree_verify_attn: one CTA runs
// one (request, KV head, row tile) over a contiguous range of 128-key KV
// tiles with an online softmax, then writes either the final output or an
// unnormalised partial for the combine kernel.
#pragma once

#include <cuda_bf16.h>
#include <math.h>

#include "common.cuh"

namespace rs {

constexpr int kBM = 128;           // (node, q-head-in-group) rows per tile
constexpr int kBN = 128;           // keys per KV tile (one work unit)
constexpr int kAncWords = RS_MAX_NODES / 32;
constexpr int kAttnThreads = 256;
constexpr int kAttnCtasPerSm = 2;
constexpr int kAttnSmemTiles = 2 * kBN * 128 * 2;  // K and V tiles, bf16, D <= 128

struct AttnArgs {
    const uint16_t *q, *k, *v;
    const int64_t *kv_off;
    const int32_t *ctx_len, *node_off;
    const uint32_t *anc;
    float *part_o, *part_m, *part_l;
    int B, Hq, Hkv, D;
    float scale;
    float *out, *lse;
};

struct Piece {
    int b, kvh, mtile, j0, j1;  // KV tiles [j0, j1) of segment (b, kvh, mtile)
    bool final;                  // the piece is the whole segment
    int slot;                    // partial slot when not final
};

__device__ __forceinline__ float bf16_lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t x) { return __uint_as_float(x & 0xffff0000u); }

// CUDA-core reference core: two threads per row, each owning half of D.
template <int D>
__device__ void attn_piece_fma(const AttnArgs &a, const Piece &pc, unsigned char *smem) {
    constexpr int DH = D / 2;
    const int tid = threadIdx.x;
    const int rl = tid >> 1, half = tid & 1;
    const int G = a.Hq / a.Hkv;
    const int n0 = a.node_off[pc.b];
    const int N = a.node_off[pc.b + 1] - n0;
    const int S = a.ctx_len[pc.b];
    const int T = S + N;
    const long long kv0 = a.kv_off[pc.b];
    const int rr = pc.mtile * kBM + rl;
    const bool valid = rr < N * G;
    const int i = valid ? rr / G : 0;
    const int h = pc.kvh * G + (valid ? rr - i * G : 0);

    float q[DH], o[DH];
    const uint16_t *qp = a.q + ((long long)(n0 + i) * a.Hq + h) * D + half * DH;
#pragma unroll
    for (int d = 0; d < DH; d += 2) {
        uint32_t x = *reinterpret_cast<const uint32_t *>(qp + d);
        q[d] = bf16_lo(x) * a.scale;
        q[d + 1] = bf16_hi(x) * a.scale;
        o[d] = o[d + 1] = 0.f;
    }
    uint32_t bits[kAncWords];
#pragma unroll
    for (int w = 0; w < kAncWords; ++w) bits[w] = valid ? a.anc[(long long)(n0 + i) * kAncWords + w] : 0u;
    float m = -INFINITY, l = 0.f;

    uint16_t *sK = reinterpret_cast<uint16_t *>(smem);
    uint16_t *sV = sK + kBN * D;
    for (int jt = pc.j0; jt < pc.j1; ++jt) {
        __syncthreads();
        // stage the K and V tiles (rows past the request's keys are zero)
        for (int x = tid; x < kBN * D / 8; x += kAttnThreads) {
            const int r = x / (D / 8), c8 = x - r * (D / 8);
            const int j = jt * kBN + r;
            uint4 kk = make_uint4(0, 0, 0, 0), vv = kk;
            if (j < T) {
                const long long off = ((kv0 + j) * a.Hkv + pc.kvh) * D + c8 * 8;
                kk = *reinterpret_cast<const uint4 *>(a.k + off);
                vv = *reinterpret_cast<const uint4 *>(a.v + off);
            }
            reinterpret_cast<uint4 *>(sK)[x] = kk;
            reinterpret_cast<uint4 *>(sV)[x] = vv;
        }
        __syncthreads();
        const int jn = min(kBN, T - jt * kBN);
        for (int jj = 0; jj < jn; ++jj) {
            const int j = jt * kBN + jj;
            const uint32_t *kr = reinterpret_cast<const uint32_t *>(sK + jj * D + half * DH);
            float s = 0.f;
#pragma unroll
            for (int d = 0; d < DH; d += 2) {
                uint32_t x = kr[d >> 1];
                s = fmaf(q[d], bf16_lo(x), s);
                s = fmaf(q[d + 1], bf16_hi(x), s);
            }
            s += __shfl_xor_sync(0xffffffffu, s, 1);
            bool allowed = j < S || ((bits[(j - S) >> 5] >> ((j - S) & 31)) & 1u);
            if (allowed) {
                const float mn = fmaxf(m, s);
                const float corr = __expf(m - mn);
                const float pj = __expf(s - mn);
                l = l * corr + pj;
                const uint32_t *vr = reinterpret_cast<const uint32_t *>(sV + jj * D + half * DH);
#pragma unroll
                for (int d = 0; d < DH; d += 2) {
                    uint32_t x = vr[d >> 1];
                    o[d] = fmaf(pj, bf16_lo(x), o[d] * corr);
                    o[d + 1] = fmaf(pj, bf16_hi(x), o[d + 1] * corr);
                }
                m = mn;
            }
        }
    }
    __syncthreads();
    if (!valid) return;
    if (pc.final) {
        const long long orow = (long long)(n0 + i) * a.Hq + h;
        const float inv = 1.f / l;
#pragma unroll
        for (int d = 0; d < DH; ++d) a.out[orow * D + half * DH + d] = o[d] * inv;
        if (half == 0) a.lse[orow] = m + __logf(l);
    } else {
        const long long prow = (long long)pc.slot * kBM + rl;
#pragma unroll
        for (int d = 0; d < DH; ++d) a.part_o[prow * D + half * DH + d] = o[d];
        if (half == 0) {
            a.part_m[prow] = m;
            a.part_l[prow] = l;
        }
    }
}

__device__ __forceinline__ void attn_piece(const AttnArgs &a, const Piece &pc, unsigned char *smem) {
    if (a.D == 128) attn_piece_fma<128>(a, pc, smem);
    else attn_piece_fma<64>(a, pc, smem);
}

}  // namespace rs
