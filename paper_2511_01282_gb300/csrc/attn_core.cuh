// attn_core.cuh -- the tensor-core (tcgen05) core of rs_tree_verify_attn and
// the shared work schedule.
//
// One CTA per SM walks its contiguous range of KV-tile units (see attn.cu).
// Within a CTA, warps are specialised:
//   warp 4 (1 thread)  TMA: K and V tiles of 128 keys x D into a 2-stage
//                      ring of 128-byte-swizzled shared-memory buffers;
//   warp 5 (1 thread)  MMA: S = Q K^T into one of two TMEM buffers, then
//                      O += P V with P read from TMEM (bf16, written over
//                      S by the softmax warps) and V from shared memory;
//   warps 0-3          one thread per row of the 128-row tile: load Q, mask
//                      (prefix always visible, tree slots by the ancestor
//                      bit set, other requests' keys never), online softmax in
//                      base 2 with lazy rescaling of O (only when the running
//                      maximum grows by more than 2^8), write P, and the
//                      epilogue (final O / l and log-sum-exp, or a partial).
// TMEM columns: O [0, D), S/P buffer b at [128 + 128 b, 256 + 128 b).
// Every mbarrier wait is bounded: on a time-out the CTA raises an abort flag,
// every role leaves its loop, in-flight copies and MMAs are drained (again
// bounded), TMEM is released and RS_ST_TIMEOUT is OR-ed into the status of
// the requests the CTA was working on.
#pragma once

#include <cuda_bf16.h>
#include <math.h>

#include "common.cuh"
#include "sm100.cuh"

namespace rs {

constexpr int kBM = 128;  // (node, q-head-in-group) rows per tile
constexpr int kBN = 128;  // keys per KV tile (one work unit)
constexpr int kAncWords = RS_MAX_NODES / 32;
constexpr int kAttnThreads = 192;
constexpr int kNS = 2;                             // K/V ring stages
constexpr int kTileBytes = kBM * 128 * 2;          // one 128 x 128 bf16 tile
constexpr int kSmemQ = 0;
constexpr int kSmemK = kTileBytes;
constexpr int kSmemV = kSmemK + kNS * kTileBytes;
constexpr int kSmemBar = kSmemV + kNS * kTileBytes;
constexpr int kNumBars = 3 * kNS + 8;
constexpr int kSmemMisc = kSmemBar + kNumBars * 8;  // tmem base, abort flag
constexpr int kSmemPref = kSmemMisc + 16;
constexpr int kAttnMaxB = 8192;
constexpr long long kWaitLimit = 4000000000ll;     // clock cycles (~2 s)
constexpr uint32_t kTmemCols = 512;

inline size_t attn_smem_bytes(int B) { return 1024 + kSmemPref + (size_t)(B + 1) * sizeof(int); }

struct ReqInfo {
    int units;  // Hkv * mt * nt, 0 for a rejected request
    int mt;     // row tiles
    int nt;     // KV tiles
    int ok;
};

struct AttnArgs {
    const uint16_t *q;
    const int64_t *kv_off;
    const int32_t *ctx_len, *node_off;
    const uint32_t *anc;
    float *part_o, *part_m, *part_l;
    int B, Hq, Hkv, D;
    float scale;
    float *out, *lse;
    int32_t *status;
};

// ------------------------------------------------------------------ schedule
// Exclusive prefix of per-request units into s_pref[0..B] (s_pref[B] = W).
__device__ inline void unit_prefix(const ReqInfo *__restrict__ info, int B, int *s_pref) {
    __shared__ int s_carry;
    __shared__ int s_w[32];
    if (threadIdx.x == 0) s_carry = 0;
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) >> 5;
    for (int base = 0; base < B; base += blockDim.x) {
        int i = base + threadIdx.x;
        int v = i < B ? info[i].units : 0;
        int x = v;
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) s_w[warp] = x;
        __syncthreads();
        if (warp == 0) {
            int w = lane < nw ? s_w[lane] : 0;
            int z = w;
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, z, o);
                if (lane >= o) z += y;
            }
            s_w[lane] = z - w;
        }
        __syncthreads();
        int incl = s_carry + s_w[warp] + x;
        if (i < B) s_pref[i + 1] = incl;
        __syncthreads();
        if (threadIdx.x == blockDim.x - 1) s_carry = incl;
        __syncthreads();
    }
    if (threadIdx.x == 0) s_pref[0] = 0;
    __syncthreads();
}

// last b with s_pref[b] <= u (so that request b owns unit u)
__device__ __forceinline__ int find_req(const int *s_pref, int B, long long u) {
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        int mid = (lo + hi + 1) >> 1;
        if (s_pref[mid] <= u) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ long long range_lo(long long c, long long W, long long G) { return c * W / G; }
__device__ __forceinline__ long long owner_of(long long u, long long W, long long G) {
    return ((u + 1) * G - 1) / W;
}

struct Piece {
    int b, kvh, mtile, j0, j1;  // KV tiles [j0, j1) of segment (b, kvh, mtile)
    bool final;                  // the piece is the whole segment
    int slot;                    // partial slot when not final
    long long end;               // unit index after the piece
};

__device__ __forceinline__ Piece piece_at(const ReqInfo *__restrict__ info, const int *s_pref, int B,
                                          long long u, long long u0, long long u1, long long c) {
    Piece pc;
    pc.b = find_req(s_pref, B, u);
    const ReqInfo ri = info[pc.b];
    const long long local = u - s_pref[pc.b];
    const int seg = (int)(local / ri.nt);
    pc.j0 = (int)(local - (long long)seg * ri.nt);
    const long long seg_start = s_pref[pc.b] + (long long)seg * ri.nt;
    const long long seg_end = seg_start + ri.nt;
    pc.end = seg_end < u1 ? seg_end : u1;
    pc.kvh = seg / ri.mt;
    pc.mtile = seg - pc.kvh * ri.mt;
    pc.j1 = pc.j0 + (int)(pc.end - u);
    pc.final = (seg_start >= u0 && seg_end <= u1);
    pc.slot = (int)(2 * c + (seg_start > u0 ? 1 : 0));
    return pc;
}

// 32 mask bits for tree indices [base, base + 32): negative indices are prefix
// keys (always visible), indices >= 256 do not exist.
__device__ __forceinline__ uint32_t tree_window(const uint32_t (&anc)[kAncWords], int base) {
    if (base >= RS_MAX_NODES) return 0u;
    if (base <= -32) return 0xffffffffu;
    if (base < 0) {
        const int k = -base;
        return ((1u << k) - 1u) | (anc[0] << k);
    }
    const int w = base >> 5, sh = base & 31;
    uint32_t lo = 0, hi = 0;
#pragma unroll
    for (int q = 0; q < kAncWords; ++q) {
        if (q == w) lo = anc[q];
        if (q == w + 1) hi = anc[q];
    }
    return sh ? ((lo >> sh) | (hi << (32 - sh))) : lo;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

// ------------------------------------------------------------------ kernel
template <int D>
__global__ void __launch_bounds__(kAttnThreads, 1)
attn_tc_kernel(AttnArgs a, const ReqInfo *__restrict__ info, const __grid_constant__ CUtensorMap tmk,
               const __grid_constant__ CUtensorMap tmv) {
    using namespace sm100;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kSmemBar);
    uint64_t *kfull = bars, *vfull = bars + kNS, *kvempty = bars + 2 * kNS;
    uint64_t *sfull = bars + 3 * kNS, *pfull = sfull + 2, *odone = pfull + 2, *qready = odone + 1;
    uint64_t *ofree = qready + 1, *drain = ofree + 1;
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + kSmemMisc);
    volatile int *s_abort = reinterpret_cast<volatile int *>(smem + kSmemMisc + 4);
    int *s_pref = reinterpret_cast<int *>(smem + kSmemPref);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        for (int s = 0; s < kNS; ++s) {
            mbar_init(&kfull[s], 1);
            mbar_init(&vfull[s], 1);
            mbar_init(&kvempty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&sfull[s], 1);
            mbar_init(&pfull[s], 128);
        }
        mbar_init(odone, 1);
        mbar_init(qready, 128);
        mbar_init(ofree, 128);
        mbar_init(drain, 1);
        *s_abort = 0;
        fence_mbar_init();
    }
    if (warp == 5) tmem_alloc(s_tmem, kTmemCols);
    if (warp == 4 && lane == 0) {
        prefetch_tmap(&tmk);
        prefetch_tmap(&tmv);
    }
    unit_prefix(info, a.B, s_pref);  // contains __syncthreads
    tc_fence_after();
    const uint32_t tmem = *s_tmem;
    const long long W = s_pref[a.B];
    const long long Gc = gridDim.x, c = blockIdx.x;
    const long long u0 = range_lo(c, W, Gc), u1 = range_lo(c + 1, W, Gc);
    const int G = a.Hq / a.Hkv;
    constexpr uint32_t kTileTx = (uint32_t)kBN * D * 2;
    constexpr int kKB = D / 64;  // 64-column swizzle blocks per row

    if (warp == 4) {
        // ---------------------------------------------------------- TMA producer
        if (lane == 0) {
            long long g = 0;
            bool ok = true;
            for (long long u = u0; u < u1 && ok;) {
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                const long long kv0 = a.kv_off[pc.b];
                for (int jt = pc.j0; jt < pc.j1; ++jt, ++g) {
                    const int st = (int)(g % kNS);
                    if (!(ok = mbar_wait(&kvempty[st], (uint32_t)(((g / kNS) & 1) ^ 1), s_abort, kWaitLimit)))
                        break;
                    const int row = (int)(kv0 + (long long)jt * kBN);
                    unsigned char *sk = smem + kSmemK + st * kTileBytes;
                    unsigned char *sv = smem + kSmemV + st * kTileBytes;
                    mbar_expect_tx(&kfull[st], kTileTx);
#pragma unroll
                    for (int kb = 0; kb < kKB; ++kb) tma_load_3d(sk + kb * 16384, &tmk, &kfull[st], kb * 64, pc.kvh, row);
                    mbar_expect_tx(&vfull[st], kTileTx);
#pragma unroll
                    for (int kb = 0; kb < kKB; ++kb) tma_load_3d(sv + kb * 16384, &tmv, &vfull[st], kb * 64, pc.kvh, row);
                }
                u = pc.end;
            }
            if (!ok) {  // let the copies already issued land before the CTA exits
                for (long long t = g - kNS; t < g; ++t) {
                    if (t < 0) continue;
                    volatile int no_abort = 0;
                    mbar_wait(&kfull[t % kNS], (uint32_t)((t / kNS) & 1), &no_abort, kWaitLimit);
                    mbar_wait(&vfull[t % kNS], (uint32_t)((t / kNS) & 1), &no_abort, kWaitLimit);
                }
            }
        }
    } else if (warp == 5) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kBM, kBN, false);
            constexpr uint32_t idO = idesc_bf16_f32(kBM, D, true);
            const uint32_t q_addr = smem_u32(smem + kSmemQ);
            long long g = 0;
            int piece = 0;
            bool ok = true;
            auto issue_s = [&](long long gt) -> bool {
                const int st = (int)(gt % kNS);
                if (!mbar_wait(&kfull[st], (uint32_t)((gt / kNS) & 1), s_abort, kWaitLimit)) return false;
                tc_fence_after();
                const uint32_t k_addr = smem_u32(smem + kSmemK + st * kTileBytes);
                const uint32_t d_s = tmem + 128 + (uint32_t)(gt & 1) * 128;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (uint32_t)((kk >> 2) * 16384 + (kk & 3) * 32);
                    umma_ss(d_s, sdesc_sw128(q_addr + off, 16, 1024), sdesc_sw128(k_addr + off, 16, 1024), idS,
                            kk > 0);
                }
                umma_commit(&sfull[gt & 1]);
                return true;
            };
            for (long long u = u0; u < u1 && ok; ++piece) {
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                const int n = pc.j1 - pc.j0;
                if (!(ok = mbar_wait(qready, (uint32_t)(piece & 1), s_abort, kWaitLimit))) break;
                tc_fence_after();
                if (!(ok = issue_s(g))) break;
                for (int tl = 0; tl < n && ok; ++tl) {
                    const long long gt = g + tl;
                    if (tl + 1 < n && !(ok = issue_s(gt + 1))) break;
                    const int st = (int)(gt % kNS);
                    if (!(ok = mbar_wait(&pfull[gt & 1], (uint32_t)((gt >> 1) & 1), s_abort, kWaitLimit))) break;
                    if (!(ok = mbar_wait(&vfull[st], (uint32_t)((gt / kNS) & 1), s_abort, kWaitLimit))) break;
                    if (tl == 0 && piece > 0 &&
                        !(ok = mbar_wait(ofree, (uint32_t)((piece - 1) & 1), s_abort, kWaitLimit)))
                        break;
                    tc_fence_after();
                    const uint32_t v_addr = smem_u32(smem + kSmemV + st * kTileBytes);
                    const uint32_t p_tm = tmem + 128 + (uint32_t)(gt & 1) * 128;
#pragma unroll
                    for (int ks = 0; ks < kBN / 16; ++ks)
                        umma_ts(tmem, p_tm + ks * 8, sdesc_sw128(v_addr + ks * 2048, 16384, 1024), idO,
                                (tl > 0 || ks > 0) ? 1u : 0u);
                    umma_commit(&kvempty[st]);
                    umma_commit(odone);
                }
                g += n;
                u = pc.end;
            }
            if (!ok) {  // drain the MMAs in flight before TMEM is released
                umma_commit(drain);
                volatile int no_abort = 0;
                mbar_wait(drain, 0, &no_abort, kWaitLimit);
            }
        }
    } else {
        // ---------------------------------------------------------- softmax / epilogue (rows)
        const int r = tid;  // row of the tile == TMEM lane
        const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
        const float cexp = a.scale * 1.4426950408889634f;  // scores -> log2 domain
        long long g = 0;
        int piece = 0;
        uint32_t odone_phase = 0;
        bool ok = true;
        for (long long u = u0; u < u1 && ok; ++piece) {
            const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
            const int n0 = a.node_off[pc.b];
            const int N = a.node_off[pc.b + 1] - n0;
            const int S = a.ctx_len[pc.b];
            const int rr = pc.mtile * kBM + r;
            const bool valid = rr < N * G;
            const int i = valid ? rr / G : 0;
            const int h = pc.kvh * G + (valid ? rr - i * G : 0);

            // Q row -> swizzled shared memory (rows past the tile's end are zero)
            {
                const uint4 *qp = reinterpret_cast<const uint4 *>(a.q + ((long long)(n0 + i) * a.Hq + h) * D);
#pragma unroll
                for (int ch = 0; ch < D / 8; ++ch) {
                    uint4 x = valid ? qp[ch] : make_uint4(0, 0, 0, 0);
                    const int kb = ch >> 3, cc = ch & 7;
                    *reinterpret_cast<uint4 *>(smem + kSmemQ + kb * 16384 + r * 128 + ((cc ^ (r & 7)) << 4)) = x;
                }
            }
            uint32_t anc[kAncWords];
#pragma unroll
            for (int w = 0; w < kAncWords; ++w) anc[w] = valid ? a.anc[(long long)(n0 + i) * kAncWords + w] : 0u;
            fence_async_smem();
            mbar_arrive(qready);

            float m_used = -INFINITY, l = 0.f;
            const int n = pc.j1 - pc.j0;
            for (int tl = 0; tl < n; ++tl) {
                const long long gt = g + tl;
                const int buf = (int)(gt & 1);
                const int jt = pc.j0 + tl;
                if (!(ok = mbar_wait(&sfull[buf], (uint32_t)((gt >> 1) & 1), s_abort, kWaitLimit))) break;
                tc_fence_after();
                const uint32_t s_tm = tmem + lane_off + 128 + (uint32_t)buf * 128;
                float s[kBN];
#pragma unroll
                for (int ch = 0; ch < kBN / 32; ++ch) {
                    uint32_t x[32];
                    tmem_ld32(s_tm + ch * 32, x);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) s[ch * 32 + e] = __uint_as_float(x[e]);
                }
                float mt = -INFINITY;
                const int key0 = jt * kBN;
                if (key0 + kBN <= S) {  // prefix-only tile: nothing to mask
#pragma unroll
                    for (int j = 0; j < kBN; ++j) {
                        s[j] *= cexp;
                        mt = fmaxf(mt, s[j]);
                    }
                } else {
#pragma unroll
                    for (int ch = 0; ch < kBN / 32; ++ch) {
                        const uint32_t msk = tree_window(anc, key0 + ch * 32 - S);
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const float v = ((msk >> e) & 1u) ? s[ch * 32 + e] * cexp : -INFINITY;
                            s[ch * 32 + e] = v;
                            mt = fmaxf(mt, v);
                        }
                    }
                }
                if (tl > 0) {  // PV of the previous tile is complete: O may be rescaled
                    if (!(ok = mbar_wait(odone, odone_phase & 1, s_abort, kWaitLimit))) break;
                    ++odone_phase;
                    tc_fence_after();
                }
                // lazy rescale: move the reference maximum only when it grows by
                // more than 2^8; tcgen05.ld/st are warp-wide, so the O pass runs
                // when any row of the warp needs it (factor 1 for the others)
                const bool grow = mt > m_used + 8.f;
                const float corr = grow ? ex2(m_used - mt) : 1.f;  // 0 when m_used is -inf
                if (tl > 0 && __any_sync(0xffffffffu, grow)) {
#pragma unroll
                    for (int ch = 0; ch < D / 32; ++ch) {
                        uint32_t x[32];
                        tmem_ld32(tmem + lane_off + ch * 32, x);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e) x[e] = __float_as_uint(__uint_as_float(x[e]) * corr);
                        tmem_st32(tmem + lane_off + ch * 32, x);
                    }
                    tmem_wait_st();
                }
                if (grow) {
                    l *= corr;
                    m_used = mt;
                }
                const float base = (m_used == -INFINITY) ? 0.f : m_used;
                float sum = 0.f;
                uint32_t pw[kBN / 2];
#pragma unroll
                for (int j = 0; j < kBN / 2; ++j) {
                    const float p0 = ex2(s[2 * j] - base), p1 = ex2(s[2 * j + 1] - base);
                    sum += p0 + p1;
                    pw[j] = pack_bf16x2(p0, p1);
                }
                l += sum;
#pragma unroll
                for (int ch = 0; ch < kBN / 64; ++ch) {
                    uint32_t x[32];
#pragma unroll
                    for (int e = 0; e < 32; ++e) x[e] = pw[ch * 32 + e];
                    tmem_st32(s_tm + ch * 32, x);
                }
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(&pfull[buf]);
            }
            if (!ok) break;
            // epilogue: O of the last tile is complete
            if (!(ok = mbar_wait(odone, odone_phase & 1, s_abort, kWaitLimit))) break;
            ++odone_phase;
            tc_fence_after();
            const long long orow = (long long)(n0 + i) * a.Hq + h;
            const long long prow = (long long)pc.slot * kBM + r;
            const float inv = (l > 0.f) ? 1.f / l : 0.f;
#pragma unroll
            for (int ch = 0; ch < D / 32; ++ch) {
                uint32_t x[32];
                tmem_ld32(tmem + lane_off + ch * 32, x);
                tmem_wait_ld();
                if (valid) {
                    float4 *dst = pc.final ? reinterpret_cast<float4 *>(a.out + orow * D + ch * 32)
                                           : reinterpret_cast<float4 *>(a.part_o + prow * D + ch * 32);
                    const float f = pc.final ? inv : 1.f;
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(__uint_as_float(x[4 * e]) * f, __uint_as_float(x[4 * e + 1]) * f,
                                             __uint_as_float(x[4 * e + 2]) * f, __uint_as_float(x[4 * e + 3]) * f);
                }
            }
            if (valid) {
                const float m_nat = m_used * 0.6931471805599453f;
                if (pc.final) {
                    a.lse[orow] = m_nat + __logf(l);
                } else {
                    a.part_m[prow] = m_used == -INFINITY ? -INFINITY : m_nat;
                    a.part_l[prow] = l;
                }
            }
            tc_fence_before();
            mbar_arrive(ofree);
            g += n;
            u = pc.end;
        }
        if (!ok && r == 0) {
            for (long long u = u0; u < u1;) {  // flag every request this CTA touches
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                atomicOr(&a.status[pc.b], RS_ST_TIMEOUT);
                u = pc.end;
            }
        }
    }
    __syncthreads();
    if (warp == 5) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace rs
