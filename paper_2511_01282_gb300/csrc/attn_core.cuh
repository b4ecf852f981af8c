// attn_core.cuh -- the tensor-core (tcgen05) core of rs_tree_verify_attn and
// the shared work schedule.
//
// One CTA per SM walks its contiguous range of KV-tile units (see attn.cu
// and the Split below for how the ranges are cut).
// Within a CTA, warps are specialised:
//   warp 8 (1 thread)  TMA: K and V tiles of 128 keys x D into a 3-stage
//                      ring of 128-byte-swizzled shared-memory buffers (a
//                      K slot is refilled once the softmax warps have seen S
//                      of its tile complete, a V slot once P V is);
//   warp 9 (1 thread)  MMA: S = Q K^T into one of two TMEM buffers, then
//                      O += P V with P read from TMEM (bf16, written over
//                      S by the softmax warps) and V from shared memory;
//   warps 0-7          two softmax warpgroups over the same 128 rows (the
//                      TMEM lane of a warp is fixed by warp % 4), each
//                      taking 64 of a tile's 128 keys; they agree on the
//                      row maxima through shared memory and an mbarrier.
//                      Per row: Q into
//                      TMEM, mask
//                      (prefix always visible, tree slots by the ancestor
//                      bit set, other requests' keys never), online softmax in
//                      base 2 with lazy rescaling of O (only when the running
//                      maximum grows by more than 2^8), write P, and the
//                      epilogue (final O / l and log-sum-exp, or a partial).
// TMEM columns: O [0, D), S/P buffer b at [128 + 128 b, 256 + 128 b), Q
// (bf16, two per column) at [384, 384 + D/2).  The MMA reads Q and P as
// tensor-memory A operands; only K and V go through shared memory.
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
constexpr int kSoftThreads = 256;  // two softmax warpgroups (warps 0-7)
constexpr int kTmaWarp = 8, kMmaWarp = 9;
constexpr int kAttnThreads = 320;
constexpr int kNS = 3;                             // K/V ring stages
constexpr int kTileBytes = kBN * 128 * 2;          // one 128-key x 128-dim bf16 tile
constexpr int kSmemK = 0;
constexpr int kSmemV = kSmemK + kNS * kTileBytes;
constexpr int kSmemBar = kSmemV + kNS * kTileBytes;
constexpr int kNumBars = 4 * kNS + 12;
constexpr int kSmemMisc = kSmemBar + kNumBars * 8;  // tmem base, abort flag
constexpr int kSmemPref = kSmemMisc + 16;
constexpr int kAttnMaxB = 3840;  // requests per call (the two prefixes over them live in shared memory)
constexpr int kAttnMaxGrid = 256;  // CTAs (one per SM, at most this many)
constexpr long long kWaitLimit = 4000000000ll;     // clock cycles (~2 s)
constexpr uint32_t kTmemCols = 512;
// TMEM columns: O [0, 128), S/P buffers [128, 256) and [256, 384), Q [384, 448)
constexpr uint32_t kTmO = 0, kTmS = 128, kTmQ = 384;

// In the split of the work over the CTAs each segment (request, KV head, row
// tile) costs its KV tiles plus beta = min(kSegCostMax, W / (2 G)) tiles (W
// units, G CTAs): a piece boundary (Q loaded, pipeline restarted, epilogue)
// costs several tiles' worth, so CTAs whose ranges cut many short segments
// were the stragglers.  The cap keeps small launches (a few units per CTA)
// close to an even split of the units, and launches with long ranges
// (>= kSegCostOff units per CTA, where a boundary is a small part of a range
// and every CTA has about the same number of pieces) keep the even split.
constexpr int kSegCostMax = 8;
constexpr int kSegCostOff = 128;
// unit and segment prefixes over the requests: 2 (B + 1) ints after kSmemPref
inline size_t attn_smem_bytes(int B) { return 1024 + kSmemPref + 2 * (size_t)(B + 1) * sizeof(int); }
// Epilogue staging (calls of at most kStageMaxB requests, where it fits):
// per softmax warp 32 rows x 16 columns of O at a row stride of 20 floats,
// after the prefixes (256-byte aligned).
constexpr int kStageMaxB = 1024;
constexpr int kStageFloats = 32 * 20;  // per warp
__host__ __device__ inline size_t attn_stage_offset(int B) { return (kSmemPref + 2 * (size_t)(B + 1) * sizeof(int) + 255) & ~size_t(255); }
inline size_t attn_smem_bytes_staged(int B) { return 1024 + attn_stage_offset(B) + 8 * kStageFloats * sizeof(float); }

struct ReqInfo {
    int units;  // Hkv * mt * nt, 0 for a rejected request
    int mt;     // row tiles (row-tile pairs in the two-tile form) per KV head
    int nt;     // KV tiles
    int rows;   // (node, q-head-in-group) rows per KV head: N * Hq / Hkv
};

// The split segment a CTA starts, for attn_combine: the segment that begins
// in the CTA's range and continues past it (at most one per CTA).
struct CombJob {
    long long W;     // units of the launch
    int b;           // request (-1: the CTA starts no split segment)
    int kvh, mtile;  // the segment's KV head and row tile
    int n0, N;       // the request's first node and node count
    int first_slot;  // partial slot of the segment's first piece
    int c1;          // last CTA holding a piece of the segment
    int pad;
};

struct AttnArgs {
    const uint16_t *q;
    const int64_t *kv_off;
    const int32_t *ctx_len, *node_off;
    const uint32_t *anc;
    float *part_o, *part_m, *part_l;
    CombJob *jobs;  // [gridDim.x]
    int2 *ranges;   // [gridDim.x]: each CTA's unit range [x, y)
    int kv_stream;  // the launch's K/V is large next to L2: stream tiles read once
    int seg_rows;   // rows per segment and per partial slot: 128, or 256 in the two-tile form
    int stage;      // one-tile form: O rows leave through shared memory (attn_smem_bytes_staged)
    int q_tma;      // two-tile form: Q tiles are copied by TMA (128 % (Hq / Hkv) == 0)
    long long wait_limit;  // clock cycles a pipeline wait may take before the CTA gives up
    int B, Hq, Hkv, D;
    float scale;
    float *out, *lse;
    int32_t *status;
};

// ------------------------------------------------------------------ schedule
// Exclusive prefixes over the requests of their units (s_pref[0..B],
// s_pref[B] = W) and of their segments (s_spref).
__device__ inline void unit_prefix(const ReqInfo *__restrict__ info, int B, int *s_pref, int *s_spref) {
    __shared__ int s_carry[2];
    __shared__ int s_w[2][32];
    if (threadIdx.x == 0) s_carry[0] = s_carry[1] = 0;
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) >> 5;
    for (int base = 0; base < B; base += blockDim.x) {
        const int i = base + threadIdx.x;
        int v[2] = {0, 0};
        if (i < B) {
            const ReqInfo ri = info[i];
            v[0] = ri.units;
            v[1] = ri.nt > 0 ? ri.units / ri.nt : 0;
        }
        int x[2] = {v[0], v[1]};
#pragma unroll
        for (int k = 0; k < 2; ++k) {
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, x[k], o);
                if (lane >= o) x[k] += y;
            }
            if (lane == 31) s_w[k][warp] = x[k];
        }
        __syncthreads();
        if (warp == 0) {
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const int w = lane < nw ? s_w[k][lane] : 0;
                int z = w;
                for (int o = 1; o < 32; o <<= 1) {
                    const int y = __shfl_up_sync(0xffffffffu, z, o);
                    if (lane >= o) z += y;
                }
                s_w[k][lane] = z - w;
            }
        }
        __syncthreads();
        const int incl0 = s_carry[0] + s_w[0][warp] + x[0];
        const int incl1 = s_carry[1] + s_w[1][warp] + x[1];
        if (i < B) {
            s_pref[i + 1] = incl0;
            s_spref[i + 1] = incl1;
        }
        __syncthreads();
        if (threadIdx.x == blockDim.x - 1) {
            s_carry[0] = incl0;
            s_carry[1] = incl1;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) s_pref[0] = s_spref[0] = 0;
    __syncthreads();
}

// floor(a * b / d) for a, b >= 0 and d > 0, in 32-bit arithmetic whenever
// the product fits (64-bit division is a long instruction sequence, and the
// work split sits on every CTA's path to its first tile).
__device__ __forceinline__ long long muldiv(long long a, long long b, long long d) {
    const unsigned long long p = (unsigned long long)a * (unsigned long long)b;
    if ((p >> 32) == 0 && d <= 0xffffffffll) return (long long)((uint32_t)p / (uint32_t)d);
    return (long long)(p / (unsigned long long)d);
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

// The work split.  Cost positions: request b's segments occupy
// [cost(b), cost(b + 1)), cost(b) = s_pref[b] + beta s_spref[b], nt + beta
// each; CTA c takes [c C / G, (c + 1) C / G) (C = cost(B)).  A position in a
// segment's first beta maps to the segment's first unit, so the ranges are
// unit ranges that tile [0, W) in order (some may be empty).
struct Split {
    const int *pref, *spref;
    int B, beta, G;
    __device__ __forceinline__ int cost(int b) const { return pref[b] + beta * spref[b]; }
    __device__ __forceinline__ long long unit_at(int x) const {
        if (x >= cost(B)) return pref[B];
        int lo = 0, hi = B - 1;  // last b with cost(b) <= x: a request with units
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (cost(mid) <= x) lo = mid;
            else hi = mid - 1;
        }
        const int nt = (pref[lo + 1] - pref[lo]) / (spref[lo + 1] - spref[lo]);
        const int local = x - cost(lo);
        const int seg = local / (nt + beta);
        const int off = local - seg * (nt + beta) - beta;
        return pref[lo] + seg * nt + (off > 0 ? off : 0);
    }
    __device__ __forceinline__ long long range_lo(long long c) const {
        if (beta == 0) return muldiv(c, pref[B], G);  // an even split of the units
        return unit_at((int)muldiv(c, cost(B), G));
    }
    // The CTA holding the last unit of segment [s0, s1) of request b: that
    // unit's cost position x lies in CTA c's cost interval for
    // c = ((x + 1) G - 1) / C, and the unit ranges follow the cost intervals.
    __device__ __forceinline__ long long owner_of_seg_end(int b, long long s0, long long s1) const {
        const int nt = (int)(s1 - s0);
        const int seg = (int)((s0 - pref[b]) / nt);
        const long long x = (long long)cost(b) + (long long)(seg + 1) * (nt + beta) - 1;
        return ((x + 1) * G - 1) / cost(B);
    }
};
__device__ __forceinline__ Split make_split(const int *s_pref, const int *s_spref, int B, int G) {
    const int W = s_pref[B];
    int beta = W / (2 * G);
    if (beta > kSegCostMax) beta = kSegCostMax;
    if (W >= kSegCostOff * G) beta = 0;
    return Split{s_pref, s_spref, B, beta, G};
}

struct Piece {
    int b, kvh, mtile, j0, j1;  // KV tiles [j0, j1) of segment (b, kvh, mtile)
    bool final;                  // the piece is the whole segment
    int slot;                    // partial slot when not final
    long long end;               // unit index after the piece
    long long seg_start, seg_end;  // units of the whole segment
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
    pc.seg_start = seg_start;
    pc.seg_end = seg_end;
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

// Warp-uniform bounded wait for the softmax warps: every lane waits, and the
// warp gives up together if any lane gave up, so warp-wide instructions
// (tcgen05.ld/st, vote) that follow always see the whole warp.
__device__ __forceinline__ bool warp_wait(uint64_t *bar, uint32_t parity, volatile int *abort, long long limit) {
    const bool ok = sm100::mbar_wait(bar, parity, abort, limit);
    return __all_sync(0xffffffffu, ok);
}

// The calling warp arrives once for all its 32 lanes (after every lane's
// prior shared-memory and tensor-memory work is ordered by __syncwarp).
__device__ __forceinline__ void warp_arrive(uint64_t *bar) {
    __syncwarp();
    if ((threadIdx.x & 31) == 0) sm100::mbar_arrive_cnt(bar, 32);
}

// ------------------------------------------------------------------ kernel
template <int D>
__global__ void __launch_bounds__(kAttnThreads, 1)
attn_tc_kernel(AttnArgs a, const ReqInfo *__restrict__ info, const __grid_constant__ CUtensorMap tmk,
               const __grid_constant__ CUtensorMap tmv) {
    pdl_launch_next();
    using namespace sm100;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kSmemBar);
    uint64_t *kfull = bars, *vfull = bars + kNS, *kempty = bars + 2 * kNS, *vempty = bars + 3 * kNS;
    uint64_t *sfull = bars + 4 * kNS, *pfull = sfull + 2, *qready = pfull + 2;
    uint64_t *ofree = qready + 1, *drain = ofree + 1;
    uint64_t *mxready = drain + 1, *lready = mxready + 2;  // softmax warpgroup exchanges
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + kSmemMisc);
    volatile int *s_abort = reinterpret_cast<volatile int *>(smem + kSmemMisc + 4);
    int *s_pref = reinterpret_cast<int *>(smem + kSmemPref);
    int *s_spref = s_pref + (a.B + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        for (int s = 0; s < kNS; ++s) {
            mbar_init(&kfull[s], 1);
            mbar_init(&vfull[s], 1);
            mbar_init(&kempty[s], kSoftThreads);  // released by the softmax warps
            mbar_init(&vempty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&sfull[s], 1);
            mbar_init(&pfull[s], kSoftThreads);
        }
        mbar_init(qready, kSoftThreads);
        mbar_init(ofree, kSoftThreads);
        mbar_init(drain, 1);
        mbar_init(&mxready[0], kSoftThreads);
        mbar_init(&mxready[1], kSoftThreads);
        mbar_init(lready, kSoftThreads);
        *s_abort = 0;
        fence_mbar_init();
    }
    if (warp == kMmaWarp) tmem_alloc(s_tmem, kTmemCols);
    if (warp == kTmaWarp && lane == 0) {
        prefetch_tmap(&tmk);
        prefetch_tmap(&tmv);
    }
    pdl_wait_prev();  // the prologue above touches no global memory
    unit_prefix(info, a.B, s_pref, s_spref);  // contains __syncthreads
    tc_fence_after();
    const uint32_t tmem = *s_tmem;
    const long long W = s_pref[a.B];
    const long long Gc = gridDim.x, c = blockIdx.x;
    const Split split = make_split(s_pref, s_spref, a.B, (int)Gc);
    const long long u0 = split.range_lo(c), u1 = split.range_lo(c + 1);
    const int G = a.Hq / a.Hkv;
    constexpr uint32_t kTileTx = (uint32_t)kBN * D * 2;
    constexpr int kKB = D / 64;  // 64-column swizzle blocks per row

    if (warp == kTmaWarp) {
        // ---------------------------------------------------------- TMA producer
        if (lane == 0) {
            long long g = 0;
            bool ok = true;
            // K/V of a segment with a single row tile is read once per launch;
            // when the launch's K/V is large next to L2 it is streamed with
            // evict-first, so it does not push the rest out of L2
            const uint64_t once = l2_evict_first_policy();
            for (long long u = u0; u < u1 && ok;) {
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                const long long kv0 = a.kv_off[pc.b];
                const bool reread = !a.kv_stream || info[pc.b].mt > 1;  // kept in L2
                for (int jt = pc.j0; jt < pc.j1; ++jt, ++g) {
                    const int st = (int)(g % kNS);
                    const uint32_t free_par = (uint32_t)(((g / kNS) & 1) ^ 1);
                    const int row = (int)(kv0 + (long long)jt * kBN);
                    unsigned char *sk = smem + kSmemK + st * kTileBytes;
                    unsigned char *sv = smem + kSmemV + st * kTileBytes;
                    // K is released as soon as S = Q K^T of the tile is done, V after P V
                    if (!(ok = mbar_wait(&kempty[st], free_par, s_abort, a.wait_limit))) break;
                    mbar_expect_tx(&kfull[st], kTileTx);
#pragma unroll
                    for (int kb = 0; kb < kKB; ++kb) {
                        if (reread) tma_load_3d(sk + kb * 16384, &tmk, &kfull[st], kb * 64, pc.kvh, row);
                        else tma_load_3d_hint(sk + kb * 16384, &tmk, &kfull[st], kb * 64, pc.kvh, row, once);
                    }
                    if (!(ok = mbar_wait(&vempty[st], free_par, s_abort, a.wait_limit))) {
                        volatile int no_abort = 0;  // this tile's K copy is in flight: let it land
                        mbar_wait(&kfull[st], (uint32_t)((g / kNS) & 1), &no_abort, kWaitLimit);
                        break;
                    }
                    mbar_expect_tx(&vfull[st], kTileTx);
#pragma unroll
                    for (int kb = 0; kb < kKB; ++kb) {
                        if (reread) tma_load_3d(sv + kb * 16384, &tmv, &vfull[st], kb * 64, pc.kvh, row);
                        else tma_load_3d_hint(sv + kb * 16384, &tmv, &vfull[st], kb * 64, pc.kvh, row, once);
                    }
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
        __syncwarp();
        if (lane == 1) {  // after the producer loop: off the critical path
            // the split segment this CTA starts (its last piece, when that piece
            // begins inside the range and ends past it), for attn_combine
            CombJob job{W, -1, 0, 0, 0, 0, 0, 0, 0};
            if (u0 < u1) {
                const Piece pl = piece_at(info, s_pref, a.B, u1 - 1, u0, u1, c);
                if (pl.seg_start >= u0 && pl.seg_end > u1) {
                    job.b = pl.b;
                    job.kvh = pl.kvh;
                    job.mtile = pl.mtile;
                    job.n0 = a.node_off[pl.b];
                    job.N = a.node_off[pl.b + 1] - job.n0;
                    job.first_slot = (int)(2 * c + (pl.seg_start > u0 ? 1 : 0));
                    job.c1 = (int)split.owner_of_seg_end(pl.b, pl.seg_start, pl.seg_end);
                }
            }
            a.jobs[c] = job;
            a.ranges[c] = make_int2((int)u0, (int)u1);
        }
    } else if (warp == kMmaWarp) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kBM, kBN, false);
            constexpr uint32_t idO = idesc_bf16_f32(kBM, D, true);
            const uint32_t q_tm = tmem + kTmQ;
            long long g = 0;
            int piece = 0;
            bool ok = true;
            auto issue_s = [&](long long gt) -> bool {
                const int st = (int)(gt % kNS);
                if (!mbar_wait(&kfull[st], (uint32_t)((gt / kNS) & 1), s_abort, a.wait_limit)) return false;
                tc_fence_after();
                const uint32_t k_addr = smem_u32(smem + kSmemK + st * kTileBytes);
                const uint32_t d_s = tmem + kTmS + (uint32_t)(gt & 1) * 128;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (uint32_t)((kk >> 2) * 16384 + (kk & 3) * 32);
                    umma_ts(d_s, q_tm + kk * 8, sdesc_sw128(k_addr + off, 16, 1024), idS, kk > 0);
                }
                umma_commit(&sfull[gt & 1]);
                return true;
            };
            for (long long u = u0; u < u1 && ok; ++piece) {
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                const int n = pc.j1 - pc.j0;
                if (!(ok = mbar_wait(qready, (uint32_t)(piece & 1), s_abort, a.wait_limit))) break;
                tc_fence_after();
                if (!(ok = issue_s(g))) break;
                for (int tl = 0; tl < n && ok; ++tl) {
                    const long long gt = g + tl;
                    if (tl + 1 < n && !(ok = issue_s(gt + 1))) break;
                    const int st = (int)(gt % kNS);
                    if (!(ok = mbar_wait(&pfull[gt & 1], (uint32_t)((gt >> 1) & 1), s_abort, a.wait_limit))) break;
                    if (!(ok = mbar_wait(&vfull[st], (uint32_t)((gt / kNS) & 1), s_abort, a.wait_limit))) break;
                    if (tl == 0 && piece > 0 &&
                        !(ok = mbar_wait(ofree, (uint32_t)((piece - 1) & 1), s_abort, a.wait_limit)))
                        break;
                    tc_fence_after();
                    const uint32_t v_addr = smem_u32(smem + kSmemV + st * kTileBytes);
                    const uint32_t p_tm = tmem + kTmS + (uint32_t)(gt & 1) * 128;
#pragma unroll
                    for (int ks = 0; ks < kBN / 16; ++ks)
                        umma_ts(tmem + kTmO, p_tm + ks * 8, sdesc_sw128(v_addr + ks * 2048, 16384, 1024), idO,
                                (tl > 0 || ks > 0) ? 1u : 0u);
                    umma_commit(&vempty[st]);
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
        // P V of tile t commits vempty[t % kNS] (which also frees V's stage);
        // the softmax waits on it when it must read O (a rescale or the
        // epilogue).  Once S of tile t has been seen complete, every P V up to
        // t - 2 is complete (S_t is issued after P V_{t-2}), and P V of t + 3
        // needs this thread's own P, so the barrier has exactly the asked
        // phase pending: the parity wait is unambiguous.
        // Warpgroup hw (0 or 1) owns keys [64 hw, 64 hw + 64) of every tile,
        // O columns [hw D/2, (hw + 1) D/2) for rescales and the epilogue, and
        // its own partial row sum; both keep the same reference maximum.
        // The per-tile maxima and the final sums are exchanged through
        // shared memory guarded by mbarriers (mxready[tile & 1], lready).
        __shared__ float s_mx[2][2][kBM];  // [tile parity][warpgroup][row]
        __shared__ float s_l[2][kBM];
        const int r = tid & (kBM - 1);      // row of the tile == TMEM lane
        const int hw = tid >> 7;            // warpgroup
        const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
        const float cexp = a.scale * 1.4426950408889634f;  // scores -> log2 domain (scale > 0)
        constexpr int kHalfO = D / 2;       // O columns per warpgroup
        long long g = 0;
        int piece = 0;
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

            // Q row -> TMEM (bf16 pairs, 64 elements per 32 columns; zero past the tile)
            if (hw < D / 64) {
                const uint4 *qp = reinterpret_cast<const uint4 *>(a.q + ((long long)(n0 + i) * a.Hq + h) * D) + hw * 8;
                uint32_t x[32];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const uint4 v = valid ? qp[e] : make_uint4(0, 0, 0, 0);
                    x[4 * e + 0] = v.x;
                    x[4 * e + 1] = v.y;
                    x[4 * e + 2] = v.z;
                    x[4 * e + 3] = v.w;
                }
                tmem_st32(tmem + lane_off + kTmQ + hw * 32, x);
                tmem_wait_st();
            }
            uint32_t anc[kAncWords];
#pragma unroll
            for (int w = 0; w < kAncWords; ++w) anc[w] = valid ? a.anc[(long long)(n0 + i) * kAncWords + w] : 0u;
            tc_fence_before();
            warp_arrive(qready);

            float m_used = -INFINITY, l = 0.f;
            const int n = pc.j1 - pc.j0;
            for (int tl = 0; tl < n; ++tl) {
                const long long gt = g + tl;
                const int buf = (int)(gt & 1);
                const int jt = pc.j0 + tl;
                if (!(ok = warp_wait(&sfull[buf], (uint32_t)((gt >> 1) & 1), s_abort, a.wait_limit))) break;
                tc_fence_after();
                // S of this tile is complete, so its K stage is free: released
                // here rather than by a second commit on the MMA thread
                warp_arrive(&kempty[(int)(gt % kNS)]);
                const uint32_t s_tm = tmem + lane_off + kTmS + (uint32_t)buf * 128;
                float s[64];
                {  // both halves in flight, one wait
                    uint32_t xa[32], xb[32];
                    tmem_ld32(s_tm + hw * 64, xa);
                    tmem_ld32(s_tm + hw * 64 + 32, xb);
                    tmem_wait_ld();
                    tmem_regs_ready(xa);
                    tmem_regs_ready(xb);
#pragma unroll
                    for (int e = 0; e < 32; ++e) {
                        s[e] = __uint_as_float(xa[e]);
                        s[32 + e] = __uint_as_float(xb[e]);
                    }
                }
                // raw-score maximum over this half's visible keys
                float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                const int key0 = jt * kBN + hw * 64;
                if (key0 + 64 <= S) {  // prefix-only: nothing to mask
#pragma unroll
                    for (int j = 0; j < 64; ++j) mx4[j & 3] = fmaxf(mx4[j & 3], s[j]);
                } else {
#pragma unroll
                    for (int ch = 0; ch < 2; ++ch) {
                        const uint32_t msk = tree_window(anc, key0 + ch * 32 - S);
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const float v = ((msk >> e) & 1u) ? s[ch * 32 + e] : -INFINITY;
                            s[ch * 32 + e] = v;
                            mx4[e & 3] = fmaxf(mx4[e & 3], v);
                        }
                    }
                }
                // exchange the two halves' maxima through an mbarrier (bounded
                // wait: a named barrier could not give up if a peer aborted)
                s_mx[buf][hw][r] = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
                warp_arrive(&mxready[buf]);
                if (!(ok = warp_wait(&mxready[buf], (uint32_t)((gt >> 1) & 1), s_abort, a.wait_limit))) break;
                const float mt = fmaxf(s_mx[buf][0][r], s_mx[buf][1][r]) * cexp;
                // lazy rescale: move the reference maximum only when it grows by
                // more than 2^8; tcgen05.ld/st are warp-wide, so the O pass runs
                // when any row of the warp needs it (factor 1 for the others)
                const bool grow = mt > m_used + 8.f;
                const float corr = grow ? ex2(m_used - mt) : 1.f;  // 0 when m_used is -inf
                if (tl > 0 && __any_sync(0xffffffffu, grow)) {
                    const long long pv = gt - 1;  // O must hold PV of the previous tile
                    if (!(ok = warp_wait(&vempty[(int)(pv % kNS)], (uint32_t)((pv / kNS) & 1), s_abort, a.wait_limit))) break;
                    tc_fence_after();
#pragma unroll
                    for (int ch = 0; ch < kHalfO / 32; ++ch) {
                        uint32_t x[32];
                        const uint32_t o_tm = tmem + lane_off + kTmO + hw * kHalfO + ch * 32;
                        tmem_ld32(o_tm, x);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 32; ++e) x[e] = __float_as_uint(__uint_as_float(x[e]) * corr);
                        tmem_st32(o_tm, x);
                    }
                    tmem_wait_st();
                }
                if (grow) {
                    l *= corr;
                    m_used = mt;
                }
                const float nb = (m_used == -INFINITY) ? 0.f : -m_used;
                float sum4[4] = {0.f, 0.f, 0.f, 0.f};
                uint32_t x[32];
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const float p0 = ex2(fmaf(s[2 * e], cexp, nb));
                    const float p1 = ex2(fmaf(s[2 * e + 1], cexp, nb));
                    sum4[e & 3] += p0 + p1;
                    x[e] = pack_bf16x2(p0, p1);
                }
                tmem_st32(s_tm + hw * 32, x);
                l += (sum4[0] + sum4[1]) + (sum4[2] + sum4[3]);
                tmem_wait_st();
                tc_fence_before();
                warp_arrive(&pfull[buf]);
            }
            if (!ok) break;
            // epilogue: the row sum is the two warpgroups' partial sums
            s_l[hw][r] = l;
            warp_arrive(lready);
            if (!(ok = warp_wait(lready, (uint32_t)(piece & 1), s_abort, a.wait_limit))) break;
            const float lt = s_l[0][r] + s_l[1][r];
            {
                const long long pv = g + n - 1;  // wait for PV of the last tile
                if (!(ok = warp_wait(&vempty[(int)(pv % kNS)], (uint32_t)((pv / kNS) & 1), s_abort, a.wait_limit))) break;
            }
            tc_fence_after();
            const long long orow = (long long)(n0 + i) * a.Hq + h;
            const long long prow = (long long)pc.slot * kBM + r;
            const float f = pc.final ? ((lt > 0.f) ? 1.f / lt : 0.f) : 1.f;
            uint32_t xo[kHalfO / 32][32];  // this half of O, all chunks in flight, one wait
#pragma unroll
            for (int ch = 0; ch < kHalfO / 32; ++ch) tmem_ld32(tmem + lane_off + kTmO + hw * kHalfO + ch * 32, xo[ch]);
            tmem_wait_ld();
#pragma unroll
            for (int ch = 0; ch < kHalfO / 32; ++ch) tmem_regs_ready(xo[ch]);
            if (a.stage) {
                // rows leave through shared memory so that a store instruction
                // writes 8 rows x 64 contiguous bytes instead of 32 rows x 16:
                // the warp stages 32 rows x 16 columns (row stride 20 floats,
                // conflict-free writes), then each lane stores 4 columns of a row
                float *dst = (pc.final ? a.out + orow * D : a.part_o + prow * D) + hw * kHalfO;
                const unsigned vmask = __ballot_sync(0xffffffffu, valid);
                float *stage = reinterpret_cast<float *>(smem + attn_stage_offset(a.B)) + warp * kStageFloats;
#pragma unroll
                for (int c16 = 0; c16 < kHalfO / 16; ++c16) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const uint32_t *x = &xo[c16 >> 1][(c16 & 1) * 16 + 4 * e];
                        *reinterpret_cast<float4 *>(stage + lane * 20 + 4 * e) =
                            make_float4(__uint_as_float(x[0]) * f, __uint_as_float(x[1]) * f,
                                        __uint_as_float(x[2]) * f, __uint_as_float(x[3]) * f);
                    }
                    __syncwarp();
#pragma unroll
                    for (int it = 0; it < 4; ++it) {
                        const int rw = it * 8 + (lane >> 2);  // row of the warp this lane writes
                        float *d = reinterpret_cast<float *>(
                            __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(dst), rw));
                        const float4 v4 = *reinterpret_cast<const float4 *>(stage + rw * 20 + (lane & 3) * 4);
                        if ((vmask >> rw) & 1u) *reinterpret_cast<float4 *>(d + c16 * 16 + (lane & 3) * 4) = v4;
                    }
                    __syncwarp();
                }
            }
#pragma unroll
            for (int ch = 0; ch < kHalfO / 32; ++ch) {
                const int col = hw * kHalfO + ch * 32;
                if (valid && !a.stage) {
                    float4 *dst = pc.final ? reinterpret_cast<float4 *>(a.out + orow * D + col)
                                           : reinterpret_cast<float4 *>(a.part_o + prow * D + col);
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        dst[e] = make_float4(__uint_as_float(xo[ch][4 * e]) * f, __uint_as_float(xo[ch][4 * e + 1]) * f,
                                             __uint_as_float(xo[ch][4 * e + 2]) * f,
                                             __uint_as_float(xo[ch][4 * e + 3]) * f);
                }
            }
            if (valid && hw == 0) {
                const float m_nat = m_used * 0.6931471805599453f;
                if (pc.final) {
                    a.lse[orow] = m_nat + __logf(lt);
                } else {
                    a.part_m[prow] = m_used == -INFINITY ? -INFINITY : m_nat;
                    a.part_l[prow] = lt;
                }
            }
            tc_fence_before();
            warp_arrive(ofree);
            g += n;
            u = pc.end;
        }
        if (!ok && tid == 0) {
            for (long long u = u0; u < u1;) {  // flag every request this CTA touches
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                atomicOr(&a.status[pc.b], RS_ST_TIMEOUT);
                u = pc.end;
            }
        }
    }
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace rs
