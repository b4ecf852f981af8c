// attn_pair.cuh -- the two-row-tile form of the tensor-core attention core,
// for launches whose requests have more than one 128-row tile per KV head
// (GQA groups over long trees, batched trees).
//
// A segment is (request, KV head, pair of 128-row tiles): rows
// [256 p, 256 p + 256) of the request's (node, q-head-in-group) rows.  Each
// 128-key K/V tile the CTA loads is used by both row tiles, and the single
// MMA-issuing thread alternates between them so that one tile's softmax runs
// while the tensor core works on the other tile:
//     S_A(t)  S_B(t)  PV_A(t)  S_A(t+1)  PV_B(t)  S_B(t+1)  PV_A(t+1) ...
// Each softmax has two MMA bursts of time (PV of the other tile and its next
// S) between its S and the PV that consumes its P, and every wait and commit
// of the issuing thread is spread over twice the MMA work of the one-tile
// kernel.  A pair whose second tile is empty (the last pair of a request with
// an odd tile count, or a request of one tile) runs in "half" mode: one tile,
// its S double-buffered in the two S columns ranges, in the order of the
// one-tile kernel (S(t+1) issued before PV(t)).
//
// Warps: 0-3 softmax of tile A (thread = row, all 128 keys of a tile),
// 4-7 softmax of tile B (idle in half mode), 8 TMA producer, 9 MMA issuer,
// 10-11 idle.  A softmax thread holds a whole 128-key row of S, so the
// producer warpgroup (8-11) gives registers up to the softmax warpgroups
// (setmaxnreg: 128 x 72 + 256 x 216 = 384 x 168, the launch's budget).
// Tensor memory (512 columns): O_A [0, 128), O_B [128, 256), S/P buffer 0
// [256, 384), S/P buffer 1 [384, 512); in full mode buffer x belongs to tile
// x, in half mode tile A uses them alternately.  Q has no room in tensor
// memory, so both Q tiles sit in shared memory (K-major, 128-byte swizzle,
// written by the softmax threads) and S = Q K^T reads both operands from
// shared memory; P stays in tensor memory for O += P V as in the one-tile
// kernel.  K and V use a two-stage ring (a K/V tile now serves 256 rows).
// When G = Hq / Hkv divides 128 a Q tile is whole nodes and the TMA warp
// copies it (qfull / qfree barriers): a CTA's first Q tiles right after its
// first K tile when K/V stays in L2 (the buffers are still unused), all
// others after the piece's second K/V tile, each once the tile's warps have
// finished their epilogue, which stages O rows in the same buffer;
// otherwise the softmax threads write it (qready).
//
// Barrier phases: every role walks the same pieces in the same order and
// counts, per S buffer, how many S it has held (use counts), so a wait's
// parity is always that of the next pending phase.  The tile-B warps wait for
// the end of every piece (ofree) before they start the next one, which keeps
// them from running a piece ahead of the tile-A warps through pieces in
// which they have nothing to do.
#pragma once

#include "attn_core.cuh"

namespace rs {

constexpr int kPairRows = 2 * kBM;  // rows per segment
constexpr int kPairNS = 2;          // K/V ring stages
// Cost weights of a K/V tile in the work split: a full pair runs two row
// tiles on it, a half pair one.  When K/V tiles come from L2 (re-read by
// several pairs) the tile costs mostly its compute: a fit of per-CTA
// lifetimes (global timer) on GQA-16K with a cold L2 gave 1.49 and 0.90 us
// per full and half pair tile (weights 5 : 3; warm-L2 clock stamps, 3.43 k
// and 1.92 k cycles, suggested 9 : 5).  When they stream from HBM once
// (kv_stream) a tile costs mostly its bytes, the same for both: the fit on
// the batched workload gave 1.61 and 1.09 us (3 : 2).  A segment start is
// charged beta = min(cap, W / 2G) half-pair tiles: the fits put a piece
// boundary at ~9 half-pair tiles from L2 and ~4 when streaming (the
// streaming K/V copies run on through the boundary).
constexpr int kPairWF = 5, kPairWH = 3;              // the larger pair, for bounds
constexpr int kPairWFStream = 3, kPairWHStream = 2;
constexpr int kPairSegCostStream = 4;  // the cap of beta when streaming (kSegCostMax otherwise)
constexpr int kPairMaxB = 2048;  // requests per call in this form (three prefixes in shared memory)
constexpr int kPairThreads = 384;
constexpr uint32_t kPairRegsSoft = 216, kPairRegsProd = 72;
static_assert(2 * 128 * kPairRegsSoft + 128 * kPairRegsProd == kPairThreads * 168, "register split");
constexpr int kP2SmemK = 0;
constexpr int kP2SmemV = kP2SmemK + kPairNS * kTileBytes;
constexpr int kP2SmemQ = kP2SmemV + kPairNS * kTileBytes;  // Q tile x at + x * kTileBytes
constexpr int kP2SmemBar = kP2SmemQ + 2 * kTileBytes;
constexpr int kP2NumBars = 6 * kPairNS + 7;
constexpr int kP2SmemMisc = kP2SmemBar + kP2NumBars * 8;  // tmem base, abort flag
constexpr int kP2SmemPref = kP2SmemMisc + 16;
constexpr uint32_t kTm2S = 256;  // S/P buffer b at kTm2S + 128 b; O of tile x at 128 x
// unit, segment and weighted-unit prefixes over the requests: 3 (B + 1) ints
inline size_t attn_pair_smem_bytes(int B) { return 1024 + kP2SmemPref + 3 * (size_t)(B + 1) * sizeof(int); }

// Exclusive prefixes over the requests of their units (s_pref), segments
// (s_spref) and weighted units (s_apref: wf per unit of a full pair, wh per
// unit of a half pair).
__device__ inline void pair_prefix(const ReqInfo *__restrict__ info, int B, int Hkv, int wf, int wh, int *s_pref,
                                   int *s_spref, int *s_apref) {
    __shared__ int s_carry[3];
    __shared__ int s_w[3][32];
    if (threadIdx.x == 0) s_carry[0] = s_carry[1] = s_carry[2] = 0;
    __syncthreads();
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nw = (blockDim.x + 31) >> 5;
    for (int base = 0; base < B; base += blockDim.x) {
        const int i = base + threadIdx.x;
        int v[3] = {0, 0, 0};
        if (i < B) {
            const ReqInfo ri = info[i];
            if (ri.units > 0) {
                v[0] = ri.units;
                v[1] = ri.units / ri.nt;
                const bool last_half = ri.rows - (ri.mt - 1) * kPairRows <= kBM;
                v[2] = wf * ri.units - (last_half ? (wf - wh) * Hkv * ri.nt : 0);
            }
        }
        int x[3] = {v[0], v[1], v[2]};
#pragma unroll
        for (int k = 0; k < 3; ++k) {
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, x[k], o);
                if (lane >= o) x[k] += y;
            }
            if (lane == 31) s_w[k][warp] = x[k];
        }
        __syncthreads();
        if (warp == 0) {
#pragma unroll
            for (int k = 0; k < 3; ++k) {
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
        int incl[3];
#pragma unroll
        for (int k = 0; k < 3; ++k) incl[k] = s_carry[k] + s_w[k][warp] + x[k];
        if (i < B) {
            s_pref[i + 1] = incl[0];
            s_spref[i + 1] = incl[1];
            s_apref[i + 1] = incl[2];
        }
        __syncthreads();
        if (threadIdx.x == blockDim.x - 1) {
#pragma unroll
            for (int k = 0; k < 3; ++k) s_carry[k] = incl[k];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) s_pref[0] = s_spref[0] = s_apref[0] = 0;
    __syncthreads();
}

// The work split of the pair form: the one-tile form's cost split with
// weighted units.  Request b occupies cost positions [cost(b), cost(b + 1)),
// cost(b) = apref[b] + beta spref[b]; within it the KV heads follow each
// other, and within a KV head its pairs, each costing nt w + beta (w = wf,
// or wh for a half pair, which can only be the last).
struct PairSplit {
    const int *pref, *spref, *apref;
    int B, beta, G, Hkv, wf, wh;
    struct Req {
        int nt, mt;
        bool last_half;
        int cF, cL, ck;  // full-pair, last-pair and per-KV-head costs
    };
    __device__ __forceinline__ int cost(int b) const { return apref[b] + beta * spref[b]; }
    __device__ __forceinline__ Req req(int b) const {
        Req r;
        const int units = pref[b + 1] - pref[b], segs = spref[b + 1] - spref[b];
        r.nt = units / segs;
        r.mt = segs / Hkv;
        r.last_half = apref[b + 1] - apref[b] < wf * units;
        r.cF = r.nt * wf + beta;
        r.cL = r.nt * (r.last_half ? wh : wf) + beta;
        r.ck = (r.mt - 1) * r.cF + r.cL;
        return r;
    }
    __device__ __forceinline__ long long unit_at(long long x) const {
        if (x >= cost(B)) return pref[B];
        int lo = 0, hi = B - 1;  // last b with cost(b) <= x: a request with units
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (cost(mid) <= x) lo = mid;
            else hi = mid - 1;
        }
        const Req r = req(lo);
        const int local = (int)(x - cost(lo));
        const int kvh = local / r.ck;
        int rem = local - kvh * r.ck;
        int p = rem / r.cF;
        if (p > r.mt - 1) p = r.mt - 1;
        rem -= p * r.cF;
        const int w = (p == r.mt - 1 && r.last_half) ? wh : wf;
        const int off = rem - beta;
        return pref[lo] + (long long)(kvh * r.mt + p) * r.nt + (off > 0 ? off / w : 0);
    }
    __device__ __forceinline__ long long range_lo(long long c) const { return unit_at(muldiv(c, cost(B), G)); }
    // The CTA holding the last unit of segment [s0, s1) of request b: the
    // segment's cost interval ends at x_end, and CTA c's range holds the unit
    // at cost position x_end - 1 for c = (x_end G - 1) / C.
    __device__ __forceinline__ long long owner_of_seg_end(int b, long long s0, long long /*s1*/) const {
        const Req r = req(b);
        const int sg = (int)((s0 - pref[b]) / r.nt);
        const int kvh = sg / r.mt, p = sg - kvh * r.mt;
        const int w = (p == r.mt - 1 && r.last_half) ? wh : wf;
        const long long x_end = (long long)cost(b) + (long long)kvh * r.ck + (long long)p * r.cF + beta + r.nt * w;
        return (x_end * G - 1) / cost(B);
    }
};

// ------------------------------------------------------------------ kernel
template <int D>
__global__ void __launch_bounds__(kPairThreads, 1)
attn_pair_kernel(AttnArgs a, const ReqInfo *__restrict__ info, const __grid_constant__ CUtensorMap tmk,
                 const __grid_constant__ CUtensorMap tmv, const __grid_constant__ CUtensorMap tmq) {
    pdl_launch_next();
    using namespace sm100;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                            ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kP2SmemBar);
    uint64_t *kfull = bars, *vfull = bars + kPairNS, *kempty = bars + 2 * kPairNS, *vempty = bars + 3 * kPairNS;
    uint64_t *sfull = bars + 4 * kPairNS, *pfull = sfull + 2;
    uint64_t *qready = pfull + 2, *ofree = qready + 1, *drain = ofree + 1;
    uint64_t *qfull = drain + 1, *qfree = qfull + 2;  // Q tiles copied by TMA (a.q_tma)
    uint32_t *s_tmem = reinterpret_cast<uint32_t *>(smem + kP2SmemMisc);
    volatile int *s_abort = reinterpret_cast<volatile int *>(smem + kP2SmemMisc + 4);
    int *s_pref = reinterpret_cast<int *>(smem + kP2SmemPref);
    int *s_spref = s_pref + (a.B + 1);
    int *s_apref = s_spref + (a.B + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        for (int s = 0; s < kPairNS; ++s) {
            mbar_init(&kfull[s], 1);
            mbar_init(&vfull[s], 1);
            mbar_init(&kempty[s], kBM);  // the softmax warps that see the last S reading K arrive
            mbar_init(&vempty[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&sfull[s], 1);
            mbar_init(&pfull[s], kBM);
        }
        mbar_init(qready, kSoftThreads);
        for (int x = 0; x < 2; ++x) {
            mbar_init(&qfull[x], 1);
            mbar_init(&qfree[x], kBM);  // the tile's softmax warps, after their epilogue
        }
        mbar_init(ofree, kSoftThreads);
        mbar_init(drain, 1);
        *s_abort = 0;
        fence_mbar_init();
    }
    if (warp == kMmaWarp) tmem_alloc(s_tmem, kTmemCols);
    if (warp == kTmaWarp && lane == 0) {
        prefetch_tmap(&tmk);
        prefetch_tmap(&tmv);
        if (a.q_tma) prefetch_tmap(&tmq);
    }
    pdl_wait_prev();  // the prologue above touches no global memory
    const int wf = a.kv_stream ? kPairWFStream : kPairWF, wh = a.kv_stream ? kPairWHStream : kPairWH;
    pair_prefix(info, a.B, a.Hkv, wf, wh, s_pref, s_spref, s_apref);  // contains __syncthreads
    tc_fence_after();
    const uint32_t tmem = *s_tmem;
    const long long W = s_pref[a.B];
    const long long Gc = gridDim.x, c = blockIdx.x;
    PairSplit split{s_pref, s_spref, s_apref, a.B, 0, (int)Gc, a.Hkv, wf, wh};
    {
        int beta = (int)muldiv(W, 1, 2 * Gc);
        const int cap = a.kv_stream ? kPairSegCostStream : kSegCostMax;
        if (beta > cap) beta = cap;
        split.beta = wh * beta;  // in the weighted units (a half-pair K/V tile weighs wh)
    }
    // the range's two ends in two lanes at once: each is a chain of dependent
    // divisions on every CTA's path to its first tile (0.6 us apart when
    // computed in turn), and with them in one call the compiler also spills
    // less (GQA-16K call 66.4 -> 64.5 us, batched 107.2 -> 105.4 us)
    const long long u_end = split.range_lo(c + (lane & 1));
    const long long u0 = __shfl_sync(0xffffffffu, u_end, 0), u1 = __shfl_sync(0xffffffffu, u_end, 1);
    const int G = a.Hq / a.Hkv;
    constexpr uint32_t kTileTx = (uint32_t)kBN * D * 2;
    constexpr int kKB = D / 64;  // 64-column swizzle blocks per row

    if (warp >= kTmaWarp) {
      reg_dealloc<kPairRegsProd>();
      if (warp == kTmaWarp) {
        // ---------------------------------------------------------- TMA producer
        if (lane == 0) {
            uint32_t g = 0;
            uint32_t quse[2] = {0, 0};  // Q tiles copied into buffers A and B so far
            bool ok = true;
            const uint64_t once = l2_evict_first_policy();
            for (long long u = u0; u < u1 && ok;) {
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                const long long kv0 = a.kv_off[pc.b];
                const ReqInfo ri = info[pc.b];
                const bool reread = !a.kv_stream || ri.mt > 1;  // kept in L2
                const bool full = ri.rows - pc.mtile * kPairRows > kBM;
                // Where K/V stays in L2 the CTA's first Q tiles follow its first
                // K tile: every CTA starts at once and S needs only K and Q.
                // Otherwise, and for later pieces, they follow the second K/V
                // tile (below).
                const bool q_early = a.q_tma && u == u0 && !a.kv_stream;
                for (int jt = pc.j0; jt < pc.j1; ++jt, ++g) {
                    const int st = (int)(g & 1);
                    const uint32_t free_par = ((g >> 1) & 1) ^ 1;
                    const int row = (int)(kv0 + (long long)jt * kBN);
                    unsigned char *sk = smem + kP2SmemK + st * kTileBytes;
                    unsigned char *sv = smem + kP2SmemV + st * kTileBytes;
                    if (!(ok = mbar_wait(&kempty[st], free_par, s_abort, a.wait_limit))) break;
                    mbar_expect_tx(&kfull[st], kTileTx);
#pragma unroll
                    for (int kb = 0; kb < kKB; ++kb) {
                        if (reread) tma_load_3d(sk + kb * 16384, &tmk, &kfull[st], kb * 64, pc.kvh, row);
                        else tma_load_3d_hint(sk + kb * 16384, &tmk, &kfull[st], kb * 64, pc.kvh, row, once);
                    }
                    if (q_early && jt == pc.j0) {  // the buffers are unused: no wait
                        const int node0 = a.node_off[pc.b] + (pc.mtile * kPairRows) / G;
                        for (int x = 0; x < (full ? 2 : 1); ++x) {
                            ++quse[x];
                            mbar_expect_tx(&qfull[x], (uint32_t)kBM * D * 2);
#pragma unroll
                            for (int kb = 0; kb < kKB; ++kb)
                                tma_load_3d(smem + kP2SmemQ + x * kTileBytes + kb * 16384, &tmq, &qfull[x], kb * 64,
                                            pc.kvh * G, node0 + x * (kBM / G));
                        }
                    }
                    if (!(ok = mbar_wait(&vempty[st], free_par, s_abort, a.wait_limit))) {
                        volatile int no_abort = 0;  // this tile's K copy is in flight: let it land
                        mbar_wait(&kfull[st], (g >> 1) & 1, &no_abort, kWaitLimit);
                        break;
                    }
                    mbar_expect_tx(&vfull[st], kTileTx);
#pragma unroll
                    for (int kb = 0; kb < kKB; ++kb) {
                        if (reread) tma_load_3d(sv + kb * 16384, &tmv, &vfull[st], kb * 64, pc.kvh, row);
                        else tma_load_3d_hint(sv + kb * 16384, &tmv, &vfull[st], kb * 64, pc.kvh, row, once);
                    }
                    if (a.q_tma && !q_early && jt == (pc.j1 - pc.j0 >= 2 ? pc.j0 + 1 : pc.j0)) {
                        // the piece's Q tiles, once its first two K/V copies are
                        // under way (they wait only for ring stages), each after
                        // its buffer's previous piece has left it: rows (node,
                        // head in group) of 128 / G nodes x G heads, the layout
                        // the S MMA reads; rows past the request's end belong to
                        // no output and are never stored
                        const int node0 = a.node_off[pc.b] + (pc.mtile * kPairRows) / G;
                        for (int x = 0; x < (full ? 2 : 1) && ok; ++x) {
                            if (quse[x] > 0 &&
                                !(ok = mbar_wait(&qfree[x], (quse[x] - 1) & 1, s_abort, a.wait_limit)))
                                break;
                            ++quse[x];
                            mbar_expect_tx(&qfull[x], (uint32_t)kBM * D * 2);
#pragma unroll
                            for (int kb = 0; kb < kKB; ++kb)
                                tma_load_3d(smem + kP2SmemQ + x * kTileBytes + kb * 16384, &tmq, &qfull[x], kb * 64,
                                            pc.kvh * G, node0 + x * (kBM / G));
                        }
                        if (!ok) break;
                    }
                }
                u = pc.end;
            }
            if (!ok) {  // let the copies already issued land before the CTA exits
                for (uint32_t t = g >= kPairNS ? g - kPairNS : 0; t < g; ++t) {
                    volatile int no_abort = 0;
                    mbar_wait(&kfull[t & 1], (t >> 1) & 1, &no_abort, kWaitLimit);
                    mbar_wait(&vfull[t & 1], (t >> 1) & 1, &no_abort, kWaitLimit);
                }
                for (int x = 0; x < 2; ++x)
                    if (quse[x] > 0) {
                        volatile int no_abort = 0;
                        mbar_wait(&qfull[x], (quse[x] - 1) & 1, &no_abort, kWaitLimit);
                    }
            }
        }
        __syncwarp();
        if (lane == 1) {  // the split segment this CTA starts, for attn_combine
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
            // Shared-memory descriptors: the high words (stride, version,
            // swizzle) are common to K, V and Q; the low words hold the start
            // address >> 4 and the leading byte offset.  The per-call bases
            // pass through an empty asm so that the compiler rebuilds the
            // per-MMA offsets in each burst instead of keeping every
            // combination of stage, tile and K-slice alive in registers.
            const uint64_t dK0 = sdesc_sw128(smem_u32(smem + kP2SmemK), 16, 1024);
            const uint32_t d_hi = (uint32_t)(dK0 >> 32);
            const uint32_t k_lo0 = (uint32_t)dK0;
            const uint32_t q_lo0 = (uint32_t)sdesc_sw128(smem_u32(smem + kP2SmemQ), 16, 1024);
            const uint32_t v_lo0 = (uint32_t)sdesc_sw128(smem_u32(smem + kP2SmemV), 16384, 1024);
            constexpr uint32_t kTileDesc = kTileBytes >> 4;
            uint32_t g = 0;             // KV tiles of the CTA so far
            uint32_t use0 = 0, use1 = 0;  // S held so far by S/P buffers 0 and 1
            uint32_t quse0 = 0, quse1 = 0;  // Q tiles received in buffers A and B
            int piece = 0;
            bool ok = true;
            // S of tile t (stage t & 1) for row tile xq into buffer buf
            auto issue_s = [=](uint32_t t, int xq, int buf) {
                uint32_t k_lo = k_lo0 + (t & 1) * kTileDesc, q_lo = q_lo0 + (uint32_t)xq * kTileDesc;
                asm volatile("" : "+r"(k_lo), "+r"(q_lo));
                const uint32_t d_s = tmem + kTm2S + (uint32_t)buf * 128;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (uint32_t)(((kk >> 2) * 16384 + (kk & 3) * 32) >> 4);
                    umma_ss(d_s, desc_of(q_lo + off, d_hi), desc_of(k_lo + off, d_hi), idS, kk > 0);
                }
                umma_commit(&sfull[buf]);
            };
            // O of row tile xo += P (buffer buf) V of tile t
            auto issue_pv = [=](uint32_t t, int xo, int buf, bool acc) {
                uint32_t v_lo = v_lo0 + (t & 1) * kTileDesc;
                asm volatile("" : "+r"(v_lo));
                const uint32_t p_tm = tmem + kTm2S + (uint32_t)buf * 128;
                const uint32_t o_tm = tmem + (uint32_t)xo * 128;
#pragma unroll
                for (int ks = 0; ks < kBN / 16; ++ks)
                    umma_ts(o_tm, p_tm + ks * 8, desc_of(v_lo + (uint32_t)((ks * 2048) >> 4), d_hi), idO,
                            (acc || ks > 0) ? 1u : 0u);
            };
            for (long long u = u0; u < u1 && ok; ++piece) {
                const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
                const int n = pc.j1 - pc.j0;
                const bool full = info[pc.b].rows - pc.mtile * kPairRows > kBM;
                if (a.q_tma) {  // the piece's Q tiles have landed
                    if (!(ok = mbar_wait(&qfull[0], quse0 & 1, s_abort, a.wait_limit))) break;
                    if (full && !(ok = mbar_wait(&qfull[1], quse1 & 1, s_abort, a.wait_limit))) break;
                    ++quse0;
                    quse1 += full ? 1 : 0;
                } else if (!(ok = mbar_wait(qready, (uint32_t)(piece & 1), s_abort, a.wait_limit))) {
                    break;
                }
                if (!(ok = mbar_wait(&kfull[g & 1], (g >> 1) & 1, s_abort, a.wait_limit))) break;
                tc_fence_after();
                issue_s(g, 0, 0);
                if (full) {
                    issue_s(g, 1, 1);
                    for (int tl = 0; tl < n; ++tl) {
                        const uint32_t t = g + tl;
                        const bool more = tl + 1 < n;
                        if (!(ok = mbar_wait(&pfull[0], (use0 + tl) & 1, s_abort, a.wait_limit))) break;
                        if (!(ok = mbar_wait(&vfull[t & 1], (t >> 1) & 1, s_abort, a.wait_limit))) break;
                        if (tl == 0 && piece > 0 &&
                            !(ok = mbar_wait(ofree, (uint32_t)((piece - 1) & 1), s_abort, a.wait_limit)))
                            break;
                        tc_fence_after();
                        issue_pv(t, 0, 0, tl > 0);
                        if (more) {
                            if (!(ok = mbar_wait(&kfull[(t + 1) & 1], ((t + 1) >> 1) & 1, s_abort, a.wait_limit)))
                                break;
                            tc_fence_after();
                            issue_s(t + 1, 0, 0);
                        }
                        if (!(ok = mbar_wait(&pfull[1], (use1 + tl) & 1, s_abort, a.wait_limit))) break;
                        tc_fence_after();
                        issue_pv(t, 1, 1, tl > 0);
                        umma_commit(&vempty[t & 1]);
                        if (more) issue_s(t + 1, 1, 1);
                    }
                    use0 += n;
                    use1 += n;
                } else {
                    for (int tl = 0; tl < n; ++tl) {
                        const uint32_t t = g + tl;
                        const int b = tl & 1;
                        if (tl + 1 < n) {
                            if (!(ok = mbar_wait(&kfull[(t + 1) & 1], ((t + 1) >> 1) & 1, s_abort, a.wait_limit)))
                                break;
                            tc_fence_after();
                            issue_s(t + 1, 0, b ^ 1);
                        }
                        const uint32_t par = ((b ? use1 : use0) + (tl >> 1)) & 1;
                        if (!(ok = mbar_wait(&pfull[b], par, s_abort, a.wait_limit))) break;
                        if (!(ok = mbar_wait(&vfull[t & 1], (t >> 1) & 1, s_abort, a.wait_limit))) break;
                        if (tl == 0 && piece > 0 &&
                            !(ok = mbar_wait(ofree, (uint32_t)((piece - 1) & 1), s_abort, a.wait_limit)))
                            break;
                        tc_fence_after();
                        issue_pv(t, 0, b, tl > 0);
                        umma_commit(&vempty[t & 1]);
                    }
                    use0 += (n + 1) >> 1;
                    use1 += n >> 1;
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
      }
    } else {
        reg_alloc<kPairRegsSoft>();
        // ---------------------------------------------------------- softmax / epilogue (rows)
        const int x = warp >> 2;            // row tile of this warpgroup
        const int r = tid & (kBM - 1);      // row of the tile == TMEM lane
        const uint32_t lane_off = (uint32_t)((warp & 3) * 32) << 16;
        const float cexp = a.scale * 1.4426950408889634f;  // scores -> log2 domain (scale > 0)
        unsigned char *qs = smem + kP2SmemQ + x * kTileBytes;
        uint32_t g = 0, use0 = 0, use1 = 0;
        int piece = 0;
        bool ok = true;
        for (long long u = u0; u < u1 && ok; ++piece) {
            const Piece pc = piece_at(info, s_pref, a.B, u, u0, u1, c);
            const int n = pc.j1 - pc.j0;
            const int rows = info[pc.b].rows;
            const bool full = rows - pc.mtile * kPairRows > kBM;
            const bool active = x == 0 || full;
            const int rr = pc.mtile * kPairRows + x * kBM + r;
            const bool valid = active && rr < rows;
            const int n0 = a.node_off[pc.b];
            const int S = a.ctx_len[pc.b];
            const int i = valid ? rr / G : 0;
            const int h = pc.kvh * G + (valid ? rr - i * G : 0);
            if (active && !a.q_tma) {
                // Q row -> shared memory, K-major with the 128-byte swizzle: the
                // 16-byte chunk c of 64-column block kb of row r sits at
                // kb * 16384 + r * 128 + ((c ^ (r & 7)) * 16)
                const uint4 *qp = reinterpret_cast<const uint4 *>(a.q + ((long long)(n0 + i) * a.Hq + h) * D);
                uint4 v[D / 8];
#pragma unroll
                for (int e = 0; e < D / 8; ++e) v[e] = valid ? qp[e] : make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int e = 0; e < D / 8; ++e)
                    *reinterpret_cast<uint4 *>(qs + (e >> 3) * 16384 + r * 128 + (((e & 7) ^ (r & 7)) << 4)) = v[e];
                fence_async_smem();
            }
            if (!a.q_tma) warp_arrive(qready);
            if (active) {
                float m_used = -INFINITY, l = 0.f;
                for (int tl = 0; tl < n; ++tl) {
                    const uint32_t t = g + tl;
                    const int jt = pc.j0 + tl;
                    const int b = full ? x : (tl & 1);
                    const uint32_t par = full ? ((b ? use1 : use0) + tl) & 1 : ((b ? use1 : use0) + (tl >> 1)) & 1;
                    const int key0 = jt * kBN;
                    const bool masked = key0 + kBN > S;
                    // the row's ancestor set, for a tile with tree slots: loaded
                    // before the wait for S so that the wait covers its latency
                    uint32_t anc[kAncWords];
#pragma unroll
                    for (int w = 0; w < kAncWords; ++w)
                        anc[w] = (valid && masked) ? a.anc[(long long)(n0 + i) * kAncWords + w] : 0u;
                    if (!(ok = warp_wait(&sfull[b], par, s_abort, a.wait_limit))) break;
                    tc_fence_after();
                    // every S reading K of this tile is complete (in full mode S_A
                    // was issued before S_B): release its stage
                    if (x == 1 || !full) warp_arrive(&kempty[t & 1]);
                    const uint32_t s_tm = tmem + lane_off + kTm2S + (uint32_t)b * 128;
                    float s[kBN];
                    {
                        uint32_t xa[32], xb[32], xc[32], xd[32];
                        tmem_ld32(s_tm, xa);
                        tmem_ld32(s_tm + 32, xb);
                        tmem_ld32(s_tm + 64, xc);
                        tmem_ld32(s_tm + 96, xd);
                        tmem_wait_ld();
                        tmem_regs_ready(xa);
                        tmem_regs_ready(xb);
                        tmem_regs_ready(xc);
                        tmem_regs_ready(xd);
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            s[e] = __uint_as_float(xa[e]);
                            s[32 + e] = __uint_as_float(xb[e]);
                            s[64 + e] = __uint_as_float(xc[e]);
                            s[96 + e] = __uint_as_float(xd[e]);
                        }
                    }
                    float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                    if (!masked) {  // prefix-only: nothing to mask
#pragma unroll
                        for (int j = 0; j < kBN; ++j) mx4[j & 3] = fmaxf(mx4[j & 3], s[j]);
                    } else {  // tree slots in this tile: the row's ancestor set decides
#pragma unroll
                        for (int ch = 0; ch < kBN / 32; ++ch) {
                            const uint32_t msk = tree_window(anc, key0 + ch * 32 - S);
#pragma unroll
                            for (int e = 0; e < 32; ++e) {
                                const float v = ((msk >> e) & 1u) ? s[ch * 32 + e] : -INFINITY;
                                s[ch * 32 + e] = v;
                                mx4[e & 3] = fmaxf(mx4[e & 3], v);
                            }
                        }
                    }
                    const float mt = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3])) * cexp;
                    // lazy rescale: move the reference maximum only when it grows
                    // by more than 2^8 (warp-wide O pass, factor 1 for other rows)
                    const bool grow = mt > m_used + 8.f;
                    const float corr = grow ? ex2(m_used - mt) : 1.f;  // 0 when m_used is -inf
                    if (grow) {
                        l *= corr;
                        m_used = mt;
                    }
                    const float nb = (m_used == -INFINITY) ? 0.f : -m_used;
                    float sum4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                    for (int hh = 0; hh < 2; ++hh) {
                        uint32_t xp[32];
#pragma unroll
                        for (int e = 0; e < 32; ++e) {
                            const float p0 = ex2(fmaf(s[hh * 64 + 2 * e], cexp, nb));
                            const float p1 = ex2(fmaf(s[hh * 64 + 2 * e + 1], cexp, nb));
                            sum4[e & 3] += p0 + p1;
                            xp[e] = pack_bf16x2(p0, p1);
                        }
                        tmem_st32(s_tm + hh * 32, xp);
                    }
                    l += (sum4[0] + sum4[1]) + (sum4[2] + sum4[3]);
                    // O's rescale comes after P is written, when S no longer
                    // holds registers; P V of this tile waits for pfull anyway
                    if (tl > 0 && __any_sync(0xffffffffu, grow)) {
                        // O must hold P V of the previous tile: in full mode that
                        // P V was issued before this S; in half mode after it
                        if (!full) {
                            const uint32_t pv = t - 1;
                            if (!(ok = warp_wait(&vempty[pv & 1], (pv >> 1) & 1, s_abort, a.wait_limit))) break;
                            tc_fence_after();
                        }
#pragma unroll
                        for (int ch = 0; ch < D / 32; ++ch) {
                            uint32_t xo[32];
                            const uint32_t o_tm = tmem + lane_off + (uint32_t)x * 128 + ch * 32;
                            tmem_ld32(o_tm, xo);
                            tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 32; ++e) xo[e] = __float_as_uint(__uint_as_float(xo[e]) * corr);
                            tmem_st32(o_tm, xo);
                        }
                    }
                    tmem_wait_st();
                    tc_fence_before();
                    warp_arrive(&pfull[b]);
                }
                if (ok) {
                    // epilogue: wait for P V of the last tile (its V stage's
                    // release is committed after it)
                    const uint32_t pv = g + n - 1;
                    ok = warp_wait(&vempty[pv & 1], (pv >> 1) & 1, s_abort, a.wait_limit);
                }
                if (ok) {
                    // O rows leave through shared memory (this tile's Q buffer:
                    // every S of the piece has completed), so that each store
                    // instruction writes whole 128-byte lines: a warp stages 32
                    // rows x 32 columns (row stride 36 floats, conflict-free
                    // both ways) and then writes 4 rows x 32 columns per store.
                    tc_fence_after();
                    const long long orow = (long long)(n0 + i) * a.Hq + h;
                    const long long prow = (long long)pc.slot * kPairRows + x * kBM + r;
                    const float f = pc.final ? ((l > 0.f) ? 1.f / l : 0.f) : 1.f;
                    float *dst = pc.final ? a.out + orow * D : a.part_o + prow * D;
                    const unsigned vmask = __ballot_sync(0xffffffffu, valid);
                    float *stage = reinterpret_cast<float *>(qs + (warp & 3) * 8192);
#pragma unroll 1
                    for (int ch = 0; ch < D / 32; ++ch) {
                        uint32_t xo[32];
                        tmem_ld32(tmem + lane_off + (uint32_t)x * 128 + ch * 32, xo);
                        tmem_wait_ld();
                        tmem_regs_ready(xo);
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            *reinterpret_cast<float4 *>(stage + lane * 36 + 4 * e) =
                                make_float4(__uint_as_float(xo[4 * e]) * f, __uint_as_float(xo[4 * e + 1]) * f,
                                            __uint_as_float(xo[4 * e + 2]) * f, __uint_as_float(xo[4 * e + 3]) * f);
                        __syncwarp();
#pragma unroll
                        for (int it = 0; it < 8; ++it) {
                            const int rw = it * 4 + (lane >> 3);  // row of the warp this lane writes
                            float *d = reinterpret_cast<float *>(
                                __shfl_sync(0xffffffffu, reinterpret_cast<unsigned long long>(dst), rw));
                            const float4 val = *reinterpret_cast<const float4 *>(stage + rw * 36 + (lane & 7) * 4);
                            if ((vmask >> rw) & 1u) *reinterpret_cast<float4 *>(d + ch * 32 + (lane & 7) * 4) = val;
                        }
                        __syncwarp();
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
                }
                if (!ok) break;
                if (a.q_tma) {  // this tile's Q buffer (staging included) is free for the next copy
                    fence_async_smem();
                    warp_arrive(&qfree[x]);
                }
            }
            if (full) {
                use0 += n;
                use1 += n;
            } else {
                use0 += (n + 1) >> 1;
                use1 += n >> 1;
            }
            warp_arrive(ofree);
            // the tile-B warps may not start the next piece before the tile-A
            // warps have finished this one (see the header)
            if (x == 1 && !(ok = warp_wait(ofree, (uint32_t)(piece & 1), s_abort, a.wait_limit))) break;
            g += n;
            u = pc.end;
        }
    }
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
    if (tid == 0 && *s_abort) {  // any role gave up: flag every request this CTA touches
        // the range is recomputed (after the barrier, from shared memory) so
        // that no role keeps it in registers through its loop
        const long long v0 = split.range_lo(c), v1 = split.range_lo(c + 1);
        for (long long u = v0; u < v1;) {
            const Piece pc = piece_at(info, s_pref, a.B, u, v0, v1, c);
            atomicOr(&a.status[pc.b], RS_ST_TIMEOUT);
            u = pc.end;
        }
    }
}

}  // namespace rs
