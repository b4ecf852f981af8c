// sample.cu -- rs_tree_sample: lossless verification of model-drafted nodes
// by sampling (Section 3.4, "For Drafter Module outputs": standard lossless
// speculative sampling).
//
// With deterministic (top-w) model children, speculative sampling over the
// siblings has the law of: draw y from the target row at temperature T,
// accept the model child that carries y and continue from it, otherwise emit
// y as the correction token.  Each row's draw is the inverse CDF, in
// token-id order, of a caller-supplied uniform u:  the smallest id v with
// S(v) = sum_{w <= v} exp((z_w - max z) / T) > u Z, Z = S(V - 1).
//
// The draws are exact: every one is the fp64 inverse CDF.  Most rows are
// settled by an fp32 pass that carries a rigorous error bound; the few whose
// uniform lies within that bound of a CDF step are redone in fp64.
//
// Kernel 1 (sample_partial): one CTA per (row, 8192-logit chunk), staged
// through shared memory with coalesced loads; thread t owns the 32
// consecutive ids c0 + 32 t .. c0 + 32 t + 31.  Per chunk it stores the
// maximum m_c, the mass s_c = sum_v 2^(x_v) with x_v = (z_v - m_c) log2(e)/T
// (pairwise over a thread's 32 ids, then a butterfly and a tree: depth 13)
// and q_c = sum_v 2^(x_v) |x_v|, which sizes the error from rounding x_v.
// Kernel 2 (sample_pick): one CTA per row.  Warp 0 weights the chunks by
// f_c = exp((m_c - M)/T) in fp64 (M the row maximum), forms Z and u Z in fp64
// and finds the chunk holding the crossing; the CTA recomputes that chunk's
// terms, scans the thread sums in fp64, and the holder thread's warp scans its
// 32 terms in fp64 to place the draw.  With u_32 = 2^-24 and e_x the relative
// error of ex2.approx, every computed prefix Ŝ and the computed u Ẑ are
// within E = (13 u_32 + e_x) Z + 2.8 u_32 sum_c f_c q_c of the exact values
// (13 u_32: the summation depth; 2.8 u_32 |x|: 4 roundings in x_v, times
// ln 2; f_c and everything after the chunk sums carry fp64 error only).  A
// draw whose two margins Ŝ(v) - u Ẑ and u Ẑ - Ŝ(v-1) both exceed 2 E is the
// exact draw; any other row (and any row that took a rounding fallback) is
// appended to the flagged list.
// Kernel 3 (sample_exact): the flagged rows in fp64, spread over the whole
// GPU as (row, 256-id slice) items: exp((z_v - M)/T) per id, one sum per
// slice; the CTA that completes a row's last slice (an atomic count, no
// waiting) scans the slice sums, finds the slice holding u Z and walks it with
// a block scan.  A uniform >= 1 (u Z at or past the total) takes the row's
// last id with mass.
// Kernel 4 (sample_walk): one warp per request loads its nodes and draws into
// registers, checks the tree and follows, from the root, the model child
// (source 1) carrying the current node's draw.
#include <limits.h>
#include <algorithm>
#include <math.h>
#include <stdlib.h>

#include "common.cuh"

namespace rs {
namespace {

constexpr int kSmpThreads = 256;
constexpr int kSmpWarps = kSmpThreads / 32;
constexpr int kSmpVpt = 32;                       // consecutive ids per thread
constexpr int kSmpChunk = kSmpThreads * kSmpVpt;  // 8192 ids per chunk
constexpr int kExIds = 2;                         // consecutive ids per thread in the exact pass
constexpr int kExSlice = kSmpThreads * kExIds;    // 512 ids per slice of the exact pass
constexpr float kL2E = 1.4426950408889634f;
constexpr double kU32 = 5.9604644775390625e-08;   // 2^-24, fp32 unit roundoff
// ex2.approx.f32: the PTX ISA bounds its error by 2 ulp (relative 2^-22);
// the certificate takes twice that
constexpr double kEx2Err = 4.76837158203125e-07;  // 2^-21

struct ChunkMass {
    float m;  // chunk maximum (-inf: no mass)
    float s;  // sum over the chunk of 2^x_v, x_v = (z_v - m) log2(e) / T
    float q;  // sum over the chunk of 2^x_v |x_v|
    float pad;
};
struct FlagRow {
    int row;
    float M;  // the row maximum
};
// 2^(i/64), i = 0..63, each as an fp32 (high, low) pair whose sum is within
// 2^-48 relative of the value (filled on the host from fp64)
struct Exp2Tab {
    float2 t[64];
};

// ---------------------------------------------------------------- double-float
// A value h + l held in two fp32 numbers (|l| <= ulp(h) / 2 after
// renormalisation), about 48 significant bits, on the fp32 pipe.  The error-
// free transformations are the standard ones (Knuth's TwoSum, Dekker's
// Fast2Sum, the FMA TwoProduct), written with _rn intrinsics so that the
// compiler neither contracts nor reassociates them.
struct DF {
    float h, l;
};
__device__ __forceinline__ DF two_sum(float a, float b) {
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return DF{s, e};
}
__device__ __forceinline__ DF fast_two_sum(float a, float b) {  // |a| >= |b|
    const float s = __fadd_rn(a, b);
    return DF{s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ DF two_prod(float a, float b) {
    const float p = __fmul_rn(a, b);
    return DF{p, __fmaf_rn(a, b, -p)};
}
__device__ __forceinline__ DF df_add(DF a, DF b) {
    const DF s = two_sum(a.h, b.h);
    return fast_two_sum(s.h, __fadd_rn(s.l, __fadd_rn(a.l, b.l)));
}
__device__ __forceinline__ double df_to_d(DF a) { return (double)a.h + (double)a.l; }
__device__ __forceinline__ DF df_add_f(DF a, float b) {
    const DF s = two_sum(a.h, b);
    return fast_two_sum(s.h, __fadd_rn(s.l, a.l));
}
__device__ __forceinline__ DF df_mul_f(DF a, float b) {
    const DF p = two_prod(a.h, b);
    return fast_two_sum(p.h, __fmaf_rn(a.l, b, p.l));
}
__device__ __forceinline__ DF df_mul(DF a, DF b) {
    const DF p = two_prod(a.h, b.h);
    return fast_two_sum(p.h, __fmaf_rn(a.h, b.l, __fmaf_rn(a.l, b.h, p.l)));
}
__device__ __forceinline__ DF df_neg(DF a) { return DF{-a.h, -a.l}; }
__device__ __forceinline__ bool df_gt(DF a, DF b) { return a.h > b.h || (a.h == b.h && a.l > b.l); }
__device__ __forceinline__ DF shfl_df(DF a, int src) {
    return DF{__shfl_sync(0xffffffffu, a.h, src), __shfl_sync(0xffffffffu, a.l, src)};
}
__device__ __forceinline__ DF shfl_up_df(DF a, int o) {
    return DF{__shfl_up_sync(0xffffffffu, a.h, o), __shfl_up_sync(0xffffffffu, a.l, o)};
}

constexpr double kLn2 = 0.693147180559945309417;
constexpr float kLn2H = (float)kLn2;
constexpr float kLn2L = (float)(kLn2 - (double)kLn2H);

// 2^y for y = yh + yl <= 0 (yl the low part of a double-float), by Tang's
// table-driven method: y = j + i/64 + r with |r| <= 1/128, so 2^y =
// 2^j 2^(i/64) e^s, s = r ln 2 (|s| < 0.0055), e^s from its Taylor series to
// s^5 (the next term is below 4e-17).  The linear and square terms are kept
// in double-float, the cubic tail (< 3e-8) in fp32.  Relative error about
// 2^-46; terms below 2^-125 return 0 (each < 2^-125 of the row maximum).
__device__ __forceinline__ DF exp2_df(float yh, float yl, const float2 *tab) {
    if (!(yh >= -125.f)) return DF{0.f, 0.f};
    const float k = rintf(yh * 64.f);  // yh * 64 is exact
    const int ki = (int)k;
    const int i = ki & 63, j = ki >> 6;  // k = 64 j + i, 0 <= i < 64
    const DF t = two_sum(__fsub_rn(yh, k * (1.f / 64.f)), yl);  // r + yl; the first difference is exact
    DF s = two_prod(t.h, kLn2H);
    s = fast_two_sum(s.h, __fmaf_rn(t.h, kLn2L, __fmaf_rn(t.l, kLn2H, s.l)));
    const DF s2 = two_prod(s.h, s.h);
    const float s3 = s.h * s2.h;
    const float tail = s3 * fmaf(fmaf(s.h, 1.f / 120.f, 1.f / 24.f), s.h, 1.f / 6.f);
    const DF a = fast_two_sum(s.h, 0.5f * s2.h);  // s + s^2 / 2
    const DF b = fast_two_sum(1.f, a.h);
    const float lo = b.l + (a.l + (s.l + (0.5f * s2.l + (s.h * s.l + tail))));
    const DF e = fast_two_sum(b.h, lo);  // e^s
    const float2 T = tab[i];
    DF m = two_prod(T.x, e.h);
    m = fast_two_sum(m.h, __fmaf_rn(T.x, e.l, __fmaf_rn(T.y, e.h, m.l)));
    const float sc = __int_as_float((j + 127) << 23);  // 2^j, j >= -127 here
    return DF{m.h * sc, m.l * sc};
}

// exp((z - M) / T) = 2^((z - M) lambda), lambda = log2(e) / T given as the
// double-float (lh, ll); z - M is formed exactly (TwoSum), the product in
// double-float.  z = -inf (or far below M) gives 0.
__device__ __forceinline__ DF term_df(float z, float M, float lh, float ll, const float2 *tab) {
    if (!(z > -INFINITY)) return DF{0.f, 0.f};
    const DF d = two_sum(z, -M);
    DF y = two_prod(d.h, lh);
    y = fast_two_sum(y.h, __fmaf_rn(d.h, ll, __fmaf_rn(d.l, lh, y.l)));
    return exp2_df(y.h, y.l, tab);
}

__device__ __forceinline__ float ex2f(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// This thread's 32 logits of chunk c0 (ids >= V read as -inf).
template <int kW>
__device__ __forceinline__ void load32(const float *__restrict__ row, int V, int c0, float (&z)[kSmpVpt]) {
    const int base = c0 + threadIdx.x * kSmpVpt;
    if (kW >= 4 && base + kSmpVpt <= V) {
        const float4 *p = reinterpret_cast<const float4 *>(row + base);
#pragma unroll
        for (int q = 0; q < kSmpVpt / 4; ++q) {
            const float4 x = __ldg(p + q);
            z[4 * q] = x.x;
            z[4 * q + 1] = x.y;
            z[4 * q + 2] = x.z;
            z[4 * q + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int j = 0; j < kSmpVpt; ++j) z[j] = base + j < V ? __ldg(row + base + j) : -INFINITY;
    }
}

// The same 32 logits, read through shared memory: the CTA streams the chunk
// with coalesced 128-bit loads into a buffer padded by four floats after
// every 32 (so that neither the stores nor the per-thread 128-bit reads of 32
// consecutive ids meet bank conflicts), then each thread takes its own ids.
// Chunks that end past V fall back to load32.  The values are the same either
// way, so the per-thread sums do not depend on the path.
constexpr int kSmpPadded = kSmpChunk + kSmpChunk / 8;  // 36 floats per thread

// kW: logits per streaming load (8: V % 8 == 0 and 32-byte aligned logits;
// 4: V % 4 == 0 and 16-byte alignment; 1: no staging).
template <int kW>
__device__ __forceinline__ void load32_staged(const float *__restrict__ row, int V, int c0, float *s_buf,
                                              float (&z)[kSmpVpt]) {
    if (kW >= 4 && c0 + kSmpChunk <= V) {  // uniform over the CTA
        const int tid = threadIdx.x;
        if (kW == 8) {
#pragma unroll
            for (int j = 0; j < kSmpVpt / 8; ++j) {
                const int e = 8 * (j * kSmpThreads + tid);  // 8 ids in one padded 32-group
                float x[8];
                ldg_stream8(row + c0 + e, x);
                float4 *d = reinterpret_cast<float4 *>(s_buf + e + 4 * (e >> 5));
                d[0] = make_float4(x[0], x[1], x[2], x[3]);
                d[1] = make_float4(x[4], x[5], x[6], x[7]);
            }
        } else {
#pragma unroll
            for (int j = 0; j < kSmpVpt / 4; ++j) {
                const int e = 4 * (j * kSmpThreads + tid);
                const float4 x = ldg_stream4(reinterpret_cast<const float4 *>(row + c0 + e));
                *reinterpret_cast<float4 *>(s_buf + e + 4 * (e >> 5)) = x;
            }
        }
        __syncthreads();
        const float4 *p = reinterpret_cast<const float4 *>(s_buf + tid * (kSmpVpt + 4));
#pragma unroll
        for (int q = 0; q < kSmpVpt / 4; ++q) {
            const float4 x = p[q];
            z[4 * q] = x.x;
            z[4 * q + 1] = x.y;
            z[4 * q + 2] = x.z;
            z[4 * q + 3] = x.w;
        }
    } else {
        load32<kW>(row, V, c0, z);
    }
}

__device__ __forceinline__ float block_max(float v, float *s_w) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_max(v);
    if (lane == 0) s_w[warp] = v;
    __syncthreads();
    float r = s_w[0];
#pragma unroll
    for (int w = 1; w < kSmpWarps; ++w) r = fmaxf(r, s_w[w]);
    __syncthreads();
    return r;
}

// One thread's 32 terms 2^x_v, x_v = (z_v - m) scale: their sum, pairwise
// in id order (depth 5), and sum 2^x_v |x_v| (for the error bound).  The
// same code in both kernels, so a chunk's terms are the same in both.
__device__ __forceinline__ float term(float z, float m, float scale) { return ex2f((z - m) * scale); }

__device__ __forceinline__ void thread_terms(const float (&z)[kSmpVpt], float m, float scale, float &s, float &q) {
    float e[kSmpVpt];
    q = 0.f;
#pragma unroll
    for (int j = 0; j < kSmpVpt; ++j) {
        const float x = (z[j] - m) * scale;
        e[j] = ex2f(x);
        q = fmaf(e[j], fminf(-x, 3.0e38f), q);  // x <= 0; z = -inf gives e = 0 (and a finite factor)
    }
#pragma unroll
    for (int w = 1; w < kSmpVpt; w <<= 1)
#pragma unroll
        for (int j = 0; j < kSmpVpt; j += 2 * w) e[j] += e[j + w];
    s = e[0];
}

__device__ __forceinline__ double warp_incl_scan_d(double v) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, v, o);
        if (lane >= o) v += y;
    }
    return v;
}

// Exclusive prefix of one double per thread in thread order, and the total
// (the same on every thread).  Ends with a barrier, so s_wd may be reused.
__device__ __forceinline__ double block_excl_scan_d(double v, double *s_wd, double *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const double x = warp_incl_scan_d(v);
    double xe = __shfl_up_sync(0xffffffffu, x, 1);
    if (lane == 0) xe = 0.0;
    if (lane == 31) s_wd[warp] = x;
    __syncthreads();
    double before = 0.0, sum = 0.0;
#pragma unroll
    for (int w = 0; w < kSmpWarps; ++w) {
        const double y = s_wd[w];
        if (w < warp) before += y;
        sum += y;
    }
    __syncthreads();
    *total = sum;
    return before + xe;
}

// Lowest thread of the CTA whose predicate holds, INT_MAX if none (all
// threads).  Ends with a barrier.
__device__ __forceinline__ int block_first(bool pred, int *s_i) {
    if (threadIdx.x == 0) *s_i = INT_MAX;
    __syncthreads();
    const unsigned b = __ballot_sync(0xffffffffu, pred);
    if ((threadIdx.x & 31) == 0 && b) atomicMin(s_i, (threadIdx.x & ~31) + __ffs(b) - 1);
    __syncthreads();
    const int r = *s_i;
    __syncthreads();
    return r;
}

// The decision the row's leader CTA takes from the chunk masses.
struct RowDecision {
    int chunk;   // the chunk holding the crossing; -1: no mass; -2: none found
    float M;     // the row maximum
    float mc;    // the chosen chunk's maximum
    float tol;   // the certificate's margin, in the chunk's units
    DF tl;       // u Z - (mass before the chunk), in the chunk's units
};

// The leader's warp 0: chunk weights f_c = exp((m_c - M) / T), Z and the
// chunk prefix in double-float, sum_c f_c q_c (only the bound uses it) in
// fp32, and the chunk holding u Z.  One pass when the row has at most 32
// chunks (the inclusive scan's last lane is Z), two otherwise.
__device__ __forceinline__ RowDecision decide_row(const ChunkMass *pr, int nchunks, float ur, float lam_h,
                                                  float lam_l, const float2 *tab) {
    const int lane = threadIdx.x & 31;
    float M = -INFINITY;
    for (int c = lane; c < nchunks; c += 32) M = fmaxf(M, pr[c].m);
    M = warp_max(M);
    DF Z{0.f, 0.f}, target, pb{0.f, 0.f}, inv_f{1.f, 0.f};
    float A = 0.f, mc = 0.f;
    int pick = -1;
    if (nchunks <= 32) {
        const ChunkMass cm = lane < nchunks ? pr[lane] : ChunkMass{-INFINITY, 0.f, 0.f, 0.f};
        const DF f = term_df(cm.m, M, lam_h, lam_l, tab);
        // 1 / f_c, below 2^125 wherever f_c > 0 (the only chunks that can be picked)
        const DF fi = cm.m > -INFINITY ? term_df(M, cm.m, lam_h, lam_l, tab) : DF{0.f, 0.f};
        const DF w = df_mul_f(f, cm.s);
        A = warp_sum(f.h * cm.q);
        DF x = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const DF y = shfl_up_df(x, o);
            if (lane >= o) x = df_add(x, y);
        }
        Z = shfl_df(x, 31);
        target = df_mul_f(Z, ur);
        const unsigned cross = __ballot_sync(0xffffffffu, w.h > 0.f && df_gt(x, target));
        if (cross) {
            const int l = __ffs(cross) - 1;
            pick = l;
            DF xe = shfl_up_df(x, 1);
            if (lane == 0) xe = DF{0.f, 0.f};
            pb = shfl_df(xe, l);
            inv_f = shfl_df(fi, l);
            mc = __shfl_sync(0xffffffffu, cm.m, l);
        }
    } else {
        for (int c0 = 0; c0 < nchunks; c0 += 32) {
            const int c = c0 + lane;
            const ChunkMass cm = c < nchunks ? pr[c] : ChunkMass{-INFINITY, 0.f, 0.f, 0.f};
            const DF f = term_df(cm.m, M, lam_h, lam_l, tab);
            DF w = df_mul_f(f, cm.s);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) w = df_add(w, shfl_df(w, lane ^ o));
            Z = df_add(Z, w);
            A += warp_sum(f.h * cm.q);
        }
        target = df_mul_f(Z, ur);
        DF carry{0.f, 0.f};
        for (int c0 = 0; c0 < nchunks && pick < 0; c0 += 32) {
            const int c = c0 + lane;
            const ChunkMass cm = c < nchunks ? pr[c] : ChunkMass{-INFINITY, 0.f, 0.f, 0.f};
            const DF f = term_df(cm.m, M, lam_h, lam_l, tab);
            const DF w = df_mul_f(f, cm.s);
            DF x = w;  // inclusive prefix within the round
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const DF y = shfl_up_df(x, o);
                if (lane >= o) x = df_add(x, y);
            }
            DF xe = shfl_up_df(x, 1);
            if (lane == 0) xe = DF{0.f, 0.f};
            const unsigned cross = __ballot_sync(0xffffffffu, w.h > 0.f && df_gt(df_add(carry, x), target));
            if (cross) {
                const int l = __ffs(cross) - 1;
                pick = c0 + l;
                pb = df_add(carry, shfl_df(xe, l));
                mc = __shfl_sync(0xffffffffu, cm.m, l);
                inv_f = term_df(M, mc, lam_h, lam_l, tab);
            }
            carry = df_add(carry, shfl_df(x, 31));
        }
    }
    RowDecision d;
    d.M = M;
    d.mc = mc;
    d.tol = 0.f;
    d.tl = DF{0.f, 0.f};
    if (M == -INFINITY) {
        d.chunk = -1;
    } else if (pick < 0 || !(ur < 1.f)) {
        d.chunk = -2;  // u Z at or past the total: left to the exact pass
    } else {
        const float E = (float)(13.0 * kU32 + kEx2Err) * Z.h + (float)(2.8 * kU32) * A;
        d.chunk = pick;
        d.tl = df_mul(df_add(target, df_neg(pb)), inv_f);
        d.tol = (2.02f * E + 1e-12f * Z.h) * inv_f.h;
    }
    return d;
}

// Kernel 1: one CTA per (row, 8192-logit chunk): the chunk's maximum m_c,
// mass s_c and q_c (staged loads, terms, butterfly then tree sums).
template <int kW>
__global__ void __launch_bounds__(kSmpThreads)
sample_partial(const float *__restrict__ logits, int V, int nchunks, float scale, ChunkMass *__restrict__ part,
               int *__restrict__ n_flag) {
    pdl_enter();
    if (blockIdx.x == 0 && threadIdx.x == 0) *n_flag = 0;  // the flagged list of this call (filled by kernel 2)
    __shared__ float s_w[kSmpWarps];
    __shared__ float2 s_w2[kSmpWarps];
    __shared__ __align__(16) float s_buf[kSmpPadded];
    const int r = blockIdx.x / nchunks, c = blockIdx.x - r * nchunks;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float *row = logits + (long long)r * V;
    float z[kSmpVpt];
    load32_staged<kW>(row, V, c * kSmpChunk, s_buf, z);
    float mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < kSmpVpt; ++j) mx = fmaxf(mx, z[j]);
    const float m = block_max(mx, s_w);
    float s = 0.f, q = 0.f;
    if (m != -INFINITY) thread_terms(z, m, scale, s, q);
    s = warp_sum(s);
    q = warp_sum(q);
    if (lane == 0) s_w2[warp] = make_float2(s, q);
    __syncthreads();
    if (tid == 0) {
        float2 t[kSmpWarps];
#pragma unroll
        for (int w = 0; w < kSmpWarps; ++w) t[w] = s_w2[w];
        static_assert(kSmpWarps == 8, "the tree below sums 8 warps");
        const float S = ((t[0].x + t[1].x) + (t[2].x + t[3].x)) + ((t[4].x + t[5].x) + (t[6].x + t[7].x));
        const float Q = ((t[0].y + t[1].y) + (t[2].y + t[3].y)) + ((t[4].y + t[5].y) + (t[6].y + t[7].y));
        part[blockIdx.x] = ChunkMass{m, S, Q, 0.f};
    }
}

// Kernel 2: one CTA per row.  Warp 0 decides the chunk holding u Z from the
// chunk masses; the CTA re-reads that chunk, scans it and places and
// certifies the draw.  A row whose draw is not certified is appended to the
// flagged list (row, maximum) for the exact pass.
template <int kW>
__global__ void __launch_bounds__(kSmpThreads)
sample_pick(const float *__restrict__ logits, int V, int nchunks, float scale, float lam_h, float lam_l,
            const Exp2Tab tab, const ChunkMass *__restrict__ part, const float *__restrict__ uniforms, int force,
            int *__restrict__ n_flag, FlagRow *__restrict__ flags, int *__restrict__ done,
            int32_t *__restrict__ draw) {
    pdl_enter();
    __shared__ float2 s_tab[64];
    __shared__ RowDecision s_dec;
    __shared__ float s_wt[kSmpWarps];
    __shared__ DF s_wo[kSmpWarps];
    __shared__ int s_i, s_draw, s_ok;
    __shared__ __align__(16) float s_buf[kSmpPadded];
    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float *row = logits + (long long)r * V;
    if (tid < 64) s_tab[tid] = tab.t[tid];
    __syncthreads();
    if (warp == 0) {
        const RowDecision d = decide_row(part + (long long)r * nchunks, nchunks, uniforms[r], lam_h, lam_l, s_tab);
        if (lane == 0) s_dec = d;
    }
    __syncthreads();
    const RowDecision d = s_dec;
    if (d.chunk < 0) {
        if (tid == 0) {  // no mass: the first id; none found: the exact pass
            draw[r] = 0;
            if (d.chunk == -2) {
                done[r] = 0;
                flags[atomicAdd(n_flag, 1)] = FlagRow{r, d.M};
            }
        }
        return;
    }
    const int c = d.chunk;
    const bool staged = kW >= 4 && c * kSmpChunk + kSmpChunk <= V;
    float z[kSmpVpt];
    load32_staged<kW>(row, V, c * kSmpChunk, s_buf, z);
    const float m = d.mc;
    float s, q;
    thread_terms(z, m, scale, s, q);
    // exclusive prefix of the thread sums: fp32 within the warp (depth 5),
    // the warp offsets in double-float
    float xs = s;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, xs, o);
        if (lane >= o) xs += y;
    }
    float xe = __shfl_up_sync(0xffffffffu, xs, 1);
    if (lane == 0) xe = 0.f;
    if (lane == 31) s_wt[warp] = xs;
    if (tid == 0) {
        s_draw = 0;
        s_ok = 0;
    }
    __syncthreads();
    if (warp == 0) {
        DF y{lane < kSmpWarps ? s_wt[lane] : 0.f, 0.f};
#pragma unroll
        for (int o = 1; o < kSmpWarps; o <<= 1) {
            const DF t = shfl_up_df(y, o);
            if (lane >= o) y = df_add(y, t);
        }
        DF ye = shfl_up_df(y, 1);
        if (lane == 0) ye = DF{0.f, 0.f};
        if (lane < kSmpWarps) s_wo[lane] = ye;
    }
    __syncthreads();
    const DF ex = df_add_f(s_wo[warp], xe);
    const int h = block_first(s > 0.f && df_gt(df_add_f(ex, s), d.tl), &s_i);
    if (h != INT_MAX && warp == (h >> 5)) {
        // the holder's 32 ids, one per lane (from the staged chunk, or the
        // row), scanned in fp32 (depth 5); the draw's two margins in
        // double-float
        const DF ntl = df_neg(d.tl);
        const DF exh = shfl_df(ex, h & 31);
        const int base = c * kSmpChunk + h * kSmpVpt;
        const float zl = staged ? s_buf[h * (kSmpVpt + 4) + lane] : base + lane < V ? row[base + lane] : -INFINITY;
        float loc = term(zl, m, scale);
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const float y = __shfl_up_sync(0xffffffffu, loc, o);
            if (lane >= o) loc += y;
        }
        float pre = __shfl_up_sync(0xffffffffu, loc, 1);
        if (lane == 0) pre = 0.f;
        const DF hi = df_add(df_add_f(exh, loc), ntl);
        const DF lo = df_add(d.tl, df_neg(df_add_f(exh, pre)));
        const unsigned hit = __ballot_sync(0xffffffffu, hi.h > 0.f || (hi.h == 0.f && hi.l > 0.f));
        if (hit) {
            const int v = __ffs(hit) - 1;
            const bool ok = __shfl_sync(0xffffffffu, hi.h > d.tol && lo.h > d.tol, v);
            if (lane == 0) {
                s_draw = base + v;
                s_ok = ok;
            }
        }
    }
    __syncthreads();
    if (tid == 0) {
        draw[r] = s_draw;
        if (!s_ok || force) {  // not certified: the exact pass rewrites this draw
            done[r] = 0;
            flags[atomicAdd(n_flag, 1)] = FlagRow{r, d.M};
        }
    }
}

// Block maximum of one int, on every thread.
__device__ __forceinline__ int block_max_i(int v, int *s_wi) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    if (lane == 0) s_wi[warp] = v;
    __syncthreads();
    int r = s_wi[0];
#pragma unroll
    for (int w = 1; w < kSmpWarps; ++w) r = max(r, s_wi[w]);
    __syncthreads();
    return r;
}

// Sums of non-negative double-floats: warp scan (depth 5), then the warp
// totals scanned by warp 0; the exclusive prefix of each thread and the
// block total (every thread).  Ends with a barrier.
__device__ __forceinline__ DF block_excl_scan_df(DF v, DF *s_w, DF *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    DF x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const DF y = shfl_up_df(x, o);
        if (lane >= o) x = df_add(x, y);
    }
    DF xe = shfl_up_df(x, 1);
    if (lane == 0) xe = DF{0.f, 0.f};
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const DF t = lane < kSmpWarps ? s_w[lane] : DF{0.f, 0.f};
        DF y = t;
#pragma unroll
        for (int o = 1; o < kSmpWarps; o <<= 1) {
            const DF z = shfl_up_df(y, o);
            if (lane >= o) y = df_add(y, z);
        }
        DF ye = shfl_up_df(y, 1);
        if (lane == 0) ye = DF{0.f, 0.f};
        const DF tot = shfl_df(y, kSmpWarps - 1);
        if (lane < kSmpWarps) s_w[lane] = ye;
        if (lane == 0) s_w[kSmpWarps] = tot;
    }
    __syncthreads();
    const DF r = df_add(s_w[warp], xe);
    *total = s_w[kSmpWarps];
    __syncthreads();
    return r;
}

// The terms of ids v0 .. v0 + kExIds - 1 (0 past V) and their double-float
// sum in id order.
__device__ __forceinline__ DF thread_terms_df(const float *row, int V, long long v0, float M, float lh, float ll,
                                              const float2 *tab, DF (&t)[kExIds]) {
    DF acc{0.f, 0.f};
#pragma unroll
    for (int j = 0; j < kExIds; ++j) {
        t[j] = v0 + j < V ? term_df(row[v0 + j], M, lh, ll, tab) : DF{0.f, 0.f};
        acc = df_add(acc, t[j]);
    }
    return acc;
}

// Whether exp((z - M) / T) is above zero in fp64, as the fp64 definition
// decides it: certain above -745.0, certainly zero below -745.5 (the fp64
// underflow threshold is near -745.13), exp() itself in between.
__device__ __forceinline__ bool has_mass(float z, float M, double inv_t, double T) {
    if (!(z > -INFINITY)) return false;
    const double x = ((double)z - (double)M) * inv_t;
    if (x > -745.0) return true;
    if (x < -745.5) return false;
    return exp(((double)z - (double)M) / T) > 0.0;
}

// The last id < end with mass (-1 if none), searched backwards a block of
// ids at a time.
__device__ int last_with_mass(const float *row, long long end, float M, double inv_t, double T, int *s_wi) {
    for (long long w0 = end - kSmpThreads;; w0 -= kSmpThreads) {
        const long long v = w0 + threadIdx.x;
        const int best = block_max_i(v >= 0 && has_mass(row[v], M, inv_t, T) ? (int)v : -1, s_wi);
        if (best >= 0 || w0 <= 0) return best;
    }
}

// The flagged rows exactly.  The work is (flagged row, group of G
// consecutive 512-id slices) items, G chosen so that the items about fill the
// grid; a CTA writes each slice's sum, and the CTA that completes a row's last
// slice (an atomic count of slices, no waiting) finishes the row.  Terms,
// sums and scans in double-float on the fp32 pipe; fp64 only on the rare
// paths (u Z below 2^-40 Z, the last id with mass).
__global__ void __launch_bounds__(kSmpThreads)
sample_exact(const float *__restrict__ logits, int V, int nslices, float lam_h, float lam_l, double inv_t, double T,
             const Exp2Tab tab, const float *__restrict__ uniforms, const int *__restrict__ n_flag,
             const FlagRow *__restrict__ flags, int *__restrict__ done, float2 *__restrict__ slice_sum,
             int32_t *__restrict__ draw) {
    pdl_enter();
    __shared__ float2 s_tab[64];
    __shared__ DF s_w[kSmpWarps + 1];
    __shared__ double s_wd[kSmpWarps];
    __shared__ int s_wi[kSmpWarps];
    __shared__ int s_i, s_fin;
    __shared__ DF s_pk;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n = *n_flag;
    const long long want = (long long)n * nslices;
    const int G = (int)max(1ll, (want + gridDim.x - 1) / gridDim.x);  // slices per item
    const int ng = (nslices + G - 1) / G;                              // items per row
    const long long items = (long long)n * ng;
    if (blockIdx.x >= items) return;  // uniform over the CTA
    if (tid < 64) s_tab[tid] = tab.t[tid];
    __syncthreads();
    {
        for (long long it = blockIdx.x; it < items; it += gridDim.x) {
            const int f = (int)(it / ng);
            const int g = (int)(it - (long long)f * ng);
            const FlagRow fr = flags[f];
            const int fr_row = fr.row;
            const float fr_M = fr.M;
            const float *row = logits + (long long)fr_row * V;
            float2 *ss = slice_sum + (long long)fr_row * nslices;
            DF t[kExIds];
            const int k0s = g * G, k1s = min(nslices, k0s + G);
            for (int k = k0s; k < k1s; ++k) {  // each slice's sum: butterfly within the warp, the warps in order
                DF acc = thread_terms_df(row, V, (long long)k * kExSlice + tid * kExIds, fr_M, lam_h, lam_l, s_tab, t);
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) acc = df_add(acc, shfl_df(acc, lane ^ o));
                if (lane == 0) s_w[warp] = acc;
                __syncthreads();
                if (tid == 0) {
                    DF S = s_w[0];
#pragma unroll
                    for (int w = 1; w < kSmpWarps; ++w) S = df_add(S, s_w[w]);
                    ss[k] = make_float2(S.h, S.l);
                }
                __syncthreads();
            }
            if (tid == 0) {
                __threadfence();
                s_fin = atomicAdd(done + fr_row, k1s - k0s) + (k1s - k0s) == nslices;
            }
            __syncthreads();
            if (!s_fin) continue;  // uniform over the CTA
            // this CTA completed the row: every slice's sum is visible
            __threadfence();
            // Z: the slice sums in slice order, 256 at a time; the first round's
            // prefixes are kept (with at most 256 slices the crossing needs no
            // second scan)
            DF Z{0.f, 0.f}, tot, ex0{0.f, 0.f}, sig0{0.f, 0.f}, tot0{0.f, 0.f};
            for (int k0 = 0; k0 < nslices; k0 += kSmpThreads) {
                const int kk = k0 + tid;
                const float2 v = kk < nslices ? __ldcg(ss + kk) : make_float2(0.f, 0.f);
                const DF sig{v.x, v.y};
                const DF ex = block_excl_scan_df(sig, s_w, &tot);
                if (k0 == 0) {
                    ex0 = ex;
                    sig0 = sig;
                    tot0 = tot;
                }
                Z = df_add(Z, tot);
            }
            const float ur = uniforms[fr_row];
            const DF target = df_mul_f(Z, ur);
            if (ur < 1.f && target.h < 0x1p-40f * Z.h) {
                // u Z below 2^-40 Z (u = 0 included): the crossing lies among
                // terms the double-float form drops (below 2^-125), so walk from
                // id 0 with the fp64 terms themselves; windows without mass add
                // nothing and are skipped
                const double tg = (double)ur * df_to_d(Z);
                double c = 0.0, dtot;
                int d = -1;
                for (long long w0 = 0; w0 < V && d < 0; w0 += kSmpThreads) {
                    const long long v = w0 + tid;
                    const bool mz = v < V && has_mass(row[v], fr_M, inv_t, T);
                    if (!__syncthreads_or(mz)) continue;  // uniform over the CTA
                    const double e = mz ? exp(((double)row[v] - (double)fr_M) / T) : 0.0;
                    const double ex = block_excl_scan_d(e, s_wd, &dtot);
                    const int tt = block_first(v < V && c + (ex + e) > tg, &s_i);
                    if (tt != INT_MAX) d = (int)(w0 + tt);
                    c += dtot;
                }
                if (d < 0) d = max(last_with_mass(row, V, fr_M, inv_t, T, s_wi), 0);
                if (tid == 0) draw[fr_row] = d;
                __syncthreads();
                continue;
            }
            int ks = -1;
            DF pk{0.f, 0.f}, carry{0.f, 0.f};
            // u >= 1 (no prefix passes u Z): straight to the last id with mass
            for (int k0 = 0; k0 < nslices && ks < 0 && ur < 1.f; k0 += kSmpThreads) {  // the slice holding u Z
                const int kk = k0 + tid;
                DF sig = sig0, ex = ex0;
                tot = tot0;
                if (k0 > 0) {
                    const float2 v = kk < nslices ? __ldcg(ss + kk) : make_float2(0.f, 0.f);
                    sig = DF{v.x, v.y};
                    ex = df_add(carry, block_excl_scan_df(sig, s_w, &tot));
                }
                const int tt = block_first(kk < nslices && df_gt(df_add(ex, sig), target), &s_i);
                if (tt != INT_MAX) {
                    ks = k0 + tt;
                    if (tid == tt) s_pk = ex;
                    __syncthreads();
                    pk = s_pk;
                    __syncthreads();
                }
                carry = df_add(carry, tot);
            }
            int d = -1;
            long long end = V;  // where the fallback search for the last id with mass starts
            if (ks >= 0) {  // walk the slice: thread sums scanned, then the holder's ids in order
                const long long v0 = (long long)ks * kExSlice + tid * kExIds;
                const DF ts = thread_terms_df(row, V, v0, fr_M, lam_h, lam_l, s_tab, t);
                const DF ex = df_add(pk, block_excl_scan_df(ts, s_w, &tot));
                const int h = block_first(v0 < V && df_gt(df_add(ex, ts), target), &s_i);
                if (h != INT_MAX) {
                    if (tid == h) {
                        DF cum = ex;
                        int v = -1;
#pragma unroll
                        for (int j = 0; j < kExIds; ++j) {
                            cum = df_add(cum, t[j]);
                            if (v < 0 && df_gt(cum, target)) v = j;
                        }
                        s_i = v < 0 ? -1 : (int)(v0 + v);
                    }
                    __syncthreads();
                    d = s_i;
                    __syncthreads();
                }
                end = min((long long)V, (long long)(ks + 1) * kExSlice);
            }
            if (d < 0) d = max(last_with_mass(row, end, fr_M, inv_t, T, s_wi), 0);
            if (tid == 0) draw[fr_row] = d;
            __syncthreads();
        }
    }
}

// One warp per request: the tree check and the walk along model children.
__global__ void __launch_bounds__(32)
sample_walk(const int32_t *__restrict__ node_off, int R, const int32_t *__restrict__ tokens,
            const int32_t *__restrict__ parents, const uint8_t *__restrict__ source,
            const int32_t *__restrict__ draw, int acc_cap, int32_t *__restrict__ acc_len,
            int32_t *__restrict__ acc_nodes, int32_t *__restrict__ bonus, int32_t *__restrict__ status) {
    pdl_enter();
    constexpr int kPer = RS_MAX_NODES / 32;
    const int b = blockIdx.x, lane = threadIdx.x;
    const int n0 = node_off[b];
    const int N = node_off[b + 1] - n0;
    int32_t *an = acc_nodes + (long long)b * acc_cap;
    for (int j = lane; j < acc_cap; j += 32) an[j] = -1;
    int st = 0;
    if (n0 < 0 || N < 0 || (long long)n0 + N > R) st = RS_ST_BAD_OFFSET;  // rows outside [0, R): not read
    else if (N > RS_MAX_NODES) st = RS_ST_TOO_LARGE;
    else if (N < 1) st = RS_ST_BAD_TREE;
    // node i = lane + 32 q lives in register slot q
    int par[kPer], tok[kPer], drw[kPer];
    bool model[kPer];
    bool bad = false;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
        const int i = lane + 32 * q;
        par[q] = -2;
        tok[q] = -1;
        drw[q] = 0;
        model[q] = false;
        if (st == 0 && i < N) {
            const int pa = parents[n0 + i], sr = source[n0 + i];
            par[q] = pa;
            tok[q] = tokens[n0 + i];
            drw[q] = draw[n0 + i];
            model[q] = sr == 1;
            if (i == 0) bad |= pa != -1 || sr != 0;
            else bad |= pa < 0 || pa >= i || sr < 1 || sr > 2;
        }
    }
    if (st == 0 && __any_sync(0xffffffffu, bad)) st = RS_ST_BAD_TREE;
    if (st != 0) {
        if (lane == 0) {
            acc_len[b] = 0;
            bonus[b] = -1;
            status[b] = st;
        }
        return;
    }
    int cur = 0, len = 0;
    for (;;) {
        int y = 0;  // the current node's draw, from the register copies
#pragma unroll
        for (int q = 0; q < kPer; ++q) {
            const int yq = __shfl_sync(0xffffffffu, drw[q], cur & 31);
            if ((cur >> 5) == q) y = yq;
        }
        int next = -1;
#pragma unroll
        for (int q = 0; q < kPer; ++q) {  // lowest index among the model children carrying y
            const unsigned hit = __ballot_sync(0xffffffffu, model[q] && par[q] == cur && tok[q] == y);
            if (next < 0 && hit) next = 32 * q + __ffs(hit) - 1;
        }
        if (next < 0) {
            if (lane == 0) bonus[b] = y;
            break;
        }
        if (lane == 0 && len < acc_cap) an[len] = next;
        ++len;
        cur = next;
    }
    if (lane == 0) {
        acc_len[b] = len;
        status[b] = len > acc_cap ? RS_ST_TRUNCATED : 0;
    }
}

}  // namespace
}  // namespace rs

using namespace rs;

namespace {
// Workspace layout: chunk masses, the flagged-row count and list, the per-row
// completion counts and the slice sums of the exact pass.
struct SampleWs {
    size_t part, n_flag, flags, done, sums, total;
};
SampleWs sample_ws(int R, int V) {
    const size_t nchunks = (size_t)(V + kSmpChunk - 1) / kSmpChunk;
    const size_t nslices = (size_t)(V + kExSlice - 1) / kExSlice;
    SampleWs w;
    size_t off = 0;
    w.part = off;
    off = align_up(off + (size_t)R * nchunks * sizeof(ChunkMass), 256);
    w.n_flag = off;
    off = align_up(off + sizeof(int), 256);
    w.flags = off;
    off = align_up(off + (size_t)R * sizeof(FlagRow), 256);
    w.done = off;
    off = align_up(off + (size_t)R * sizeof(int), 256);
    w.sums = off;
    off = align_up(off + (size_t)R * nslices * sizeof(float2), 256);
    w.total = off;
    return w;
}

// 2^(i/64) split into fp32 (high, low) pairs, from fp64 exp2.
const Exp2Tab &exp2_table() {
    static const Exp2Tab tab = [] {
        Exp2Tab t;
        for (int i = 0; i < 64; ++i) {
            const double v = exp2(i / 64.0);
            const float h = (float)v;
            t.t[i] = make_float2(h, (float)(v - (double)h));
        }
        return t;
    }();
    return tab;
}
}  // namespace

extern "C" size_t rs_tree_sample_workspace_size(int R, int V) {
    if (R < 1 || V < 1) return 0;
    return sample_ws(R, V).total;
}

extern "C" rs_status rs_tree_sample(const float *logits, int R, int V, const int32_t *node_off, int B,
                                    const int32_t *tokens, const int32_t *parents, const uint8_t *source,
                                    float temperature, const float *uniforms, int acc_cap, int32_t *draw,
                                    int32_t *acc_len, int32_t *acc_nodes, int32_t *bonus, int32_t *status,
                                    void *workspace, size_t workspace_bytes, void *stream) {
    clear_error();
    RS_CHECK_ARG(R >= 0 && B >= 0, "rs_tree_sample: negative size (R=%d, B=%d)", R, B);
    RS_CHECK_ARG(V >= 1, "rs_tree_sample: V must be >= 1 (got %d)", V);
    RS_CHECK_ARG(isfinite(temperature) && temperature > 0.f, "rs_tree_sample: temperature must be finite and > 0");
    RS_CHECK_ARG(acc_cap >= 1, "rs_tree_sample: acc_cap must be >= 1");
    RS_CHECK_ARG(R == 0 || (logits && uniforms && draw), "rs_tree_sample: null row pointer");
    RS_CHECK_ARG(B == 0 || (node_off && tokens && parents && source && acc_len && acc_nodes && bonus && status),
                 "rs_tree_sample: null request pointer");
    const int nchunks = (V + kSmpChunk - 1) / kSmpChunk;
    const int nslices = (V + kExSlice - 1) / kExSlice;
    RS_CHECK_ARG((long long)R * nslices < (1ll << 31), "rs_tree_sample: R*V too large");
    const size_t need = rs_tree_sample_workspace_size(R, V);
    if (workspace_bytes < need || (need && !workspace)) {
        set_error("rs_tree_sample: workspace %zu bytes < %zu required", workspace_bytes, need);
        return RS_ERR_CAPACITY;
    }
    cudaStream_t st = (cudaStream_t)stream;
    const float scale = kL2E / temperature;
    const double T = (double)temperature, inv_t = 1.0 / T;
    const double lam = 1.4426950408889634074 / T;  // log2(e) / T as a double-float
    const float lam_h = (float)lam, lam_l = (float)(lam - (double)lam_h);
    const Exp2Tab &tab = exp2_table();
    // a test hook: RS_DEBUG_SAMPLE_EXACT=1 sends every row with mass through
    // the exact pass
    int force = 0;
    if (const char *e = getenv("RS_DEBUG_SAMPLE_EXACT")) force = atoi(e) != 0;
    if (R > 0) {
        const SampleWs L = sample_ws(R, V);
        char *ws = static_cast<char *>(workspace);
        ChunkMass *part = reinterpret_cast<ChunkMass *>(ws + L.part);
        int *n_flag = reinterpret_cast<int *>(ws + L.n_flag);
        FlagRow *flags = reinterpret_cast<FlagRow *>(ws + L.flags);
        int *done = reinterpret_cast<int *>(ws + L.done);
        float2 *sums = reinterpret_cast<float2 *>(ws + L.sums);
        const int w = (V % 8 == 0 && ((uintptr_t)logits & 31) == 0) ? 8
                      : (V % 4 == 0 && ((uintptr_t)logits & 15) == 0) ? 4 : 1;
        const unsigned blocks = (unsigned)((long long)R * nchunks);
        const dim3 blk(kSmpThreads);
        if (w == 8) launch_pdl(sample_partial<8>, dim3(blocks), blk, 0, st, logits, V, nchunks, scale, part, n_flag);
        else if (w == 4) launch_pdl(sample_partial<4>, dim3(blocks), blk, 0, st, logits, V, nchunks, scale, part, n_flag);
        else launch_pdl(sample_partial<1>, dim3(blocks), blk, 0, st, logits, V, nchunks, scale, part, n_flag);
        RS_CHECK_LAUNCH("rs_tree_sample/partial");
        if (w == 8)
            launch_pdl(sample_pick<8>, dim3(R), blk, 0, st, logits, V, nchunks, scale, lam_h, lam_l, tab, part,
                       uniforms, force, n_flag, flags, done, draw);
        else if (w == 4)
            launch_pdl(sample_pick<4>, dim3(R), blk, 0, st, logits, V, nchunks, scale, lam_h, lam_l, tab, part,
                       uniforms, force, n_flag, flags, done, draw);
        else
            launch_pdl(sample_pick<1>, dim3(R), blk, 0, st, logits, V, nchunks, scale, lam_h, lam_l, tab, part,
                       uniforms, force, n_flag, flags, done, draw);
        RS_CHECK_LAUNCH("rs_tree_sample/pick");
        const long long items = (long long)R * nslices;
        const unsigned egrid = (unsigned)std::min<long long>(items, 2ll * num_sms());
        launch_pdl(sample_exact, dim3(egrid), blk, 0, st, logits, V, nslices, lam_h, lam_l, inv_t, T, tab, uniforms,
                   n_flag, flags, done, sums, draw);
        RS_CHECK_LAUNCH("rs_tree_sample/exact");
    }
    if (B > 0) {
        launch_pdl(sample_walk, dim3(B), dim3(32), 0, st, node_off, R, tokens, parents, source, draw, acc_cap, acc_len,
            acc_nodes, bonus, status);
        RS_CHECK_LAUNCH("rs_tree_sample/walk");
    }
    return RS_OK;
}
