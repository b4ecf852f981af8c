// sample.cu -- rs_tree_sample: lossless verification of model-drafted nodes
// by sampling (Section 3.4, "For Drafter Module outputs": standard lossless
// speculative sampling).
//
// With deterministic (top-w) model children, speculative sampling over the
// siblings has the law of: draw y from the target row at temperature T,
// accept the model child that carries y and continue from it, otherwise emit
// y as the correction token.  Each row's draw is the inverse CDF, in
// token-id order, of a caller-supplied uniform u:  the smallest id v with
// sum_{w <= v} p_T(w) > u.
//
// Kernel 1 (sample_partial): one CTA per (row, 8192-logit chunk), staged
// through shared memory with coalesced loads; thread t
// owns the 32 consecutive ids c0 + 32 t .. c0 + 32 t + 31 and sums
// e_v = 2^((z_v - m_c) log2(e) / T) over them in id order, m_c being the
// chunk maximum; the chunk's (m_c, s_c) go to the workspace.
// Kernel 2 (sample_pick): one CTA per row.  Warp 0 rescales the chunk sums to
// the row maximum, takes their inclusive prefix in chunk order and finds the
// chunk where it passes u Z; the CTA then recomputes that chunk's e_v (the
// same per-thread sums as kernel 1), scans the thread sums and lets the
// thread holding the crossing walk its 32 ids.  Rounding that leaves u Z at
// or past the total picks the last id with mass.
// Kernel 3 (sample_walk): one warp per request checks the tree and follows,
// from the root, the model child (source 1) carrying the current node's draw.
#include <math.h>

#include "common.cuh"

namespace rs {
namespace {

constexpr int kSmpThreads = 256;
constexpr int kSmpVpt = 32;                       // consecutive ids per thread
constexpr int kSmpChunk = kSmpThreads * kSmpVpt;  // 8192 ids per chunk
constexpr float kL2E = 1.4426950408889634f;

struct ChunkMass {
    float m;  // chunk maximum (-inf: no mass)
    float s;  // sum over the chunk of 2^((z - m) log2(e) / T)
};

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
    for (int w = 1; w < kSmpThreads / 32; ++w) r = fmaxf(r, s_w[w]);
    __syncthreads();
    return r;
}

// Inclusive prefix of one float per thread in thread order, and the total.
__device__ __forceinline__ float block_incl_scan(float v, float *s_w, float *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    float x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) s_w[warp] = x;
    __syncthreads();
    float before = 0.f, sum = 0.f;
#pragma unroll
    for (int w = 0; w < kSmpThreads / 32; ++w) {
        const float y = s_w[w];
        before += w < warp ? y : 0.f;
        sum += y;
    }
    __syncthreads();
    *total = sum;
    return before + x;
}

template <int kW>
__global__ void __launch_bounds__(kSmpThreads)
sample_partial(const float *__restrict__ logits, int V, int nchunks, float scale, ChunkMass *__restrict__ part) {
    pdl_enter();
    __shared__ float s_w[kSmpThreads / 32];
    __shared__ __align__(16) float s_buf[kSmpPadded];
    const int r = blockIdx.x / nchunks, c = blockIdx.x - r * nchunks;
    const float *row = logits + (long long)r * V;
    float z[kSmpVpt];
    load32_staged<kW>(row, V, c * kSmpChunk, s_buf, z);
    float mx = -INFINITY;
#pragma unroll
    for (int j = 0; j < kSmpVpt; ++j) mx = fmaxf(mx, z[j]);
    const float m = block_max(mx, s_w);
    float s = 0.f;
    if (m != -INFINITY) {
        const float nb = -m * scale;
#pragma unroll
        for (int j = 0; j < kSmpVpt; ++j) s += ex2f(fmaf(z[j], scale, nb));  // id order within the thread
    }
    float tot;
    (void)block_incl_scan(s, s_w, &tot);
    if (threadIdx.x == 0) part[blockIdx.x] = ChunkMass{m, tot};
}

template <int kW>
__global__ void __launch_bounds__(kSmpThreads)
sample_pick(const float *__restrict__ logits, int V, int nchunks, float scale, const ChunkMass *__restrict__ part,
            const float *__restrict__ uniforms, int32_t *__restrict__ draw) {
    pdl_enter();
    __shared__ float s_w[kSmpThreads / 32];
    __shared__ int s_chunk;
    __shared__ float s_target;  // u Z within the chosen chunk, in its own units
    __shared__ int s_draw;
    __shared__ __align__(16) float s_buf[kSmpPadded];
    const int r = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31;
    const ChunkMass *pr = part + (long long)r * nchunks;

    if (tid < 32) {
        // row maximum, then the chunk weights in chunk order
        float M = -INFINITY;
        for (int c = lane; c < nchunks; c += 32) M = fmaxf(M, pr[c].m);
        M = warp_max(M);
        const float u = uniforms[r];
        float carry = 0.f;  // sum of the chunks before this round
        int pick = -1, last = -1;
        float pick_before = 0.f;
        float total = 0.f;
        // pass 1: the total Z (chunk order); pass 2: the crossing
        for (int c0 = 0; c0 < nchunks; c0 += 32) {
            const int c = c0 + lane;
            const ChunkMass cm = c < nchunks ? pr[c] : ChunkMass{-INFINITY, 0.f};
            const float w = cm.m == -INFINITY ? 0.f : cm.s * ex2f((cm.m - M) * scale);
            total += warp_sum(w);
        }
        const float target = u * total;
        for (int c0 = 0; c0 < nchunks && pick < 0; c0 += 32) {
            const int c = c0 + lane;
            const ChunkMass cm = c < nchunks ? pr[c] : ChunkMass{-INFINITY, 0.f};
            const float w = cm.m == -INFINITY ? 0.f : cm.s * ex2f((cm.m - M) * scale);
            float x = w;  // inclusive prefix within the round
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const float y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            const unsigned cross = __ballot_sync(0xffffffffu, w > 0.f && carry + x > target);
            const unsigned mass = __ballot_sync(0xffffffffu, w > 0.f);
            if (cross) {
                const int l = __ffs(cross) - 1;
                pick = c0 + l;
                pick_before = carry + __shfl_sync(0xffffffffu, x - w, l);
            }
            if (mass) last = c0 + 31 - __clz(mass);
            carry += __shfl_sync(0xffffffffu, x, 31);
        }
        if (lane == 0) {
            float t_loc;
            int c = pick;
            if (c < 0) {  // u Z at or past the rounded total: the last chunk with mass, its end
                c = last;
                t_loc = INFINITY;
            } else {
                const ChunkMass cm = pr[c];
                t_loc = (target - pick_before) / ex2f((cm.m - M) * scale);
            }
            s_chunk = c;
            s_target = t_loc;
        }
    }
    __syncthreads();
    const int c = s_chunk;
    if (c < 0) {  // the row has no mass at all
        if (tid == 0) draw[r] = 0;
        return;
    }
    // the chosen chunk: the same per-thread sums as sample_partial, scanned in id order
    const float m = pr[c].m;
    const float nb = -m * scale;
    const float *row = logits + (long long)r * V;
    float z[kSmpVpt];
    load32_staged<kW>(row, V, c * kSmpChunk, s_buf, z);
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < kSmpVpt; ++j) s += ex2f(fmaf(z[j], scale, nb));
    float tot;
    const float incl = block_incl_scan(s, s_w, &tot);
    const float t_loc = s_target;
    // the draw lies in the lowest thread whose inclusive prefix passes the target
    if (tid == 0) s_draw = 0x7fffffff;
    __syncthreads();
    const unsigned pass = __ballot_sync(0xffffffffu, s > 0.f && incl > t_loc);
    if (lane == 0 && pass) atomicMin(&s_draw, (tid & ~31) + __ffs(pass) - 1);
    __syncthreads();
    const int holder = s_draw;
    __syncthreads();
    if (tid == holder) {
        float cum = incl - s;  // this thread's exclusive prefix
        int v = -1, lastv = 0;
#pragma unroll
        for (int j = 0; j < kSmpVpt; ++j) {
            const float e = ex2f(fmaf(z[j], scale, nb));
            if (e > 0.f) lastv = j;
            cum += e;
            if (v < 0 && cum > t_loc) v = j;
        }
        if (v < 0) v = lastv;  // rounding: the thread's last id with mass
        s_draw = c * kSmpChunk + tid * kSmpVpt + v;
    } else if (tid == 0 && holder == 0x7fffffff) {
        s_draw = -1;
    }
    __syncthreads();
    if (tid == 0) {
        int d = s_draw;
        if (d < 0) {  // no thread passed the target: the chunk's last id with mass
            d = c * kSmpChunk;
            for (int v = min(V, (c + 1) * kSmpChunk) - 1; v >= c * kSmpChunk; --v)
                if (ex2f(fmaf(row[v], scale, nb)) > 0.f) {
                    d = v;
                    break;
                }
        }
        draw[r] = d;
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
    int par[kPer], tok[kPer];
    bool model[kPer];
    bool bad = false;
#pragma unroll
    for (int q = 0; q < kPer; ++q) {
        const int i = lane + 32 * q;
        par[q] = -2;
        tok[q] = -1;
        model[q] = false;
        if (st == 0 && i < N) {
            const int pa = parents[n0 + i], sr = source[n0 + i];
            par[q] = pa;
            tok[q] = tokens[n0 + i];
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
        const int y = draw[n0 + cur];
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

extern "C" size_t rs_tree_sample_workspace_size(int R, int V) {
    if (R < 0 || V < 1) return 0;
    const size_t nchunks = (size_t)(V + kSmpChunk - 1) / kSmpChunk;
    return align_up((size_t)R * nchunks * sizeof(ChunkMass), 256);
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
    RS_CHECK_ARG((long long)R * nchunks < (1ll << 31), "rs_tree_sample: R*chunks too large");
    const size_t need = rs_tree_sample_workspace_size(R, V);
    if (workspace_bytes < need || (need && !workspace)) {
        set_error("rs_tree_sample: workspace %zu bytes < %zu required", workspace_bytes, need);
        return RS_ERR_CAPACITY;
    }
    cudaStream_t st = (cudaStream_t)stream;
    ChunkMass *part = static_cast<ChunkMass *>(workspace);
    const float scale = kL2E / temperature;
    if (R > 0) {
        const int w = (V % 8 == 0 && ((uintptr_t)logits & 31) == 0) ? 8
                      : (V % 4 == 0 && ((uintptr_t)logits & 15) == 0) ? 4 : 1;
        const unsigned blocks = (unsigned)((long long)R * nchunks);
        const dim3 blk(kSmpThreads);
        if (w == 8) launch_pdl(sample_partial<8>, dim3(blocks), blk, 0, st, logits, V, nchunks, scale, part);
        else if (w == 4) launch_pdl(sample_partial<4>, dim3(blocks), blk, 0, st, logits, V, nchunks, scale, part);
        else launch_pdl(sample_partial<1>, dim3(blocks), blk, 0, st, logits, V, nchunks, scale, part);
        RS_CHECK_LAUNCH("rs_tree_sample/partial");
        if (w == 8) launch_pdl(sample_pick<8>, dim3(R), blk, 0, st, logits, V, nchunks, scale, part, uniforms, draw);
        else if (w == 4) launch_pdl(sample_pick<4>, dim3(R), blk, 0, st, logits, V, nchunks, scale, part, uniforms, draw);
        else launch_pdl(sample_pick<1>, dim3(R), blk, 0, st, logits, V, nchunks, scale, part, uniforms, draw);
        RS_CHECK_LAUNCH("rs_tree_sample/pick");
    }
    if (B > 0) {
        launch_pdl(sample_walk, dim3(B), dim3(32), 0, st, node_off, R, tokens, parents, source, draw, acc_cap, acc_len,
            acc_nodes, bonus, status);
        RS_CHECK_LAUNCH("rs_tree_sample/walk");
    }
    return RS_OK;
}
