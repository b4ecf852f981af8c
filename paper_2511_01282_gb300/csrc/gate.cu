// gate.cu -- rs_entropy_gate: entropy-guided adaptive trigger
// (Section 3.2.1, Eq. 1-3 and the trigger decision; Algorithm 1's triggering).
//
// Kernel 1 (entropy_partial): one CTA per (row, 8192-logit chunk).  Each
// thread streams 32 logits with 128-bit loads; relative to its warp's
// maximum m the warp forms s = sum e^(z-m) and w = sum e^(z-m) (z-m) (plain
// shuffle sums), and one thread merges the eight warp triples into the
// chunk's.  Row entropy is then H = ln s - w / s for the merged triple (the
// log-sum-exp form of -sum p ln p).
// Kernel 2 (entropy_merge): one warp per row merges its chunk triples into
// the row entropy.  Kernel 3 (gate_push): one CTA per request pushes the
// committed rows' entropies into the history and evaluates H_k, C_k, k* and
// the trigger in fp64.  rs_entropy_gate_rows runs kernel 3 alone on row
// entropies that rs_accept already produced from the same logits.
#include <math.h>

#include <mutex>

#include "common.cuh"

namespace rs {
namespace {

constexpr int kGateThreads = 256;
constexpr int kGateVpt = 32;                          // logits per thread
constexpr int kGateChunk = kGateThreads * kGateVpt;   // logits per CTA

struct Ent3 {
    float m, s, w;
};

__device__ __forceinline__ Ent3 ent_merge(Ent3 a, Ent3 b) {
    if (a.s == 0.f) return b;
    if (b.s == 0.f) return a;
    float M = fmaxf(a.m, b.m);
    float ca = __expf(a.m - M), cb = __expf(b.m - M);
    Ent3 r;
    r.m = M;
    r.s = a.s * ca + b.s * cb;
    r.w = ca * (a.w + a.s * (a.m - M)) + cb * (b.w + b.s * (b.m - M));
    return r;
}

__device__ __forceinline__ Ent3 ent_shfl(Ent3 a, int o) {
    Ent3 b;
    b.m = __shfl_xor_sync(0xffffffffu, a.m, o);
    b.s = __shfl_xor_sync(0xffffffffu, a.s, o);
    b.w = __shfl_xor_sync(0xffffffffu, a.w, o);
    return b;
}

__device__ __forceinline__ float ex2f_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// kW: logits per load (8: V % 8 == 0 and 32-byte aligned logits; 4: V % 4 ==
// 0 and 16-byte alignment; else 1).
template <int kW>
__global__ void __launch_bounds__(kGateThreads)
entropy_partial(const float *__restrict__ logits, int V, int nchunks, Ent3 *__restrict__ part) {
    pdl_enter();
    const long long blk = blockIdx.x;
    const long long r = blockIdx.x / (unsigned)nchunks;  // 32-bit division
    const int chunk = (int)(blk - r * nchunks);
    const float *row = logits + r * (long long)V;
    const int c0 = chunk * kGateChunk;
    const int tid = threadIdx.x;

    float v[kGateVpt];
    if (kW == 8) {
        // 4 x 256-bit loads per thread, each iteration a contiguous 8 KB sweep
#pragma unroll
        for (int j = 0; j < kGateVpt / 8; ++j) {
            const int idx = c0 + (j * kGateThreads + tid) * 8;
            float x[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) x[k] = -INFINITY;
            if (idx < V) ldg_stream8(row + idx, x);  // V % 8 == 0: whole groups of 8
#pragma unroll
            for (int k = 0; k < 8; ++k) v[8 * j + k] = x[k];
        }
    } else if (kW == 4) {
        // 8 x float4 per thread, each iteration a contiguous 4 KB sweep
#pragma unroll
        for (int j = 0; j < kGateVpt / 4; ++j) {
            int idx = c0 + (j * kGateThreads + tid) * 4;
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
        for (int j = 0; j < kGateVpt; ++j) {
            int idx = c0 + j * kGateThreads + tid;
            v[j] = idx < V ? ldg_stream(row + idx) : -INFINITY;
        }
    }

    // warp maximum as the common reference: the warp's triple is a plain sum
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < kGateVpt; ++i) mx = fmaxf(mx, v[i]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    Ent3 t{mx, 0.f, 0.f};
    if (mx != -INFINITY) {
        constexpr float kL2E = 1.4426950408889634f;
        float s4[4] = {0.f, 0.f, 0.f, 0.f}, w4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int i = 0; i < kGateVpt; ++i) {
            const float d = fmaxf(v[i] - mx, -1e30f);  // -inf -> -1e30: e = 0, e*d = 0
            const float e = ex2f_approx(d * kL2E);
            s4[i & 3] += e;
            w4[i & 3] = fmaf(e, d, w4[i & 3]);
        }
        float ss = (s4[0] + s4[1]) + (s4[2] + s4[3]);
        float ww = (w4[0] + w4[1]) + (w4[2] + w4[3]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            ss += __shfl_xor_sync(0xffffffffu, ss, o);
            ww += __shfl_xor_sync(0xffffffffu, ww, o);
        }
        t.s = ss;
        t.w = ww;
    }
    __shared__ Ent3 sw[kGateThreads / 32];
    if ((tid & 31) == 0) sw[tid >> 5] = t;
    __syncthreads();
    if (tid == 0) {
        Ent3 a = sw[0];
#pragma unroll
        for (int w = 1; w < kGateThreads / 32; ++w) a = ent_merge(a, sw[w]);
        part[blk] = a;
    }
}

constexpr int kMergeThreads = 256;

__global__ void __launch_bounds__(kMergeThreads)
entropy_merge(const Ent3 *__restrict__ part, int nchunks, int R, float *__restrict__ entropy) {
    pdl_enter();
    const int lane = threadIdx.x & 31;
    const long long r = (long long)blockIdx.x * (kMergeThreads / 32) + (threadIdx.x >> 5);
    if (r >= R) return;
    Ent3 t{-INFINITY, 0.f, 0.f};
    for (int c = lane; c < nchunks; c += 32) t = ent_merge(t, part[r * nchunks + c]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t = ent_merge(t, ent_shfl(t, o));
    if (lane == 0) entropy[r] = t.s > 0.f ? (__logf(t.s) - t.w / t.s) : 0.f;
}

// Per request: the committed rows' entropies, in row order, extend the
// history and the newest l entries are kept; a block scan gives every
// committed row its rank, so each surviving entry is written by its own
// thread.  Then Algorithm 1's triggering in fp64 with one lane per k (H_k, C_k)
// and a warp argmin that keeps the smallest k among equal C_k (the first
// strict minimum of the upward scan).
constexpr int kPushThreads = 256;
constexpr int kPushWarps = kPushThreads / 32;

// Exclusive prefix of one int per thread over the block (and the block sum).
__device__ __forceinline__ int push_scan(int v, int *s_w, int *total) {
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
    for (int w = 0; w < kPushWarps; ++w) {
        const int y = s_w[w];
        before += w < warp ? y : 0;
        sum += y;
    }
    __syncthreads();  // s_w reusable
    *total = sum;
    return before + x - v;
}

__global__ void __launch_bounds__(kPushThreads)
gate_push(const float *__restrict__ entropy, const int32_t *__restrict__ row_off,
          const uint8_t *__restrict__ row_commit, int R, rs_params p, float *__restrict__ hist,
          int32_t *__restrict__ hist_n, int32_t *__restrict__ k_star, float *__restrict__ h_best,
          uint8_t *__restrict__ entropy_ok) {
    pdl_enter();
    const int b = blockIdx.x, tid = threadIdx.x;
    // rows [r0, r1) must lie in [0, R) (R < 0: the row offsets' last entry);
    // a range outside them pushes nothing
    const int rend = R >= 0 ? R : row_off[gridDim.x];
    int r0 = row_off[b], r1 = row_off[b + 1];
    if (r0 < 0 || r1 < r0 || r1 > rend) r0 = r1 = 0;
    const int l = p.l;
    __shared__ float s_h[RS_MAX_L];
    __shared__ int s_w[kPushWarps];
    int n = hist_n[b];
    n = n < 0 ? 0 : (n > l ? l : n);

    // committed rows c; the newest m = min(c, l) of them and the newest
    // keep = min(n, l - m) old entries form the new history
    int cnt = 0;
    for (int r = r0 + tid; r < r1; r += kPushThreads) cnt += row_commit[r] != 0;
    int c = 0;
    (void)push_scan(cnt, s_w, &c);
    const int m = c < l ? c : l;
    const int keep = n < l - m ? n : l - m;
    const int nn = keep + m;
    const float old = tid < keep ? hist[(long long)b * l + n - keep + tid] : 0.f;
    if (tid < keep) s_h[tid] = old;
    int carry = 0;
    for (int base = r0; base < r1; base += kPushThreads) {
        const int r = base + tid;
        const bool f = r < r1 && row_commit[r] != 0;
        int tot = 0;
        const int q = carry + push_scan(f ? 1 : 0, s_w, &tot);
        if (f && q >= c - m) s_h[keep + q - (c - m)] = entropy[r];
        carry += tot;
    }
    __syncthreads();
    if (tid < nn) hist[(long long)b * l + tid] = s_h[tid];
    if (tid >= 32) return;

    const int k = tid + 1;
    double ck = INFINITY, hk = INFINITY;
    if (k <= nn) {
        double sum = 0.0;
        for (int i = nn - k; i < nn; ++i) sum = __dadd_rn(sum, (double)s_h[i]);
        hk = __ddiv_rn(sum, (double)k);
        ck = __dadd_rn(hk, __ddiv_rn((double)p.lambda_e, (double)k));
        if (ck != ck) ck = INFINITY;  // a NaN never wins the strict comparison
    }
    int bk = k;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const double oc = __shfl_xor_sync(0xffffffffu, ck, o);
        const double oh = __shfl_xor_sync(0xffffffffu, hk, o);
        const int ok = __shfl_xor_sync(0xffffffffu, bk, o);
        if (oc < ck || (oc == ck && ok < bk)) {
            ck = oc;
            hk = oh;
            bk = ok;
        }
    }
    if (tid == 0) {
        hist_n[b] = nn;
        const bool found = ck < INFINITY;
        const int kbest = found ? bk : 0;
        const double best = found ? hk : INFINITY;
        k_star[b] = kbest;
        h_best[b] = (float)best;
        entropy_ok[b] = (uint8_t)(kbest > 0 && best <= (double)p.theta_entropy);
    }
}

// The three launches of a gate call over the chunk triples in `part`.
rs_status launch_gate(const char *who, const float *logits, int R, int V, int nchunks, Ent3 *part,
                      const int32_t *row_off, const uint8_t *row_commit, int B, rs_params p, float *hist,
                      int32_t *hist_n, float *entropy, int32_t *k_star, float *h_best, uint8_t *entropy_ok,
                      cudaStream_t st) {
    if (R > 0) {
        const long long blocks = (long long)R * nchunks;
        if (blocks >= (1ll << 31)) {
            set_error("%s: R*chunks too large", who);
            return RS_ERR_INVALID_ARG;
        }
        const int w = (V % 8 == 0 && ((uintptr_t)logits & 31) == 0) ? 8
                      : (V % 4 == 0 && ((uintptr_t)logits & 15) == 0) ? 4 : 1;
        if (w == 8)
            launch_pdl(entropy_partial<8>, dim3((unsigned)blocks), dim3(kGateThreads), 0, st, logits, V, nchunks,
                part);
        else if (w == 4)
            launch_pdl(entropy_partial<4>, dim3((unsigned)blocks), dim3(kGateThreads), 0, st, logits, V, nchunks,
                part);
        else
            launch_pdl(entropy_partial<1>, dim3((unsigned)blocks), dim3(kGateThreads), 0, st, logits, V, nchunks,
                part);
        RS_CHECK_LAUNCH(who);
        launch_pdl(entropy_merge, dim3((R + kMergeThreads / 32 - 1) / (kMergeThreads / 32)), dim3(kMergeThreads),
            0, st, part, nchunks, R, entropy);
        RS_CHECK_LAUNCH(who);
    }
    if (B > 0) {
        launch_pdl(gate_push, dim3(B), dim3(kPushThreads), 0, st, entropy, row_off, row_commit, R, p, hist, hist_n,
            k_star, h_best, entropy_ok);
        RS_CHECK_LAUNCH(who);
    }
    return RS_OK;
}

}  // namespace
}  // namespace rs

using namespace rs;

extern "C" size_t rs_entropy_gate_workspace_size(int R, int V) {
    if (R < 0 || V < 1) return 0;
    int nchunks = (V + kGateChunk - 1) / kGateChunk;
    Carve cv(nullptr);
    cv.take<Ent3>((size_t)R * nchunks);
    return cv.used();
}

extern "C" rs_status rs_entropy_gate(const float *logits, int R, int V, const int32_t *row_off,
                                     const uint8_t *row_commit, int B, rs_params p, float *hist,
                                     int32_t *hist_n, float *entropy, int32_t *k_star, float *h_best,
                                     uint8_t *entropy_ok, void *workspace, size_t workspace_bytes,
                                     void *stream) {
    clear_error();
    RS_CHECK_ARG(R >= 0 && B >= 0, "rs_entropy_gate: negative size (R=%d, B=%d)", R, B);
    RS_CHECK_ARG(V >= 1, "rs_entropy_gate: V must be >= 1 (got %d)", V);
    RS_CHECK_ARG(p.l >= 1 && p.l <= RS_MAX_L, "rs_entropy_gate: l=%d outside [1, %d]", p.l, RS_MAX_L);
    RS_CHECK_ARG(R == 0 || (logits && entropy && row_commit), "rs_entropy_gate: null row pointer");
    RS_CHECK_ARG(B == 0 || (row_off && hist && hist_n && k_star && h_best && entropy_ok),
                 "rs_entropy_gate: null request pointer");
    const int nchunks = (V + kGateChunk - 1) / kGateChunk;
    const size_t need = rs_entropy_gate_workspace_size(R, V);
    if (workspace_bytes < need || (need && !workspace)) {
        set_error("rs_entropy_gate: workspace %zu bytes < %zu required", workspace_bytes, need);
        return RS_ERR_CAPACITY;
    }
    Carve cv(workspace);
    Ent3 *part = cv.take<Ent3>((size_t)R * nchunks);
    return launch_gate("rs_entropy_gate", logits, R, V, nchunks, part, row_off, row_commit, B, p, hist, hist_n,
                       entropy, k_star, h_best, entropy_ok, (cudaStream_t)stream);
}

// ============================================================ no-allocation variant
// rs_entropy_gate_noalloc runs the same three kernels as rs_entropy_gate
// (entropy_partial, entropy_merge, gate_push), with the per-chunk partials in
// the fixed device array below instead of a caller workspace, for callers
// that cannot allocate device memory.  The array (RS_GATE_NOALLOC_MAX_PARTIALS
// triples, 12 bytes each) lives on every GPU that loads this library until
// the process exits.  It needs no initialisation: every partial a call reads
// was written earlier by the same call.  All calls share it, so calls that
// overlap on the GPU (different streams, or several host threads without
// ordering) race on it.
static __device__ __align__(256) Ent3 g_gate_scratch[RS_GATE_NOALLOC_MAX_PARTIALS];

// Unique id of the calling thread's current CUDA context (0 when it cannot be
// read).  Context ids are never reused within a process, so a device reset or
// another context on the same device gives a new id.
static unsigned long long current_context_id() {
    typedef int (*ctx_get_current_t)(void **);
    typedef int (*ctx_get_id_t)(void *, unsigned long long *);
    static std::once_flag once;
    static ctx_get_current_t get_current = nullptr;
    static ctx_get_id_t get_id = nullptr;
    std::call_once(once, [] {
        void *a = nullptr, *b = nullptr;
        cudaDriverEntryPointQueryResult qa, qb;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &a, 12000, cudaEnableDefault, &qa) ==
                cudaSuccess && qa == cudaDriverEntryPointSuccess &&
            cudaGetDriverEntryPointByVersion("cuCtxGetId", &b, 12000, cudaEnableDefault, &qb) == cudaSuccess &&
            qb == cudaDriverEntryPointSuccess) {
            get_current = reinterpret_cast<ctx_get_current_t>(a);
            get_id = reinterpret_cast<ctx_get_id_t>(b);
        }
    });
    if (!get_current || !get_id) return 0;
    void *ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != 0 || !ctx || get_id(ctx, &id) != 0) return 0;
    return id;
}

// Device address of g_gate_scratch in the current context (the host-side name
// is only a stand-in for the symbol).  Looked up with cudaGetSymbolAddress on
// the first call in each context of each device and remembered with that
// context's id; when the id cannot be read the address is looked up anew.
static Ent3 *gate_scratch_address(int dev) {
    static std::mutex mu;
    static unsigned long long ctx_of[64] = {0};
    static Ent3 *addr[64] = {nullptr};
    if (dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lk(mu);
    const unsigned long long id = current_context_id();
    if (id != 0 && ctx_of[dev] == id && addr[dev]) return addr[dev];
    void *ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_gate_scratch);
    if (e != cudaSuccess) {
        set_error("rs_entropy_gate_noalloc: cudaGetSymbolAddress: %s", cudaGetErrorString(e));
        return nullptr;
    }
    addr[dev] = static_cast<Ent3 *>(ptr);
    ctx_of[dev] = current_context_id();  // the lookup made the context current if it was not
    return addr[dev];
}

extern "C" rs_status rs_entropy_gate_noalloc(const float *logits, int R, int V, const int32_t *row_off,
                                             const uint8_t *row_commit, int B, rs_params p, float *hist,
                                             int32_t *hist_n, float *entropy, int32_t *k_star, float *h_best,
                                             uint8_t *entropy_ok, void *stream) {
    clear_error();
    RS_CHECK_ARG(R >= 0 && B >= 0, "rs_entropy_gate_noalloc: negative size (R=%d, B=%d)", R, B);
    RS_CHECK_ARG(V >= 1, "rs_entropy_gate_noalloc: V must be >= 1 (got %d)", V);
    RS_CHECK_ARG(p.l >= 1 && p.l <= RS_MAX_L, "rs_entropy_gate_noalloc: l=%d outside [1, %d]", p.l, RS_MAX_L);
    RS_CHECK_ARG(R == 0 || (logits && entropy && row_commit), "rs_entropy_gate_noalloc: null row pointer");
    RS_CHECK_ARG(B == 0 || (row_off && hist && hist_n && k_star && h_best && entropy_ok),
                 "rs_entropy_gate_noalloc: null request pointer");
    const int nchunks = (V + kGateChunk - 1) / kGateChunk;
    const long long partials = (long long)R * nchunks;
    if (partials > RS_GATE_NOALLOC_MAX_PARTIALS) {
        set_error("rs_entropy_gate_noalloc: R=%d rows x %d chunks of %d logits = %lld partials exceed the "
                  "fixed scratch of %d (at most %d rows at this V)",
                  R, nchunks, kGateChunk, partials, RS_GATE_NOALLOC_MAX_PARTIALS,
                  RS_GATE_NOALLOC_MAX_PARTIALS / nchunks);
        return RS_ERR_CAPACITY;
    }
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        set_error("rs_entropy_gate_noalloc: cudaGetDevice: %s", cudaGetErrorString(e));
        return RS_ERR_CUDA;
    }
    Ent3 *part = gate_scratch_address(dev);
    if (!part) {
        if (!rs_last_error()[0]) set_error("rs_entropy_gate_noalloc: device %d not supported", dev);
        return RS_ERR_CUDA;
    }
    return launch_gate("rs_entropy_gate_noalloc", logits, R, V, nchunks, part, row_off, row_commit, B, p, hist,
                       hist_n, entropy, k_star, h_best, entropy_ok, (cudaStream_t)stream);
}

extern "C" rs_status rs_entropy_gate_rows(const float *entropy, const int32_t *row_off, const uint8_t *row_commit,
                                          int B, rs_params p, float *hist, int32_t *hist_n, int32_t *k_star,
                                          float *h_best, uint8_t *entropy_ok, void *stream) {
    clear_error();
    RS_CHECK_ARG(B >= 0, "rs_entropy_gate_rows: negative B");
    RS_CHECK_ARG(p.l >= 1 && p.l <= RS_MAX_L, "rs_entropy_gate_rows: l=%d outside [1, %d]", p.l, RS_MAX_L);
    RS_CHECK_ARG(B == 0 || (entropy && row_off && row_commit && hist && hist_n && k_star && h_best && entropy_ok),
                 "rs_entropy_gate_rows: null pointer");
    if (B == 0) return RS_OK;
    launch_pdl(gate_push, dim3(B), dim3(kPushThreads), 0, (cudaStream_t)stream, entropy, row_off, row_commit, -1,
        p, hist, hist_n, k_star, h_best, entropy_ok);
    RS_CHECK_LAUNCH("rs_entropy_gate_rows");
    return RS_OK;
}
