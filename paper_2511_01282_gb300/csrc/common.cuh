// common.cuh -- shared helpers of the sm_103a ReSpec library (host checks,
// error reporting, launch accounting, warp/block reductions).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>
#include <stdio.h>

#include <cstdarg>

#include "respec.h"

namespace rs {

// ---------------------------------------------------------------- host side
void set_error(const char *fmt, ...);
void clear_error();
void count_launch(int n = 1);

#define RS_CHECK_ARG(cond, ...)                            \
    do {                                                   \
        if (!(cond)) {                                     \
            ::rs::set_error(__VA_ARGS__);                  \
            return RS_ERR_INVALID_ARG;                     \
        }                                                  \
    } while (0)

#define RS_CHECK_LAUNCH(what)                                                        \
    do {                                                                             \
        cudaError_t e_ = cudaGetLastError();                                         \
        if (e_ != cudaSuccess) {                                                     \
            ::rs::set_error("%s: launch failed: %s", what, cudaGetErrorString(e_));  \
            return RS_ERR_CUDA;                                                      \
        }                                                                            \
        ::rs::count_launch();                                                        \
    } while (0)

// Kernels are launched with programmatic stream serialization: the next
// kernel in the stream may begin launching as soon as every block of this one
// has started (pdl_enter's first instruction), and each kernel waits for its
// predecessor's completion and memory before it touches global memory (its
// second).  Since every kernel waits, completion stays ordered along the
// whole stream.  Without a programmatic predecessor the wait returns at once.
// Persistent kernels, whose grid assumes every SM free, use launch_full
// instead: they start only once the previous kernel has finished.
template <bool kEarly = true, typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = kEarly ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}
// The same with a one-dimensional cluster of `cluster_x` CTAs along x
// (grid.x a multiple of it; at most 8, the portable cluster size).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_cluster(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                               int cluster_x, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = (unsigned)cluster_x;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}
template <typename... KArgs, typename... Args>
cudaError_t launch_full(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                        Args... args) {
    return launch_pdl<false>(kern, grid, block, smem, st, args...);
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Bump allocator over the caller's workspace (256-byte aligned slices).
struct Carve {
    char *base;
    size_t off = 0;
    explicit Carve(void *p) : base(static_cast<char *>(p)) {}
    template <class T>
    T *take(size_t n) {
        off = align_up(off, 256);
        T *p = reinterpret_cast<T *>(base ? base + off : nullptr);
        off += n * sizeof(T);
        return p;
    }
    size_t used() const { return align_up(off, 256); }
};

int num_sms();  // SM count of the current device (cached per device)
long long l2_bytes();  // L2 size of the current device (cached per device)

// ---------------------------------------------------------------- device side
// Let the next kernel start launching, then wait for the previous kernel.
__device__ __forceinline__ void pdl_launch_next() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait_prev() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_enter() {
    pdl_launch_next();
    pdl_wait_prev();
}

// The two halves of the cluster barrier, for every thread of every CTA of
// the cluster.  A CTA may write another CTA's shared memory only once that
// CTA is known to be running: arrive (relaxed) at entry, wait before the
// first remote store.  arrive_release + wait then makes the remote stores
// visible to their owners.
__device__ __forceinline__ void cluster_arrive_relaxed() { asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory"); }
__device__ __forceinline__ void cluster_arrive_release() { asm volatile("barrier.cluster.arrive.release;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire;" ::: "memory"); }

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
// (value, id) total order used for argmax / TopK: larger value first, then
// smaller id.  Returns true when (va, ia) comes strictly before (vb, ib).
__device__ __forceinline__ bool vi_before(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

// Read-only, L1-bypassing streaming loads for data read exactly once.
__device__ __forceinline__ float4 ldg_stream4(const float4 *p) {
    float4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(r.x), "=f"(r.y), "=f"(r.z), "=f"(r.w)
                 : "l"(p));
    return r;
}
// 256-bit variant (p 32-byte aligned).
__device__ __forceinline__ void ldg_stream8(const float *p, float (&r)[8]) {
    asm volatile("ld.global.nc.L1::no_allocate.v8.f32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=f"(r[0]), "=f"(r[1]), "=f"(r[2]), "=f"(r[3]), "=f"(r[4]), "=f"(r[5]), "=f"(r[6]), "=f"(r[7])
                 : "l"(p));
}
__device__ __forceinline__ float ldg_stream(const float *p) {
    float r;
    asm volatile("ld.global.nc.L1::no_allocate.f32 %0, [%1];" : "=f"(r) : "l"(p));
    return r;
}

}  // namespace rs
