// Shared device-side definitions of the MSD kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cstdint>
#include <utility>

namespace msd {

typedef __nv_bfloat16 bf16;

// One row of a layer pass: which request it belongs to, its RoPE position, how
// many cache positions it attends to ([0, plen)), and where its own K/V go (a
// cache position or a tree slot; -1 = nowhere).
struct RowDesc {
    int req;
    int pos;
    int plen;
    int dst;
};

// Device status codes (first one set wins).
enum : int {
    ST_OK = 0,
    ST_BAD_TOKEN = 1,     // token id outside [0, V)
    ST_BAD_TREE = 2,      // malformed tree (parent >= child, depth mismatch)
    ST_RANGE = 3,         // an index outside its buffer was skipped
    ST_TIMEOUT = 4,       // a bounded wait ran out
};

// Host-side count of kernel launches made by the library (profiling).
long launch_count();
void note_launch();

__device__ __forceinline__ void set_status(int *st, int code) {
    if (st) atomicCAS(st, 0, code);
}

// Lets a dependent kernel launched with programmatic stream serialization
// start its prologue now; it still waits for this grid before reading any of
// its outputs (griddepcontrol.wait). Every kernel calls it only after its own
// wait_prior(): a kernel that has started therefore implies that the kernel
// two launches back has completed, so a prologue may read, before its own
// wait, data last written two or more launches earlier (weights, caches
// written by earlier steps, row descriptors of earlier set-up kernels).
__device__ __forceinline__ void allow_dependents() {
    asm volatile("griddepcontrol.launch_dependents;");
}

// Waits until the grids this one depends on have completed and their writes
// are visible. Every kernel launched by launch_pdl calls it before it reads
// anything the previous kernel may have written, so that completion stays
// transitive along the stream.
__device__ __forceinline__ void wait_prior() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Launches `kernel` with programmatic stream serialization: its CTAs may be
// scheduled while the previous kernel on `s` finishes (its launch latency
// overlaps that kernel's tail); the kernel orders itself with wait_prior().
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t lc = {};
    lc.gridDim = grid;
    lc.blockDim = block;
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, kernel, std::forward<Args>(args)...);
}

template <typename T> __device__ __forceinline__ float to_f(T v);
template <> __device__ __forceinline__ float to_f<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f<bf16>(bf16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Block-wide sum for blockDim.x a multiple of 32 (<= 1024). `red` holds 32 floats.
__device__ __forceinline__ float block_sum(float v, float *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_sum(v);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    const int nw = blockDim.x >> 5;
    float t = (threadIdx.x < nw) ? red[threadIdx.x] : 0.f;
    if (warp == 0) t = warp_sum(t);
    if (threadIdx.x == 0) red[0] = t;
    __syncthreads();
    return red[0];
}

__device__ __forceinline__ float block_max(float v, float *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    v = warp_max(v);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    const int nw = blockDim.x >> 5;
    float t = (threadIdx.x < nw) ? red[threadIdx.x] : -INFINITY;
    if (warp == 0) t = warp_max(t);
    if (threadIdx.x == 0) red[0] = t;
    __syncthreads();
    return red[0];
}

// Total order used for every top-k / argmax decision: larger value first,
// then lower index.
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

}  // namespace msd
