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
// are visible (after a programmatic launch; a no-op after a plain one). Every
// kernel calls it before it reads anything the previous kernel may have
// written, so that the order holds however it was launched.
__device__ __forceinline__ void wait_prior() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// Launches a short kernel in plain stream order behind the previous one. (With
// programmatic serialization these kernels' griddepcontrol.wait returned
// later than a plain launch starts: measured slower.) The kernel still calls
// wait_prior(), a no-op here, and allow_dependents(), which lets a following
// programmatic launch (the tensor-core GEMMs) start early.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_chain(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                cudaStream_t s, Args &&...args) {
    cudaLaunchConfig_t lc = {};
    lc.gridDim = grid;
    lc.blockDim = block;
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
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
template <typename T> struct Vec4;
template <> struct Vec4<float> {
    static __device__ __forceinline__ float4 load(const float *g) { return *reinterpret_cast<const float4 *>(g); }
    static __device__ __forceinline__ void store(float *o, float4 v) { *reinterpret_cast<float4 *>(o) = v; }
};
template <> struct Vec4<bf16> {
    static __device__ __forceinline__ float4 load(const bf16 *g) {
        const uint2 u = *reinterpret_cast<const uint2 *>(g);
        const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162 *>(&u.x);
        const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162 *>(&u.y);
        return make_float4(__low2float(a), __high2float(a), __low2float(b), __high2float(b));
    }
    static __device__ __forceinline__ void store(bf16 *o, float4 v) {
        __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
        uint2 u;
        u.x = *reinterpret_cast<uint32_t *>(&a);
        u.y = *reinterpret_cast<uint32_t *>(&b);
        *reinterpret_cast<uint2 *>(o) = u;
    }
};

// Split-bf16 operands. Every bf16 activation that feeds a tensor-core product
// (and every K/V cache entry) is kept as a pair hi = bf16(v), lo = bf16(v - hi):
// hi + lo carries v to about 2^-17 relative, so a product of an exact bf16
// weight with the pair (two MMAs into one fp32 accumulator) is as precise as an
// fp32 product. The lo value sits `lo` elements after its hi value (one offset
// for all of a context's bf16 buffers: they are carved from one arena whose
// upper half holds the lo planes); lo = 0 means no lo plane (fp32 contexts,
// caller-owned operands). For T = float the pair is the value itself.
template <typename T> struct Split;
template <> struct Split<float> {
    static __device__ __forceinline__ void store(float *o, long, float v) { *o = v; }
    static __device__ __forceinline__ float load(const float *g, long) { return *g; }
    static __device__ __forceinline__ void store4(float *o, long, float4 v) {
        *reinterpret_cast<float4 *>(o) = v;
    }
    static __device__ __forceinline__ float4 load4(const float *g, long) {
        return *reinterpret_cast<const float4 *>(g);
    }
};
template <> struct Split<bf16> {
    static __device__ __forceinline__ void store(bf16 *o, long lo, float v) {
        const bf16 h = __float2bfloat16_rn(v);
        *o = h;
        if (lo) o[lo] = __float2bfloat16_rn(v - __bfloat162float(h));
    }
    static __device__ __forceinline__ float load(const bf16 *g, long lo) {
        return lo ? __bfloat162float(g[0]) + __bfloat162float(g[lo]) : __bfloat162float(g[0]);
    }
    static __device__ __forceinline__ void store4(bf16 *o, long lo, float4 v) {
        const __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
        uint2 u;
        u.x = *reinterpret_cast<const uint32_t *>(&a);
        u.y = *reinterpret_cast<const uint32_t *>(&b);
        *reinterpret_cast<uint2 *>(o) = u;
        if (lo) {
            const __nv_bfloat162 c = __floats2bfloat162_rn(v.x - __low2float(a), v.y - __high2float(a));
            const __nv_bfloat162 d = __floats2bfloat162_rn(v.z - __low2float(b), v.w - __high2float(b));
            u.x = *reinterpret_cast<const uint32_t *>(&c);
            u.y = *reinterpret_cast<const uint32_t *>(&d);
            *reinterpret_cast<uint2 *>(o + lo) = u;
        }
    }
    static __device__ __forceinline__ float4 load4(const bf16 *g, long lo) {
        float4 h = Vec4<bf16>::load(g);
        if (lo) {
            const float4 l = Vec4<bf16>::load(g + lo);
            h.x += l.x; h.y += l.y; h.z += l.z; h.w += l.w;
        }
        return h;
    }
};

// Row copies of the small per-row kernels, n a multiple of 4 and rows 4-element
// aligned: every thread of the CTA requests up to 4 groups of 4 elements (16-
// or 8-byte accesses) before it stores any, so one pass costs about one memory
// round trip instead of one per element.
template <typename TD, typename TS>
__device__ __forceinline__ void copy_row(TD *__restrict__ dst, const TS *__restrict__ src, int n) {
    const int n4 = n >> 2;
    for (int g0 = threadIdx.x; g0 < n4; g0 += 4 * blockDim.x) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) v[u] = Vec4<TS>::load(src + 4 * g);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) Vec4<TD>::store(dst + 4 * g, v[u]);
        }
    }
}

// One source row to two destinations (d2 nullable).
template <typename TD1, typename TD2, typename TS>
__device__ __forceinline__ void copy_row_2dst(TD1 *__restrict__ d1, TD2 *__restrict__ d2,
                                              const TS *__restrict__ src, int n) {
    const int n4 = n >> 2;
    for (int g0 = threadIdx.x; g0 < n4; g0 += 4 * blockDim.x) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) v[u] = Vec4<TS>::load(src + 4 * g);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) {
                Vec4<TD1>::store(d1 + 4 * g, v[u]);
                if (d2) Vec4<TD2>::store(d2 + 4 * g, v[u]);
            }
        }
    }
}

// Two independent row copies in one pass (s1 null: d1 gets zeros).
template <typename TD1, typename TS1, typename TD2, typename TS2>
__device__ __forceinline__ void copy_rows2(TD1 *__restrict__ d1, const TS1 *__restrict__ s1,
                                           TD2 *__restrict__ d2, const TS2 *__restrict__ s2, int n) {
    const int n4 = n >> 2;
    for (int g0 = threadIdx.x; g0 < n4; g0 += 2 * blockDim.x) {
        float4 a[2], b[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) {
                a[u] = s1 ? Vec4<TS1>::load(s1 + 4 * g) : make_float4(0.f, 0.f, 0.f, 0.f);
                b[u] = Vec4<TS2>::load(s2 + 4 * g);
            }
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) {
                Vec4<TD1>::store(d1 + 4 * g, a[u]);
                Vec4<TD2>::store(d2 + 4 * g, b[u]);
            }
        }
    }
}

// Row copy between split buffers (source lo plane at slo, destination at dlo;
// 0 = none): the pair's sum is re-split, so an exact bf16 source gets lo = 0.
template <typename TD, typename TS>
__device__ __forceinline__ void copy_row_split(TD *__restrict__ dst, long dlo, const TS *__restrict__ src,
                                               long slo, int n) {
    const int n4 = n >> 2;
    for (int g0 = threadIdx.x; g0 < n4; g0 += 4 * blockDim.x) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) v[u] = Split<TS>::load4(src + 4 * g, slo);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) Split<TD>::store4(dst + 4 * g, dlo, v[u]);
        }
    }
}

// One fp32 source row to an fp32 row (d1, nullable) and a split row (d2, lo
// plane at dlo).
template <typename TD2>
__device__ __forceinline__ void copy_row_2dst_split(float *__restrict__ d1, TD2 *__restrict__ d2, long dlo,
                                                    const float *__restrict__ src, int n) {
    const int n4 = n >> 2;
    for (int g0 = threadIdx.x; g0 < n4; g0 += 4 * blockDim.x) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) v[u] = *reinterpret_cast<const float4 *>(src + 4 * g);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) {
                if (d1) *reinterpret_cast<float4 *>(d1 + 4 * g) = v[u];
                Split<TD2>::store4(d2 + 4 * g, dlo, v[u]);
            }
        }
    }
}

// Two row copies in one pass into split rows (lo planes at dlo): d1 <- s1 (a
// split source with lo plane at s1lo, or fp32; null: zeros), d2 <- s2 (read
// as its hi values alone: exact bf16 embeddings).
template <typename TD, typename TS1, typename TS2>
__device__ __forceinline__ void copy_rows2_split(TD *__restrict__ d1, const TS1 *__restrict__ s1, long s1lo,
                                                 TD *__restrict__ d2, const TS2 *__restrict__ s2, int n,
                                                 long dlo) {
    const int n4 = n >> 2;
    for (int g0 = threadIdx.x; g0 < n4; g0 += 2 * blockDim.x) {
        float4 a[2], b[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) {
                a[u] = s1 ? Split<TS1>::load4(s1 + 4 * g, s1lo) : make_float4(0.f, 0.f, 0.f, 0.f);
                b[u] = Vec4<TS2>::load(s2 + 4 * g);
            }
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int g = g0 + u * blockDim.x;
            if (g < n4) {
                Split<TD>::store4(d1 + 4 * g, dlo, a[u]);
                Split<TD>::store4(d2 + 4 * g, dlo, b[u]);
            }
        }
    }
}

__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
    return va > vb || (va == vb && ia < ib);
}

}  // namespace msd
