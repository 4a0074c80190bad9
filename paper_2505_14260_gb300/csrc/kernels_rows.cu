// Row-wise kernels of the MSD step: embedding gather (Eq. 1-3), RMSNorm,
// SwiGLU, RoPE + K/V placement, argmax and top-k with log-softmax.
#include "kernels.h"

#include <algorithm>
#include <atomic>

namespace msd {

static std::atomic<long> g_launches{0};
long launch_count() { return g_launches.load(std::memory_order_relaxed); }
void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

// ---------------------------------------------------------------------------
// Embedding gather (Eq. 1 for text, Eq. 2's projected rows for visual slots)
// ---------------------------------------------------------------------------
template <typename T>
__global__ void embed_rows_kernel(const T *__restrict__ E, const T *__restrict__ vis,
                                  const int *__restrict__ src, int H, float *__restrict__ x,
                                  T *__restrict__ emb_out, int V, int *status) {
    allow_dependents();
    wait_prior();
    const int r = blockIdx.x;
    int s = src[r];
    const T *row;
    if (s >= 0) {
        if (s >= V) {
            if (threadIdx.x == 0) set_status(status, ST_BAD_TOKEN);
            s = 0;
        }
        row = E + (size_t)s * H;
    } else {
        row = vis + (size_t)(-1 - s) * H;
    }
    for (int j = threadIdx.x; j < H; j += blockDim.x) {
        T v = row[j];
        x[(size_t)r * H + j] = to_f(v);
        if (emb_out) emb_out[(size_t)r * H + j] = v;
    }
}

template <typename T>
void launch_embed_rows(const T *E, const T *vis, const int *src, int R, int H, float *x,
                       T *emb_out, int V, int *status, cudaStream_t s) {
    if (R <= 0) return;
    launch_pdl(embed_rows_kernel<T>, R, 256, 0, s, E, vis, src, H, x, emb_out, V, status); note_launch();
}

// ---------------------------------------------------------------------------
// RMSNorm: y = x / sqrt(mean(x^2) + eps) * g
// ---------------------------------------------------------------------------
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

// One CTA per row; the row stays in registers (H <= 8 * 4 * 256).
constexpr int RMS_THREADS = 256;
constexpr int RMS_VEC = 8;

template <typename T>
__global__ void __launch_bounds__(RMS_THREADS) rmsnorm_kernel(const float *__restrict__ x,
                                                              const T *__restrict__ g, int H,
                                                              float eps, T *__restrict__ out) {
    allow_dependents();
    wait_prior();
    __shared__ float red[32];
    const int r = blockIdx.x, n4 = H >> 2;
    const float4 *xr = reinterpret_cast<const float4 *>(x + (size_t)r * H);
    float4 v[RMS_VEC];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < RMS_VEC; ++i) {
        const int j = threadIdx.x + i * RMS_THREADS;
        v[i] = j < n4 ? xr[j] : make_float4(0.f, 0.f, 0.f, 0.f);
        ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
    }
    ss = block_sum(ss, red);
    const float inv = rsqrtf(ss / (float)H + eps);
#pragma unroll
    for (int i = 0; i < RMS_VEC; ++i) {
        const int j = threadIdx.x + i * RMS_THREADS;
        if (j < n4) {
            const float4 gg = Vec4<T>::load(g + 4 * j);
            Vec4<T>::store(out + (size_t)r * H + 4 * j,
                           make_float4(v[i].x * inv * gg.x, v[i].y * inv * gg.y,
                                       v[i].z * inv * gg.z, v[i].w * inv * gg.w));
        }
    }
}

template <typename T>
void launch_rmsnorm(const float *x, const T *g, int R, int H, float eps, T *out,
                    cudaStream_t s) {
    if (R <= 0) return;
    launch_pdl(rmsnorm_kernel<T>, R, RMS_THREADS, 0, s, x, g, H, eps, out); note_launch();
}

// ---------------------------------------------------------------------------
// SwiGLU: silu(gate) * up
// ---------------------------------------------------------------------------
template <typename T>
__global__ void swiglu_kernel(const float *__restrict__ gu, int F, int glu, T *__restrict__ act) {
    allow_dependents();
    wait_prior();
    const int r = blockIdx.y;
    const int ld = glu ? 128 * ((F + 63) / 64) : 2 * F;
    const float *row = gu + (size_t)r * ld;
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < F; j += gridDim.x * blockDim.x) {
        const int gi = glu ? ((j >> 6) << 7) + (j & 63) : j;
        const float g = row[gi], u = row[gi + (glu ? 64 : F)];
        const float sg = g / (1.f + __expf(-g));
        act[(size_t)r * F + j] = from_f<T>(sg * u);
    }
}

template <typename T>
void launch_swiglu(const float *gu, int R, int F, bool glu, T *act, cudaStream_t s) {
    if (R <= 0) return;
    dim3 grid((F + 255) / 256, R);
    launch_pdl(swiglu_kernel<T>, grid, 256, 0, s, gu, F, glu ? 1 : 0, act); note_launch();
}

// ---------------------------------------------------------------------------
// RoPE (rotate-half pairs (i, i + hd/2)) on q and k, and K/V placement.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void rope_kv_kernel(const float *__restrict__ qkv, const RowDesc *__restrict__ rows,
                               int nh, int hd, const float2 *__restrict__ tab, int max_pos,
                               T *__restrict__ q_out, T *__restrict__ kdst, T *__restrict__ vdst,
                               int slots, int *status) {
    allow_dependents();
    wait_prior();
    const int r = blockIdx.x;
    const int H = nh * hd, half = hd >> 1;
    const RowDesc d = rows[r];
    int pos = d.pos;
    if (pos < 0 || pos >= max_pos) {
        if (threadIdx.x == 0) set_status(status, ST_RANGE);
        pos = 0;
    }
    const bool write_kv = d.dst >= 0 && d.dst < slots;
    if (d.dst >= slots && threadIdx.x == 0) set_status(status, ST_RANGE);
    const float *q = qkv + (size_t)r * 3 * H;
    const float *k = q + H;
    const float *v = q + 2 * H;
    const float2 *cs = tab + (size_t)pos * half;
    for (int t = threadIdx.x; t < nh * half; t += blockDim.x) {
        const int h = t / half, i = t - h * half;
        const float2 c = cs[i];
        const int a = h * hd + i, b = a + half;
        const float qa = q[a], qb = q[b];
        q_out[(size_t)r * H + a] = from_f<T>(qa * c.x - qb * c.y);
        q_out[(size_t)r * H + b] = from_f<T>(qb * c.x + qa * c.y);
        if (write_kv) {
            const float ka = k[a], kb = k[b];
            const size_t base = ((size_t)(d.req * nh + h) * slots + d.dst) * hd;
            kdst[base + i] = from_f<T>(ka * c.x - kb * c.y);
            kdst[base + i + half] = from_f<T>(kb * c.x + ka * c.y);
            vdst[base + i] = from_f<T>(v[a]);
            vdst[base + i + half] = from_f<T>(v[b]);
        }
    }
}

template <typename T>
void launch_rope_kv(const float *qkv, const RowDesc *rows, int R, int nh, int hd,
                    const float2 *rope_tab, int max_pos, T *q_out, T *kdst, T *vdst,
                    int slots, int *status, cudaStream_t s) {
    if (R <= 0) return;
    launch_pdl(rope_kv_kernel<T>, R, 256, 0, s, qkv, rows, nh, hd, rope_tab, max_pos, q_out, kdst,
                                        vdst, slots, status); note_launch();
}

// ---------------------------------------------------------------------------
// Top-k per row with log-softmax values (argmax = top-1). The row is cut into
// chunks, one CTA each: the CTA holds its chunk in shared memory, computes the
// chunk max, the chunk sum of exp(z - max) and the chunk's top-k (k rounds of
// a block-wide best-of with removal); the last CTA of the row (ticket) merges
// the chunk results: lse = M + log(sum_c s_c exp(m_c - M)) and the top-k of the
// chunk candidates. Order: larger value, then lower index.
// ---------------------------------------------------------------------------
constexpr int TOPK_MAX = 16;
constexpr int TK_THREADS = 256;
constexpr int TK_REC = 2 + 2 * TOPK_MAX;     // floats per chunk record

__device__ __forceinline__ void block_best(float &v, int &i, float *rv, int *ri) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, v, o);
        const int oi = __shfl_xor_sync(0xffffffffu, i, o);
        if (better(ov, oi, v, i)) { v = ov; i = oi; }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) { rv[warp] = v; ri[warp] = i; }
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        v = lane < nw ? rv[lane] : -INFINITY;
        i = lane < nw ? ri[lane] : 0x7fffffff;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, v, o);
            const int oi = __shfl_xor_sync(0xffffffffu, i, o);
            if (better(ov, oi, v, i)) { v = ov; i = oi; }
        }
        if (lane == 0) { rv[0] = v; ri[0] = i; }
    }
    __syncthreads();
    v = rv[0];
    i = ri[0];
}

__global__ void __launch_bounds__(TK_THREADS)
    topk_rows_kernel(const float *__restrict__ logits, int V, int k, int *__restrict__ ids,
                     float *__restrict__ logp, float *__restrict__ ws, int *__restrict__ counters) {
    allow_dependents();
    wait_prior();
    extern __shared__ float sv[];
    __shared__ float rv[32];
    __shared__ int ri[32];
    __shared__ float sel_v[TOPK_MAX];
    __shared__ int sel_i[TOPK_MAX];
    __shared__ int s_last;
    const int r = blockIdx.y, c = blockIdx.x, nc = gridDim.x;
    const int CH = (V + nc - 1) / nc;
    const int lo = c * CH, n = max(0, min(V, lo + CH) - lo);
    const float *z = logits + (size_t)r * V + lo;
    float mx = -INFINITY;
    for (int j = threadIdx.x; j < n; j += TK_THREADS) {
        const float v = z[j];
        sv[j] = v;
        mx = fmaxf(mx, v);
    }
    mx = block_max(mx, rv);
    float se = 0.f;
    for (int j = threadIdx.x; j < n; j += TK_THREADS) se += __expf(sv[j] - mx);
    se = block_sum(se, rv);
    for (int t = 0; t < k; ++t) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        for (int j = threadIdx.x; j < n; j += TK_THREADS)
            if (better(sv[j], lo + j, bv, bi)) { bv = sv[j]; bi = lo + j; }
        block_best(bv, bi, rv, ri);
        if (threadIdx.x == 0) { sel_v[t] = bv; sel_i[t] = bi; }
        if (bi != 0x7fffffff && bi - lo >= 0 && bi - lo < n && ((bi - lo) % TK_THREADS) == threadIdx.x)
            sv[bi - lo] = -INFINITY;
        __syncthreads();
    }
    float *rec = ws + ((size_t)r * nc + c) * TK_REC;
    if (threadIdx.x == 0) { rec[0] = mx; rec[1] = se; }
    if (threadIdx.x < k) {
        rec[2 + threadIdx.x] = sel_v[threadIdx.x];
        rec[2 + TOPK_MAX + threadIdx.x] = __int_as_float(sel_i[threadIdx.x]);
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(&counters[r], 1) == nc - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    // merge the chunk records of row r
    const float *rrow = ws + (size_t)r * nc * TK_REC;
    float M = -INFINITY;
    for (int q = threadIdx.x; q < nc; q += TK_THREADS) M = fmaxf(M, __ldcg(rrow + q * TK_REC));
    M = block_max(M, rv);
    float S = 0.f;
    for (int q = threadIdx.x; q < nc; q += TK_THREADS)
        S += __ldcg(rrow + q * TK_REC + 1) * __expf(__ldcg(rrow + q * TK_REC) - M);
    S = block_sum(S, rv);
    const float lse = M + logf(S);
    float *cv = sv;                                   // candidates: nc * k
    int *ci = reinterpret_cast<int *>(sv + nc * k);
    for (int q = threadIdx.x; q < nc * k; q += TK_THREADS) {
        const int cc = q / k, t = q - cc * k;
        cv[q] = __ldcg(rrow + cc * TK_REC + 2 + t);
        ci[q] = __float_as_int(__ldcg(rrow + cc * TK_REC + 2 + TOPK_MAX + t));
    }
    __syncthreads();
    for (int t = 0; t < k; ++t) {
        float bv = -INFINITY;
        int bi = 0x7fffffff, bq = -1;
        for (int q = threadIdx.x; q < nc * k; q += TK_THREADS)
            if (better(cv[q], ci[q], bv, bi)) { bv = cv[q]; bi = ci[q]; bq = q; }
        float wv = bv;
        int wi = bi;
        block_best(wv, wi, rv, ri);
        if (bq >= 0 && bi == wi) cv[bq] = -INFINITY;   // ids are unique within a row
        if (threadIdx.x == 0) {
            ids[(size_t)r * k + t] = wi == 0x7fffffff ? 0 : wi;
            if (logp) logp[(size_t)r * k + t] = wv - lse;
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) counters[r] = 0;
}

static int topk_chunks(int V) {
    int nc = 16;
    while ((V + nc - 1) / nc > 4096) nc *= 2;
    return nc;
}

size_t topk_scratch_floats(int max_rows, int V) {
    return (size_t)max_rows * topk_chunks(V) * TK_REC;
}

void launch_topk_logp(const float *logits, int R, int V, int k, int *ids, float *logp,
                      const TopkScratch &sc, cudaStream_t s) {
    if (R <= 0) return;
    const int nc = topk_chunks(V);
    const int CH = (V + nc - 1) / nc;
    const size_t smem = sizeof(float) * std::max<size_t>(CH, (size_t)2 * nc * k);
    launch_pdl(topk_rows_kernel, dim3(nc, R), TK_THREADS, smem, s, logits, V, k, ids, logp, sc.ws,
                                                          sc.counters);
    note_launch();
}

void launch_argmax(const float *logits, int R, int V, int *out, const TopkScratch &sc,
                   cudaStream_t s) {
    launch_topk_logp(logits, R, V, 1, out, nullptr, sc, s);
}

// ---------------------------------------------------------------------------
template <typename T>
__global__ void convert_kernel(const float *__restrict__ x, T *__restrict__ y, long n) {
    wait_prior();
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x)
        y[i] = from_f<T>(x[i]);
}

template <typename T>
void launch_convert(const float *x, T *y, long n, cudaStream_t s) {
    if (n <= 0) return;
    long blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    launch_pdl(convert_kernel<T>, (int)blocks, 256, 0, s, x, y, n); note_launch();
}

__global__ void flag_status_kernel(int *status, int code) { wait_prior(); set_status(status, code); }

void launch_flag(int *status, int code, cudaStream_t s) {
    cudaGetLastError();
    launch_pdl(flag_status_kernel, 1, 1, 0, s, status, code);
    note_launch();
}

#define MSD_INST(T)                                                                          \
    template void launch_embed_rows<T>(const T *, const T *, const int *, int, int, float *,  \
                                       T *, int, int *, cudaStream_t);                       \
    template void launch_rmsnorm<T>(const float *, const T *, int, int, float, T *,          \
                                    cudaStream_t);                                           \
    template void launch_swiglu<T>(const float *, int, int, bool, T *, cudaStream_t);              \
    template void launch_rope_kv<T>(const float *, const RowDesc *, int, int, int,           \
                                    const float2 *, int, T *, T *, T *, int, int *,          \
                                    cudaStream_t);                                           \
    template void launch_convert<T>(const float *, T *, long, cudaStream_t);
MSD_INST(float)
MSD_INST(bf16)
#undef MSD_INST

}  // namespace msd
