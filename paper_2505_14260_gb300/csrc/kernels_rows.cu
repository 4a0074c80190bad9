// Row-wise kernels of the MSD step: embedding gather (Eq. 1-3), RMSNorm,
// SwiGLU, RoPE + K/V placement, argmax and top-k with log-softmax.
#include "kernels.h"

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
    embed_rows_kernel<T><<<R, 256, 0, s>>>(E, vis, src, H, x, emb_out, V, status); note_launch();
}

// ---------------------------------------------------------------------------
// RMSNorm: y = x / sqrt(mean(x^2) + eps) * g
// ---------------------------------------------------------------------------
template <typename T>
__global__ void rmsnorm_kernel(const float *__restrict__ x, const T *__restrict__ g, int H,
                               float eps, T *__restrict__ out) {
    __shared__ float red[32];
    const int r = blockIdx.x;
    const float *xr = x + (size_t)r * H;
    float ss = 0.f;
    for (int j = threadIdx.x; j < H; j += blockDim.x) {
        float v = xr[j];
        ss += v * v;
    }
    ss = block_sum(ss, red);
    const float inv = rsqrtf(ss / (float)H + eps);
    for (int j = threadIdx.x; j < H; j += blockDim.x)
        out[(size_t)r * H + j] = from_f<T>(xr[j] * inv * to_f(g[j]));
}

template <typename T>
void launch_rmsnorm(const float *x, const T *g, int R, int H, float eps, T *out,
                    cudaStream_t s) {
    if (R <= 0) return;
    rmsnorm_kernel<T><<<R, 256, 0, s>>>(x, g, H, eps, out); note_launch();
}

// ---------------------------------------------------------------------------
// SwiGLU: silu(gate) * up
// ---------------------------------------------------------------------------
template <typename T>
__global__ void swiglu_kernel(const float *__restrict__ gu, int F, T *__restrict__ act) {
    const int r = blockIdx.y;
    const float *row = gu + (size_t)r * 2 * F;
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < F; j += gridDim.x * blockDim.x) {
        float g = row[j], u = row[F + j];
        float sg = g / (1.f + __expf(-g));
        act[(size_t)r * F + j] = from_f<T>(sg * u);
    }
}

template <typename T>
void launch_swiglu(const float *gu, int R, int F, T *act, cudaStream_t s) {
    if (R <= 0) return;
    dim3 grid((F + 255) / 256, R);
    swiglu_kernel<T><<<grid, 256, 0, s>>>(gu, F, act); note_launch();
}

// ---------------------------------------------------------------------------
// RoPE (rotate-half pairs (i, i + hd/2)) on q and k, and K/V placement.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void rope_kv_kernel(const float *__restrict__ qkv, const RowDesc *__restrict__ rows,
                               int nh, int hd, const float2 *__restrict__ tab, int max_pos,
                               T *__restrict__ q_out, T *__restrict__ kdst, T *__restrict__ vdst,
                               int slots, int *status) {
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
    rope_kv_kernel<T><<<R, 256, 0, s>>>(qkv, rows, nh, hd, rope_tab, max_pos, q_out, kdst,
                                        vdst, slots, status); note_launch();
}

// ---------------------------------------------------------------------------
// Argmax per row (ties: lower index)
// ---------------------------------------------------------------------------
__global__ void argmax_kernel(const float *__restrict__ logits, int V, int *__restrict__ out) {
    __shared__ float sv[32];
    __shared__ int si[32];
    const int r = blockIdx.x;
    const float *z = logits + (size_t)r * V;
    float bv = -INFINITY;
    int bi = 0x7fffffff;
    for (int j = threadIdx.x; j < V; j += blockDim.x) {
        float v = z[j];
        if (better(v, j, bv, bi)) { bv = v; bi = j; }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        float ov = __shfl_xor_sync(0xffffffffu, bv, o);
        int oi = __shfl_xor_sync(0xffffffffu, bi, o);
        if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) { sv[warp] = bv; si[warp] = bi; }
    __syncthreads();
    if (warp == 0) {
        const int nw = blockDim.x >> 5;
        bv = lane < nw ? sv[lane] : -INFINITY;
        bi = lane < nw ? si[lane] : 0x7fffffff;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (better(ov, oi, bv, bi)) { bv = ov; bi = oi; }
        }
        if (lane == 0) out[r] = bi == 0x7fffffff ? 0 : bi;
    }
}

void launch_argmax(const float *logits, int R, int V, int *out, cudaStream_t s) {
    if (R <= 0) return;
    argmax_kernel<<<R, 512, 0, s>>>(logits, V, out); note_launch();
}

// ---------------------------------------------------------------------------
// Top-k + log-softmax per row. Each thread keeps a sorted local top-k of its
// strided elements; k block-wide selection rounds merge them.
// ---------------------------------------------------------------------------
constexpr int TOPK_MAX = 16;
constexpr int TOPK_THREADS = 256;

__global__ void topk_logp_kernel(const float *__restrict__ logits, int V, int k,
                                 int *__restrict__ ids, float *__restrict__ logp) {
    __shared__ float red[32];
    __shared__ float cand_v[TOPK_THREADS];
    __shared__ int cand_i[TOPK_THREADS];
    __shared__ float sel_v[TOPK_MAX];
    __shared__ int sel_i[TOPK_MAX];
    const int r = blockIdx.x;
    const float *z = logits + (size_t)r * V;

    float lv[TOPK_MAX];
    int li[TOPK_MAX];
#pragma unroll
    for (int t = 0; t < TOPK_MAX; ++t) { lv[t] = -INFINITY; li[t] = 0x7fffffff; }
    float mx = -INFINITY;
    for (int j = threadIdx.x; j < V; j += blockDim.x) {
        const float v = z[j];
        mx = fmaxf(mx, v);
        if (better(v, j, lv[k - 1], li[k - 1])) {
            // insert keeping lv sorted (best first); k is small
            int p = k - 1;
            while (p > 0 && better(v, j, lv[p - 1], li[p - 1])) {
                lv[p] = lv[p - 1]; li[p] = li[p - 1];
                --p;
            }
            lv[p] = v; li[p] = j;
        }
    }
    mx = block_max(mx, red);
    float se = 0.f;
    for (int j = threadIdx.x; j < V; j += blockDim.x) se += __expf(z[j] - mx);
    se = block_sum(se, red);
    const float lse = mx + logf(se);

    int head = 0;
    for (int round = 0; round < k; ++round) {
        cand_v[threadIdx.x] = head < k ? lv[head] : -INFINITY;
        cand_i[threadIdx.x] = head < k ? li[head] : 0x7fffffff;
        __syncthreads();
        for (int stride = blockDim.x >> 1; stride > 0; stride >>= 1) {
            if (threadIdx.x < stride) {
                const float ov = cand_v[threadIdx.x + stride];
                const int oi = cand_i[threadIdx.x + stride];
                if (better(ov, oi, cand_v[threadIdx.x], cand_i[threadIdx.x])) {
                    cand_v[threadIdx.x] = ov; cand_i[threadIdx.x] = oi;
                }
            }
            __syncthreads();
        }
        const int win = cand_i[0];
        if (threadIdx.x == 0) { sel_v[round] = cand_v[0]; sel_i[round] = win; }
        if (head < k && li[head] == win) ++head;   // indices are unique per row
        __syncthreads();
    }
    if (threadIdx.x < k) {
        ids[(size_t)r * k + threadIdx.x] = sel_i[threadIdx.x];
        logp[(size_t)r * k + threadIdx.x] = sel_v[threadIdx.x] - lse;
    }
}

void launch_topk_logp(const float *logits, int R, int V, int k, int *ids, float *logp,
                      cudaStream_t s) {
    if (R <= 0) return;
    topk_logp_kernel<<<R, TOPK_THREADS, 0, s>>>(logits, V, k, ids, logp); note_launch();
}

// ---------------------------------------------------------------------------
template <typename T>
__global__ void convert_kernel(const float *__restrict__ x, T *__restrict__ y, long n) {
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < n; i += (long)gridDim.x * blockDim.x)
        y[i] = from_f<T>(x[i]);
}

template <typename T>
void launch_convert(const float *x, T *y, long n, cudaStream_t s) {
    if (n <= 0) return;
    long blocks = (n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    convert_kernel<T><<<(int)blocks, 256, 0, s>>>(x, y, n); note_launch();
}

#define MSD_INST(T)                                                                          \
    template void launch_embed_rows<T>(const T *, const T *, const int *, int, int, float *,  \
                                       T *, int, int *, cudaStream_t);                       \
    template void launch_rmsnorm<T>(const float *, const T *, int, int, float, T *,          \
                                    cudaStream_t);                                           \
    template void launch_swiglu<T>(const float *, int, int, T *, cudaStream_t);              \
    template void launch_rope_kv<T>(const float *, const RowDesc *, int, int, int,           \
                                    const float2 *, int, T *, T *, T *, int, int *,          \
                                    cudaStream_t);                                           \
    template void launch_convert<T>(const float *, T *, long, cudaStream_t);
MSD_INST(float)
MSD_INST(bf16)
#undef MSD_INST

}  // namespace msd
