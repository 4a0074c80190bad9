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
    wait_prior();
    allow_dependents();
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
    copy_row_2dst(x + (size_t)r * H, emb_out ? emb_out + (size_t)r * H : nullptr, row, H);
}

template <typename T>
void launch_embed_rows(const T *E, const T *vis, const int *src, int R, int H, float *x,
                       T *emb_out, int V, int *status, cudaStream_t s) {
    if (R <= 0) return;
    launch_chain(embed_rows_kernel<T>, R, 256, 0, s, E, vis, src, H, x, emb_out, V, status); note_launch();
}

// ---------------------------------------------------------------------------
// RMSNorm: y = x / sqrt(mean(x^2) + eps) * g
// ---------------------------------------------------------------------------
// One CTA per row; the row stays in registers (H <= 8 * 4 * 256).
constexpr int RMS_THREADS = 256;
constexpr int RMS_VEC = 8;

template <typename T>
__global__ void __launch_bounds__(RMS_THREADS) rmsnorm_kernel(const float *__restrict__ x,
                                                              const T *__restrict__ g, int H,
                                                              float eps, T *__restrict__ out, long lo) {
    wait_prior();
    allow_dependents();
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
            Split<T>::store4(out + (size_t)r * H + 4 * j, lo,
                             make_float4(v[i].x * inv * gg.x, v[i].y * inv * gg.y,
                                         v[i].z * inv * gg.z, v[i].w * inv * gg.w));
        }
    }
}

template <typename T>
void launch_rmsnorm(const float *x, const T *g, int R, int H, float eps, T *out, long lo,
                    cudaStream_t s) {
    if (R <= 0) return;
    launch_chain(rmsnorm_kernel<T>, R, RMS_THREADS, 0, s, x, g, H, eps, out, lo); note_launch();
}

// ---------------------------------------------------------------------------
// SwiGLU: silu(gate) * up
// ---------------------------------------------------------------------------
template <typename T>
__global__ void swiglu_kernel(const float *__restrict__ gu, int F, int glu, T *__restrict__ act, long lo) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.y;
    const int ld = glu ? 128 * ((F + 63) / 64) : 2 * F;
    const float *row = gu + (size_t)r * ld;
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < F; j += gridDim.x * blockDim.x) {
        const int gi = glu ? ((j >> 6) << 7) + (j & 63) : j;
        const float g = row[gi], u = row[gi + (glu ? 64 : F)];
        const float sg = g / (1.f + __expf(-g));
        Split<T>::store(act + (size_t)r * F + j, lo, sg * u);
    }
}

template <typename T>
void launch_swiglu(const float *gu, int R, int F, bool glu, T *act, long lo, cudaStream_t s) {
    if (R <= 0) return;
    dim3 grid((F + 255) / 256, R);
    launch_chain(swiglu_kernel<T>, grid, 256, 0, s, gu, F, glu ? 1 : 0, act, lo); note_launch();
}

// ---------------------------------------------------------------------------
// RoPE (rotate-half pairs (i, i + hd/2)) on q and k, and K/V placement.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void rope_kv_kernel(const float *__restrict__ qkv, const RowDesc *__restrict__ rows,
                               int nh, int hd, const float2 *__restrict__ tab, int max_pos,
                               T *__restrict__ q_out, T *__restrict__ kdst, T *__restrict__ vdst,
                               int slots, long lo, int *status) {
    wait_prior();
    allow_dependents();
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
        Split<T>::store(q_out + (size_t)r * H + a, lo, qa * c.x - qb * c.y);
        Split<T>::store(q_out + (size_t)r * H + b, lo, qb * c.x + qa * c.y);
        if (write_kv) {
            const float ka = k[a], kb = k[b];
            const size_t base = ((size_t)(d.req * nh + h) * slots + d.dst) * hd;
            Split<T>::store(kdst + base + i, lo, ka * c.x - kb * c.y);
            Split<T>::store(kdst + base + i + half, lo, kb * c.x + ka * c.y);
            Split<T>::store(vdst + base + i, lo, v[a]);
            Split<T>::store(vdst + base + i + half, lo, v[b]);
        }
    }
}

template <typename T>
void launch_rope_kv(const float *qkv, const RowDesc *rows, int R, int nh, int hd,
                    const float2 *rope_tab, int max_pos, T *q_out, T *kdst, T *vdst,
                    int slots, long lo, int *status, cudaStream_t s) {
    if (R <= 0) return;
    launch_chain(rope_kv_kernel<T>, R, 256, 0, s, qkv, rows, nh, hd, rope_tab, max_pos, q_out, kdst,
                                        vdst, slots, lo, status); note_launch();
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
constexpr int TK_EPT = 16;                         // logits per thread
constexpr int TK_CHUNK = TK_THREADS * TK_EPT;      // logits per CTA
constexpr int TK_REC = 2 + 2 * TOPK_MAX;           // floats per chunk record
constexpr int TK_NONE = 0x7fffffff;                // index of an empty slot
constexpr int TK_MERGE_SLOTS = 8;                  // row merge: nc * k <= 32 * 8 candidates

// (max, sum of exp(x - max)) pairs combined exactly
__device__ __forceinline__ void lse_combine(float &m, float &s, float om, float os) {
    const float nm = fmaxf(m, om);
    if (nm == -INFINITY) return;
    s = s * __expf(m - nm) + os * __expf(om - nm);
    m = nm;
}

__device__ __forceinline__ void warp_lse(float &m, float &s) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float om = __shfl_xor_sync(0xffffffffu, m, o), os = __shfl_xor_sync(0xffffffffu, s, o);
        lse_combine(m, s, om, os);
    }
}

// Order-preserving 32-bit key of a logit: larger value, larger key; -0 as +0
// and NaN lowest, as in better().
__device__ __forceinline__ unsigned tk_key(float v) {
    if (v != v) return 0u;
    const unsigned u = __float_as_uint(v == 0.f ? 0.f : v);
    return u ^ ((u >> 31) ? 0xffffffffu : 0x80000000u);
}
__device__ __forceinline__ float tk_value(unsigned key) {
    return __uint_as_float(key ^ ((key >> 31) ? 0x80000000u : 0xffffffffu));
}

// Top-k of the NS (value, index) slots held by each lane of a warp, in k
// rounds: every lane keeps its best remaining slot (its head); a round takes
// the warp's best head with two single-instruction warp reductions (largest
// key, then lowest index among the lanes holding it), and only the winning
// lane retires that slot (by index: indices are unique, so no slot is indexed
// dynamically) and rescans for its next head. Lane 0 gets the result.
template <int NS>
__device__ __forceinline__ void warp_topk_rounds(float (&v)[NS], int (&ix)[NS], int k, float *out_v,
                                                 int *out_i) {
    float hv = -INFINITY;
    int hi = TK_NONE;
#pragma unroll
    for (int e = 0; e < NS; ++e)
        if (better(v[e], ix[e], hv, hi)) { hv = v[e]; hi = ix[e]; }
    for (int t = 0; t < k; ++t) {
        const unsigned hk = tk_key(hv);
        const unsigned mk = __reduce_max_sync(0xffffffffu, hk);
        const unsigned mi = __reduce_min_sync(0xffffffffu, hk == mk ? (unsigned)hi : 0xffffffffu);
        if ((threadIdx.x & 31) == 0) { out_v[t] = tk_value(mk); out_i[t] = (int)mi; }
        if (hk == mk && (unsigned)hi == mi) {
#pragma unroll
            for (int e = 0; e < NS; ++e)
                if (ix[e] == hi) { v[e] = -INFINITY; ix[e] = TK_NONE; }
            hv = -INFINITY;
            hi = TK_NONE;
#pragma unroll
            for (int e = 0; e < NS; ++e)
                if (better(v[e], ix[e], hv, hi)) { hv = v[e]; hi = ix[e]; }
        }
        __syncwarp();
    }
}

// Top-k of a warp's NS slots per lane by threshold and rank. The k-th best of
// the 32 lane heads (ranked by counting) is a threshold that at least k slots
// reach; the slots that reach it (NaN and empty slots never do) are compacted
// into the warp's 32-entry scratch and each ranked by counting how many beat
// it, so no step is repeated k times. More than 32 such slots (heavy ties)
// falls back to warp_topk_rounds. The result is the same ordered list as
// warp_topk_rounds: larger value first, then lower index; (-inf, TK_NONE)
// fills the places beyond the valid slots. Written by the lanes that own a
// place; the caller synchronises the warp before reading it.
template <int NS>
__device__ __forceinline__ void warp_topk(float (&v)[NS], int (&ix)[NS], int k, float *out_v, int *out_i,
                                          float *scr_v, int *scr_i) {
    const int lane = threadIdx.x & 31;
    float hv = -INFINITY;
    int hi = TK_NONE;
#pragma unroll
    for (int e = 0; e < NS; ++e)
        if (better(v[e], ix[e], hv, hi)) { hv = v[e]; hi = ix[e]; }
    // rank of this lane's head among the 32 heads
    int hr = 0;
#pragma unroll 8
    for (int j = 0; j < 32; ++j) {
        const float ov = __shfl_sync(0xffffffffu, hv, j);
        const int oi = __shfl_sync(0xffffffffu, hi, j);
        hr += better(ov, oi, hv, hi);
    }
    // threshold = the k-th best head (or no threshold if fewer than k lanes hold a slot)
    const unsigned at_k = __ballot_sync(0xffffffffu, hr == k - 1 && hi != TK_NONE);
    const int src = at_k ? __ffs(at_k) - 1 : 0;
    const float tv = __shfl_sync(0xffffffffu, hv, src);
    const int ti = at_k ? __shfl_sync(0xffffffffu, hi, src) : TK_NONE;
    int cnt = 0;
#pragma unroll
    for (int e = 0; e < NS; ++e)
        cnt += ix[e] != TK_NONE && v[e] == v[e] && (ti == TK_NONE || !better(tv, ti, v[e], ix[e]));
    int off = cnt;                                   // inclusive prefix over lanes
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, off, o);
        if (lane >= o) off += y;
    }
    const int total = __shfl_sync(0xffffffffu, off, 31);
    if (total > 32) {
        warp_topk_rounds<NS>(v, ix, k, out_v, out_i);
        return;
    }
    off -= cnt;
#pragma unroll
    for (int e = 0; e < NS; ++e)
        if (ix[e] != TK_NONE && v[e] == v[e] && (ti == TK_NONE || !better(tv, ti, v[e], ix[e]))) {
            scr_v[off] = v[e];
            scr_i[off] = ix[e];
            ++off;
        }
    __syncwarp();
    if (lane < total) {
        const float cv = scr_v[lane];
        const int ci = scr_i[lane];
        int r = 0;
        for (int j = 0; j < total; ++j) r += better(scr_v[j], scr_i[j], cv, ci);
        if (r < k) { out_v[r] = cv; out_i[r] = ci; }
    } else if (lane < k) {
        out_v[lane] = -INFINITY;
        out_i[lane] = TK_NONE;
    }
    __syncwarp();
}

// Per row: chunks of TK_CHUNK logits, one CTA each. Each warp takes the top-k
// of its 512 logits and their (max, sum exp); one warp merges the CTA's warps,
// and the row's last CTA (ticket) merges the chunks; log-probabilities are
// logit - logsumexp.
__global__ void __launch_bounds__(TK_THREADS)
    topk_rows_kernel(const float *__restrict__ logits, int V, int k, int *__restrict__ ids,
                     float *__restrict__ logp, float *__restrict__ ws, int *__restrict__ counters) {
    wait_prior();
    allow_dependents();
    constexpr int NW = TK_THREADS / 32;
    __shared__ float s_v[NW * TOPK_MAX];
    __shared__ int s_i[NW * TOPK_MAX];
    __shared__ float s_m[NW], s_s[NW];
    __shared__ float s_cv[NW * 32];         // per-warp compaction scratch of warp_topk
    __shared__ int s_ci[NW * 32];
    __shared__ int s_last;
    const int r = blockIdx.y, c = blockIdx.x, nc = gridDim.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int lo = c * TK_CHUNK + warp * (32 * TK_EPT);       // this warp's 512 logits
    const float *z = logits + (size_t)r * V;
    float x[TK_EPT];
    int xi[TK_EPT];
#pragma unroll
    for (int e = 0; e < TK_EPT; ++e) {
        const int j = lo + lane + e * 32;
        x[e] = j < V ? z[j] : -INFINITY;
        xi[e] = j < V ? j : TK_NONE;
    }
    float m = -INFINITY, sum = 0.f;
#pragma unroll
    for (int e = 0; e < TK_EPT; ++e) m = fmaxf(m, x[e]);
#pragma unroll
    for (int e = 0; e < TK_EPT; ++e)
        if (xi[e] != TK_NONE) sum += __expf(x[e] - m);
    warp_lse(m, sum);
    warp_topk<TK_EPT>(x, xi, k, s_v + warp * TOPK_MAX, s_i + warp * TOPK_MAX, s_cv + warp * 32, s_ci + warp * 32);
    if (lane == 0) { s_m[warp] = m; s_s[warp] = sum; }
    __syncthreads();
    float *rec = ws + ((size_t)r * nc + c) * TK_REC;
    if (warp == 0) {
        // the NW warps' k candidates, NW * TOPK_MAX / 32 slots per lane
        constexpr int NS = NW * TOPK_MAX / 32;
        float cv[NS];
        int ci[NS];
#pragma unroll
        for (int e = 0; e < NS; ++e) {
            const int q = lane + e * 32, w = q / TOPK_MAX, t = q - w * TOPK_MAX;
            cv[e] = t < k ? s_v[q] : -INFINITY;
            ci[e] = t < k ? s_i[q] : TK_NONE;
        }
        m = lane < NW ? s_m[lane] : -INFINITY;
        sum = lane < NW ? s_s[lane] : 0.f;
        warp_lse(m, sum);
        if (lane == 0) { rec[0] = m; rec[1] = sum; }
        __syncwarp();                      // the candidates are in registers: reuse s_v / s_i
        warp_topk<NS>(cv, ci, k, s_v, s_i, s_cv, s_ci);
        __syncwarp();
        if (lane < k) {
            rec[2 + lane] = s_v[lane];
            rec[2 + TOPK_MAX + lane] = __int_as_float(s_i[lane]);
        }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(&counters[r], 1) == nc - 1;
    __syncthreads();
    if (!s_last || warp != 0) return;
    __threadfence();
    // merge the row's chunk records: nc * k candidates, TK_MERGE_SLOTS per lane
    const float *rrow = ws + (size_t)r * nc * TK_REC;
    float cv[TK_MERGE_SLOTS];
    int ci[TK_MERGE_SLOTS];
#pragma unroll
    for (int e = 0; e < TK_MERGE_SLOTS; ++e) {
        const int q = lane + e * 32, cc = q / k, t = q - cc * k;
        const bool have = cc < nc;
        cv[e] = have ? __ldcg(rrow + cc * TK_REC + 2 + t) : -INFINITY;
        ci[e] = have ? __float_as_int(__ldcg(rrow + cc * TK_REC + 2 + TOPK_MAX + t)) : TK_NONE;
    }
    m = -INFINITY;
    sum = 0.f;
    for (int q = lane; q < nc; q += 32)
        lse_combine(m, sum, __ldcg(rrow + q * TK_REC), __ldcg(rrow + q * TK_REC + 1));
    warp_lse(m, sum);
    const float lse = m + logf(sum);
    warp_topk<TK_MERGE_SLOTS>(cv, ci, k, s_v, s_i, s_cv, s_ci);
    __syncwarp();
    if (lane < k) {
        ids[(size_t)r * k + lane] = s_i[lane] == TK_NONE ? 0 : s_i[lane];
        if (logp) logp[(size_t)r * k + lane] = s_v[lane] - lse;
    }
    if (lane == 0) counters[r] = 0;
}

static int topk_chunks(int V) { return (V + TK_CHUNK - 1) / TK_CHUNK; }

size_t topk_scratch_floats(int max_rows, int V) {
    return (size_t)max_rows * topk_chunks(V) * TK_REC;
}

void launch_topk_logp(const float *logits, int R, int V, int k, int *ids, float *logp,
                      const TopkScratch &sc, cudaStream_t s) {
    if (R <= 0 || k < 1 || k > TOPK_MAX) return;
    const int nc = topk_chunks(V);
    if (nc * k > 32 * TK_MERGE_SLOTS) return;            // refused at msd_create
    launch_chain(topk_rows_kernel, dim3(nc, R), TK_THREADS, 0, s, logits, V, k, ids, logp, sc.ws,
               sc.counters);
    note_launch();
}

bool topk_supported(int V, int k) {
    return k >= 1 && k <= TOPK_MAX && topk_chunks(V) * k <= 32 * TK_MERGE_SLOTS;
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
    launch_chain(convert_kernel<T>, (int)blocks, 256, 0, s, x, y, n); note_launch();
}

__global__ void flag_status_kernel(int *status, int code) { wait_prior(); set_status(status, code); }

void launch_flag(int *status, int code, cudaStream_t s) {
    cudaGetLastError();
    launch_chain(flag_status_kernel, 1, 1, 0, s, status, code);
    note_launch();
}

#define MSD_INST(T)                                                                          \
    template void launch_embed_rows<T>(const T *, const T *, const int *, int, int, float *,  \
                                       T *, int, int *, cudaStream_t);                       \
    template void launch_rmsnorm<T>(const float *, const T *, int, int, float, T *, long,    \
                                    cudaStream_t);                                           \
    template void launch_swiglu<T>(const float *, int, int, bool, T *, long, cudaStream_t);  \
    template void launch_rope_kv<T>(const float *, const RowDesc *, int, int, int,           \
                                    const float2 *, int, T *, T *, T *, int, long, int *,    \
                                    cudaStream_t);                                           \
    template void launch_convert<T>(const float *, T *, long, cudaStream_t);
MSD_INST(float)
MSD_INST(bf16)
#undef MSD_INST

}  // namespace msd
