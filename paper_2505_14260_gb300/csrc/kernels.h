// Host-side launchers of the MSD kernels. Every launcher enqueues on `s` and
// returns without synchronising.
#pragma once

#include <cuda_runtime.h>
#include <cstdint>

#include "common.cuh"

namespace msd {

// ---- elementwise / row kernels (kernels_rows.cu) ---------------------------

// x[r] = float(src[r] >= 0 ? E[src[r]] : vis[-1 - src[r]]); emb_out (nullable)
// receives the same row in T.
template <typename T>
void launch_embed_rows(const T *E, const T *vis, const int *src, int R, int H,
                       float *x, T *emb_out, int V, int *status, cudaStream_t s);

// out[r] = x[r] / sqrt(mean(x[r]^2) + eps) * g, split (lo plane at out + lo)
template <typename T>
void launch_rmsnorm(const float *x, const T *g, int R, int H, float eps, T *out, long lo,
                    cudaStream_t s);

// act[r][j] = T(silu(g) * u) with g = gu[r][j], u = gu[r][F + j], or, for
// glu-packed gate/up products (glu = true, rows of 128 * ceil(F / 64)),
// g = gu[r][128 (j / 64) + j % 64] and u 64 columns further.
template <typename T>
void launch_swiglu(const float *gu, int R, int F, bool glu, T *act, long lo, cudaStream_t s);

// RoPE (rotate-half, table of (cos, sin) per position and pair) on q and k of
// qkv [R][3H]; q -> q_out [R][H]; k, v -> kdst/vdst at slot rows[r].dst of
// request rows[r].req: [B][nh][slots][hd]; all outputs split (lo planes at +lo).
template <typename T>
void launch_rope_kv(const float *qkv, const RowDesc *rows, int R, int nh, int hd,
                    const float2 *rope_tab, int max_pos, T *q_out, T *kdst,
                    T *vdst, int slots, long lo, int *status, cudaStream_t s);

// Row r attends to cache[req][h][0 .. plen) and to the tree slots j of
// request req with bit j of mask[r] set.
template <typename T>
struct AttnArgs {
    const T *q;                 // [R][nh*hd]
    const RowDesc *rows;
    int R;
    const T *cache_k, *cache_v; // [B][nh][cache_slots][hd]
    int cache_slots;
    const T *tree_k, *tree_v;   // [B][nh][tree_slots][hd] (nullable)
    int tree_slots;
    const uint64_t *mask;       // [R][mask_words] (nullable = no tree part)
    int mask_words;
    int nh, hd;
    float scale;
    T *out;                     // [R][nh*hd]
    bool cache_fresh;           // the kernel launched just before may have written cache_k/v
    long lo;                    // split bf16: lo planes of q, K/V and out sit lo elements on (0: none)
};
template <typename T>
void launch_attention(const AttnArgs<T> &a, cudaStream_t s);

// Scratch of the chunked top-k: per-chunk records and per-row tickets
// (tickets must start at zero; the kernel leaves them at zero).
struct TopkScratch {
    float *ws;
    int *counters;
};
size_t topk_scratch_floats(int max_rows, int V);

// out[r] = argmax_j logits[r][j] (ties: lower j)
void launch_argmax(const float *logits, int R, int V, int *out, const TopkScratch &sc,
                   cudaStream_t s);

// Top-k of each row (ties: lower id) and their log-softmax values (logp
// nullable). k <= 16.
void launch_topk_logp(const float *logits, int R, int V, int k, int *ids, float *logp,
                      const TopkScratch &sc, cudaStream_t s);
// Whether the top-k kernel takes vocabulary V with k <= 16 (ceil(V / 4096) * k
// candidates <= 256 in its row merge).
bool topk_supported(int V, int k);

template <typename T>
void launch_convert(const float *x, T *y, long n, cudaStream_t s);

// Sets the device status word (first code wins), in stream order.
void launch_flag(int *status, int code, cudaStream_t s);

// ---- GEMM ------------------------------------------------------------------

// Y[m][o] (=|+=) sum_k X[m][k] * W[o][k], with W given as up to three row
// segments stacked along o (e.g. wq;wk;wv).
struct GemmW {
    const void *w[3];
    int rows[3];
    int nseg;
    const void *packed;   // the same weights pre-packed by gemm_pack (bf16), or null
};
enum { EPI_STORE = 0, EPI_ADD = 1, EPI_SWIGLU = 2, EPI_ROPE_KV = 3 };

template <typename T>
void launch_gemm_simt(const T *X, int ldx, int M, int K, const GemmW &W, int O,
                      float *Y, int ldy, int epi, cudaStream_t s);

}  // namespace msd
