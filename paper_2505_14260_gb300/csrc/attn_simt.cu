// Tree-masked attention on CUDA cores (the fp32 path; bf16 contexts run
// attn_tc.cu for every pass). One warp per (row, head); online softmax over the visible keys:
// the cache prefix [0, plen) of the row's request, then the tree slots whose
// bit is set in the row's mask (Sec. 3.2: a candidate sees its prefix only).
#include "kernels.h"

namespace msd {

template <typename T, int HD>
__global__ void attn_simt_kernel(AttnArgs<T> a) {
    wait_prior();
    allow_dependents();
    constexpr int EPL = HD / 32;    // elements per lane
    const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (warp >= a.R * a.nh) return;
    const int r = warp / a.nh, h = warp - r * a.nh;
    const RowDesc d = a.rows[r];
    const int H = a.nh * HD;

    float q[EPL], acc[EPL];
#pragma unroll
    for (int e = 0; e < EPL; ++e) {
        q[e] = to_f(a.q[(size_t)r * H + h * HD + lane * EPL + e]) * a.scale;
        acc[e] = 0.f;
    }
    float m = -INFINITY, l = 0.f;

    auto visit = [&](const T *kr, const T *vr) {
        float s = 0.f;
#pragma unroll
        for (int e = 0; e < EPL; ++e) s += q[e] * to_f(kr[lane * EPL + e]);
        s = warp_sum(s);
        const float mn = fmaxf(m, s);
        const float corr = __expf(m - mn);
        const float p = __expf(s - mn);
        l = l * corr + p;
#pragma unroll
        for (int e = 0; e < EPL; ++e) acc[e] = acc[e] * corr + p * to_f(vr[lane * EPL + e]);
        m = mn;
    };

    const size_t cbase = (size_t)(d.req * a.nh + h) * a.cache_slots * HD;
    const int plen = d.plen < a.cache_slots ? d.plen : a.cache_slots;
    for (int p = 0; p < plen; ++p)
        visit(a.cache_k + cbase + (size_t)p * HD, a.cache_v + cbase + (size_t)p * HD);

    if (a.mask) {
        const size_t tbase = (size_t)(d.req * a.nh + h) * a.tree_slots * HD;
        for (int w = 0; w < a.mask_words; ++w) {
            uint64_t bits = a.mask[(size_t)r * a.mask_words + w];
            while (bits) {
                const int j = w * 64 + __ffsll((long long)bits) - 1;
                bits &= bits - 1;
                if (j < a.tree_slots)
                    visit(a.tree_k + tbase + (size_t)j * HD, a.tree_v + tbase + (size_t)j * HD);
            }
        }
    }
    const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
    for (int e = 0; e < EPL; ++e)
        a.out[(size_t)r * H + h * HD + lane * EPL + e] = from_f<T>(acc[e] * inv);
}

template <typename T>
void launch_attention(const AttnArgs<T> &a, cudaStream_t s) {
    if (a.R <= 0) return;
    const long warps = (long)a.R * a.nh;
    const int threads = 128;
    const int blocks = (int)((warps * 32 + threads - 1) / threads);
    if (a.hd == 128)
        launch_chain(attn_simt_kernel<T, 128>, blocks, threads, 0, s, a);
    else
        launch_chain(attn_simt_kernel<T, 64>, blocks, threads, 0, s, a);
    note_launch();
}

template void launch_attention<float>(const AttnArgs<float> &, cudaStream_t);
template void launch_attention<bf16>(const AttnArgs<bf16> &, cudaStream_t);

}  // namespace msd
