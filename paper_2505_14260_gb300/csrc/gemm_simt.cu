// CUDA-core GEMM for the fp32 model dtype: Y[m][o] (=|+=) sum_k X[m][k] W[o][k].
// A plain shared-memory tiled kernel (64 x 64 tile, 4 x 4 per thread) with
// fp32 accumulation in a fixed k order, so every output depends only on its
// own row of X (rows are independent and results are reproducible).
#include "kernels.h"

namespace msd {

constexpr int SG_BO = 64, SG_BM = 64, SG_BK = 32;

template <typename T>
__device__ __forceinline__ const T *seg_row(const GemmW &W, int o, int K) {
    int s = 0;
    while (s < W.nseg - 1 && o >= W.rows[s]) { o -= W.rows[s]; ++s; }
    return reinterpret_cast<const T *>(W.w[s]) + (size_t)o * K;
}

template <typename T>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const T *__restrict__ X, int ldx, int M,
                                                        int K, GemmW W, int O, float *__restrict__ Y,
                                                        int ldy, int epi) {
    wait_prior();
    __shared__ float Ws[SG_BK][SG_BO + 1];
    __shared__ float Xs[SG_BK][SG_BM + 1];
    const int o0 = blockIdx.x * SG_BO, m0 = blockIdx.y * SG_BM;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[4][4] = {};

    for (int k0 = 0; k0 < K; k0 += SG_BK) {
        for (int t = threadIdx.x; t < SG_BO * SG_BK; t += 256) {
            const int oo = t / SG_BK, kk = t - oo * SG_BK;
            const int o = o0 + oo, k = k0 + kk;
            float v = 0.f;
            if (o < O && k < K) v = to_f(seg_row<T>(W, o, K)[k]);
            Ws[kk][oo] = v;
        }
        for (int t = threadIdx.x; t < SG_BM * SG_BK; t += 256) {
            const int mm = t / SG_BK, kk = t - mm * SG_BK;
            const int m = m0 + mm, k = k0 + kk;
            Xs[kk][mm] = (m < M && k < K) ? to_f(X[(size_t)m * ldx + k]) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < SG_BK; ++kk) {
            float wv[4], xv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) wv[i] = Ws[kk][tx * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) xv[j] = Xs[kk][ty * 4 + j];
#pragma unroll
            for (int j = 0; j < 4; ++j)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[j][i] = fmaf(xv[j], wv[i], acc[j][i]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const int m = m0 + ty * 4 + j;
        if (m >= M) continue;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int o = o0 + tx * 4 + i;
            if (o >= O) continue;
            float *y = Y + (size_t)m * ldy + o;
            *y = epi == EPI_ADD ? *y + acc[j][i] : acc[j][i];
        }
    }
}

template <typename T>
void launch_gemm_simt(const T *X, int ldx, int M, int K, const GemmW &W, int O, float *Y,
                      int ldy, int epi, cudaStream_t s) {
    if (M <= 0 || O <= 0) return;
    dim3 grid((O + SG_BO - 1) / SG_BO, (M + SG_BM - 1) / SG_BM);
    launch_chain(gemm_simt_kernel<T>, grid, 256, 0, s, X, ldx, M, K, W, O, Y, ldy, epi); note_launch();
}

template void launch_gemm_simt<float>(const float *, int, int, int, const GemmW &, int, float *,
                                      int, int, cudaStream_t);
template void launch_gemm_simt<bf16>(const bf16 *, int, int, int, const GemmW &, int, float *,
                                     int, int, cudaStream_t);

}  // namespace msd
