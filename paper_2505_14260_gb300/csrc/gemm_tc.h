// bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM, TMA loads).
#pragma once

#include "kernels.h"

namespace msd {

struct GemmPlan;

// Host-side plan: split-K workspace, tile counters, tensor-map cache.
bool gemm_plan_create(GemmPlan **out, int max_rows, int hidden, int ffn, int vocab);
void gemm_plan_destroy(GemmPlan *p);

// Y[m][o] (=|+=) sum_k X[m][k] W[o][k]; X, W bf16 (K contiguous, rows 16-byte
// aligned), Y fp32. Weight tiles fill the MMA's M = 128 side, tokens its N side.
void gemm_bf16(GemmPlan *p, const bf16 *X, int ldx, int M, int K, const GemmW &W, int O, float *Y,
               int ldy, int epi, int *status, cudaStream_t s);

// Pre-packed weights: the segments' 128-row x 64-column blocks, tile-major then
// K-block, each block stored exactly as the MMA reads it from shared memory
// (K-major rows of 128 bytes, 128-byte swizzle), so one contiguous 16 KB copy
// fills a pipeline stage. Rows past a segment's end and columns past K are 0.
size_t gemm_pack_bytes(const GemmW &W, int K);
void gemm_pack(const GemmW &W, int K, void *dst, cudaStream_t s);

// Profiling: while enabled, every launch is bracketed by CUDA events on its
// stream; gemm_profile_read synchronises on them and returns the launches,
// their summed durations and their algorithmic bytes (weights + X + Y),
// then starts a new window.
struct GemmProfile {
    long launches;
    double ms;
    double bytes;
    double weight_bytes;
};
void gemm_profile_enable(GemmPlan *p, bool on);
bool gemm_profile_on(const GemmPlan *p);
GemmProfile gemm_profile_read(GemmPlan *p);

}  // namespace msd
