// bf16 GEMM on the 5th-generation tensor cores (tcgen05 + TMEM, TMA loads).
#pragma once

#include "kernels.h"

namespace msd {

struct GemmPlan;
struct GemmNorm;

// Host-side plan: split-K workspace, tile counters, tensor-map cache.
bool gemm_plan_create(GemmPlan **out, int max_rows, int hidden, int ffn, int vocab);
void gemm_plan_destroy(GemmPlan *p);

// Y[m][o] (=|+=) sum_k X[m][k] W[o][k]; X, W bf16 (K contiguous, rows 16-byte
// aligned), Y fp32. Weight tiles fill the MMA's M = 128 side, tokens its N side.
// X_lo (nullable): the lo plane of a split-bf16 X (same layout): the product
// is then W (X + X_lo), two MMAs per K step into one fp32 accumulator.
// norm_out (nullable, decode shapes M <= 128 with packed W only): the
// producer side of a folded RMSNorm (GemmNorm below); returns false (nothing
// launched) when it is given for a shape off the decode path.
bool gemm_bf16(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W, int O,
               float *Y, int ldy, int epi, int *status, cudaStream_t s, const GemmNorm *norm_out = nullptr);

// Pre-packed weights: the segments' 128-row x 64-column blocks, tile-major then
// K-block, each block stored exactly as the MMA reads it from shared memory
// (K-major rows of 128 bytes, 128-byte swizzle), so one contiguous 16 KB copy
// fills a pipeline stage. Rows past a segment's end and columns past K are 0.
size_t gemm_pack_bytes(const GemmW &W, int K);
void gemm_pack(const GemmW &W, int K, void *dst, cudaStream_t s);

// Gate/up weights of a SwiGLU MLP packed interleaved: tile t holds gate rows
// 64t .. 64t+63 in its rows 0..63 and the matching up rows in rows 64..127, so
// one tile's epilogue has both operands of silu(g) * u. As a GemmW this is one
// segment of glu_rows(F) rows; its product Y[m][128t + i] is gate row 64t + i
// for i < 64 and up row 64t + i - 64 otherwise (rows past F are 0).
inline int glu_rows(int F) { return 128 * ((F + 63) / 64); }
size_t gemm_pack_glu_bytes(int F, int K);
void gemm_pack_glu(const void *gate, const void *up, int F, int K, void *dst, cudaStream_t s);

// Epilogues fused into the decode-shape GEMM (M <= 128, packed weights):
//   EPI_SWIGLU   W glu-packed; act[m][j] = bf16(silu(g) * u), j < F
//   EPI_ROPE_KV  W = wq;wk;wv (hd | 128); q rotated (RoPE, rotate-half pairs
//                (i, i + hd/2), table (cos, sin) per position) into q_out
//                [M][H]; k rotated and v into kdst/vdst [B][nh][slots][hd] at
//                slot rows[m].dst of request rows[m].req (dst < 0: not
//                written; dst >= slots or a position outside the table: status
//                ST_RANGE).
// Outputs are split bf16 pairs, lo planes `lo` elements after act, q_out,
// kdst and vdst (lo = 0: hi values only).
struct GemmFused {
    int epi;
    bf16 *act;
    int F;
    const RowDesc *rows;
    const float2 *rope_tab;
    int max_pos;
    bf16 *q_out, *kdst, *vdst;
    int slots, nh, hd;
    long lo;
};
// RMSNorm folded into a pair of decode GEMMs (the norm's per-row scale
// commutes with the projection that follows it):
//   producer (an H-output GEMM, EPI_STORE / EPI_ADD): besides Y = x, writes
//     xg[m][o] = x[m][o] * g[o] (split bf16, lo plane at xg + lo) and
//     ss[m][tile] = sum over the tile's 128 rows of x[m][o]^2 (fixed order),
//     ld = row stride of ss;
//   consumer (EPI_ROPE_KV / EPI_SWIGLU on X = xg): scales its accumulator row m
//     by 1 / sqrt(sum_{j < parts} ss[m][j] / H + eps) (summed in j order) before
//     the rotation or the SwiGLU.
struct GemmNorm {
    float *ss;
    int ld;
    bf16 *xg;
    const bf16 *g;
    int parts, H;
    float eps;
    long lo;
};

// Runs the fused GEMM and returns true when the shape takes the decode path;
// returns false (nothing launched) otherwise.
bool gemm_bf16_fused(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W,
                     int O, const GemmFused &fx, int *status, cudaStream_t s,
                     const GemmNorm *norm_in = nullptr);

// Profiling. Mode 1: every launch is bracketed by CUDA events on its stream;
// gemm_profile_read synchronises on them and returns the launches, their
// summed durations and their algorithmic bytes (weights + X + Y), then starts
// a new window. Mode 2: launches between gemm_stamp_begin and gemm_stamp_end
// (a window, e.g. one captured step graph) carry a device slot that their CTAs
// stamp with %globaltimer (earliest entry, earliest return from
// griddepcontrol.wait, latest exit); gemm_stamp_end enqueues a kernel that
// adds the window's spans and bytes to a device sum, so a replayed graph
// measures itself. gemm_profile_read then returns those sums: ms = entry to
// exit, critical_ms = wait to exit (disjoint between kernels of one stream).
struct GemmProfile {
    long launches;
    double ms;
    double bytes;
    double weight_bytes;
    double critical_ms;
    long windows;
    double flops;       // 2 M O K summed over the launches
    double mma_flops;   // as issued: x2 where the token operand is a split pair
    double prefetch_bytes;   // weight bytes requested before the wait on the previous kernel
};
// One stamp slot of the last closed window (mode 2), summed over the windows
// since the last read: kind 0 a GEMM launch (rows M, outputs O, inner K,
// algorithmic bytes per launch), kind 1 an attention launch (query rows,
// heads, head dim; bytes 0).
struct GemmSlot {
    int kind, rows, outputs, inner;
    long launches;
    double bytes, critical_ms, ms;
};
// Device address of msd_linear_noalloc's status word on the current device
// (first use sets the device up); null if that failed.
int *noalloc_status_word();

// Test hook of the bounded mbarrier waits: one CTA waits on a barrier that
// nothing arrives at, gives up after limit_ns and records ST_TIMEOUT in
// *status. Returns false if the launch failed.
bool launch_wait_probe(int *status, long long limit_ns, cudaStream_t s);

// mode 0 off, 1 events, 2 stamps (buffers made with the plan); false if the
// stamp reset fails.
bool gemm_profile_enable(GemmPlan *p, int mode);
bool gemm_profile_on(const GemmPlan *p);     // mode 1
bool gemm_stamp_on(const GemmPlan *p);       // mode 2
void gemm_stamp_begin(GemmPlan *p);
void gemm_stamp_end(GemmPlan *p, cudaStream_t s);
GemmProfile gemm_profile_read(GemmPlan *p);
// A stamp slot for another kernel of the open window (null when none is open
// or the slots are used up); its spans are summed per slot, apart from the GEMMs'.
unsigned long long *gemm_stamp_external(GemmPlan *p, int kind, int rows, int outputs, int inner);
// Per-slot sums since the last call (which it clears): GEMM slots in launch
// order, then the other kernels'. Returns the count written, -1 on a copy
// error, 0 outside mode 2.
int gemm_profile_slots(GemmPlan *p, GemmSlot *out, int max);

}  // namespace msd
