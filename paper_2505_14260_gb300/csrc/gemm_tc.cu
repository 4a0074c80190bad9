// bf16 GEMM for the decode step on the sm_103a tensor cores.
//
// Decode GEMMs multiply a few token rows (M = 7 .. 960) by large weight
// matrices, so they stream weights from HBM. The kernel swaps operands: a
// 128-row weight tile is the MMA's A operand (M = 128) and the token rows are
// its B operand (N = 16 .. 256), so the accumulator D^T[128 weight rows][N
// tokens] sits in TMEM, one weight row per TMEM lane.
//
// Per CTA (128 threads):
//   warp 0 lane 0  TMA producer: 128x64 weight tile + Nx64 token tile per
//                  stage, 128-byte swizzle, completion on a full[] mbarrier
//   warp 1         allocates TMEM; lane 0 issues tcgen05.mma (K = 16 per
//                  instruction, 4 per stage) and frees stages via
//                  tcgen05.commit -> empty[]
//   all 4 warps    epilogue: tcgen05.ld of their 32 TMEM lanes, fp32 store
//                  or accumulate into Y (coalesced along the output dim)
// Split-K: when there are too few weight tiles to cover the SMs, K is split;
// every split writes its fp32 partial to a workspace and the last CTA to
// finish a tile (atomic counter) sums the partials in split order, so results
// are deterministic, and resets the counter. No CTA waits on another.
// Every mbarrier wait is bounded (2 s of %globaltimer); on timeout the CTA
// sets the device status word and winds down.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <algorithm>
#include <cstring>
#include <mutex>
#include <unordered_map>
#include <vector>

#include "gemm_tc.h"
#include "msd.h"

namespace msd {

namespace {

constexpr int BM = 128;          // weight rows per tile (MMA M)
constexpr int BK = 64;           // K per stage: one 128-byte swizzle row of bf16
constexpr int THREADS = 128;
constexpr int MAX_STAGES = 8;
constexpr uint32_t A_BYTES = BM * BK * 2;          // 16 KB
constexpr unsigned long long TIMEOUT_NS = 2000000000ull;
constexpr size_t WS_BYTES = 64ull << 20;
constexpr int N_COUNTERS = 16384;

struct TcParams {
    int n_seg;
    int seg_tiles[3];
    int seg_rows[3];
    int seg_out[3];
    int M, kblocks, splits, kb_per_split, BN, n_tiles_n, stages, tmem_cols;
    float *Y;
    int ldy, epi;
    float *ws;
    int *counters;
    int *status;
};

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ unsigned long long gtimer() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Launch stamps (profiling): [0] the earliest CTA entry, [1] the earliest
// return from griddepcontrol.wait (the previous kernel's results are visible),
// [2] the latest CTA exit, in %globaltimer nanoseconds.
__device__ __forceinline__ void stamp_min(unsigned long long *st, int i) {
    if (st) atomicMin(st + i, gtimer());
}
__device__ __forceinline__ void stamp_max(unsigned long long *st, int i) {
    if (st) atomicMax(st + i, gtimer());
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n.reg .pred p;\n"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        "selp.b32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase with the given parity to complete: gives up when
// another thread of the CTA has set *abort_flag, or after limit_ns, when it
// sets *abort_flag and records ST_TIMEOUT in the status word.
__device__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag, int *status,
                          unsigned long long limit_ns = TIMEOUT_NS) {
    if (mbar_try(bar, parity)) return true;
    const unsigned long long t0 = gtimer();
    while (true) {
        if (mbar_try(bar, parity)) return true;
        if (*abort_flag) return false;
        if (gtimer() - t0 > limit_ns) {
            *abort_flag = 1;
            set_status(status, ST_TIMEOUT);
            return false;
        }
    }
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(map), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// Contiguous global -> shared copy completing on an mbarrier (16-byte aligned).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;"); }

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row
// core-matrix groups 1024 bytes apart, sm100 descriptor version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)1 << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B, both
// K-major, N = BN, M = 128 (256 for a two-SM tile).
__device__ __forceinline__ uint32_t instr_desc(int BN, int M = BM) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(BN >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n.reg .pred p;\n"
        "setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

// Two-SM tiles (tcgen05 cta_group::2; CTAs 2j and 2j+1 of a cluster are a
// pair). The even CTA issues M = 256 MMAs: each CTA's own 128 weight rows are A,
// at the same shared-memory offset in both; each CTA holds BN/2 token columns
// of B (the even CTA the first half); each CTA's TMEM receives its own 128 rows
// x BN. Both CTAs' copies complete on the even CTA's stage barrier.
__device__ __forceinline__ void mma_bf16_pair(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc,
                                              uint32_t accumulate) {
    asm volatile(
        "{\n.reg .pred p;\n"
        "setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(tmem_d),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
}

// Arrives, once the pair's MMAs issued so far complete, on the mbarrier at the
// same offset in each CTA of cta_mask (cluster ranks).
__device__ __forceinline__ void mma_commit_pair(uint32_t bar, uint16_t cta_mask) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
            bar),
        "h"(cta_mask)
        : "memory");
}

// 2-D tensor copy into this CTA's shared memory completing on an mbarrier of
// either CTA of the pair (a shared::cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap *map, int x, int y,
                                                 uint32_t cluster_bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.cta_group::2"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(map), "r"(x), "r"(y), "r"(cluster_bar)
        : "memory");
}

// Arrive (release, cluster scope) on an mbarrier of another CTA of the cluster.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

__device__ __forceinline__ bool mbar_try_cluster(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n.reg .pred p;\n"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
        "selp.b32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait on a barrier another CTA of the cluster arrives on.
__device__ bool mbar_wait_cluster(uint32_t bar, uint32_t parity, volatile int *abort_flag, int *status) {
    if (mbar_try_cluster(bar, parity)) return true;
    const unsigned long long t0 = gtimer();
    while (true) {
        if (mbar_try_cluster(bar, parity)) return true;
        if (*abort_flag) return false;
        if (gtimer() - t0 > TIMEOUT_NS) {
            *abort_flag = 1;
            set_status(status, ST_TIMEOUT);
            return false;
        }
    }
}

// TMEM loads of this warp's 32 lanes, 16 or 32 columns, each waited for in
// the same asm statement: the compiler sees the registers defined only once
// the data has landed, so no use can be scheduled ahead of the wait.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t *r) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,"
        "%14,%15}, [%16];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t *r) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
        "tcgen05.wait::ld.sync.aligned;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
}

// gw (16 or 32: tiles are multiples of 16 columns) columns into r[0 .. gw)
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t *r, int gw) {
    if (gw > 16) tmem_ld32(taddr, r);
    else tmem_ld16(taddr, r);
}

__global__ void __launch_bounds__(THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap mw0, const __grid_constant__ CUtensorMap mw1,
                   const __grid_constant__ CUtensorMap mw2, const __grid_constant__ CUtensorMap mx,
                   const TcParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[2 * MAX_STAGES + 1];
    __shared__ uint32_t tmem_base;
    __shared__ volatile int abort_flag;
    __shared__ int is_last;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int tile = blockIdx.x, seg = 0;
    while (seg < p.n_seg - 1 && tile >= p.seg_tiles[seg]) {
        tile -= p.seg_tiles[seg];
        ++seg;
    }
    const CUtensorMap *mw = seg == 0 ? &mw0 : (seg == 1 ? &mw1 : &mw2);
    const int row0 = tile * BM;
    const int ntile = blockIdx.y, n0 = ntile * p.BN;
    const int split = blockIdx.z;
    const int kb0 = split * p.kb_per_split;
    const int kb1 = min(p.kblocks, kb0 + p.kb_per_split);
    const int nk = kb1 - kb0;
    const int stages = p.stages;
    const uint32_t b_bytes = (uint32_t)p.BN * BK * 2;

    const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
    const uint32_t a_base = sbase, b_base = sbase + stages * A_BYTES;
    const uint32_t full0 = smem_u32(&bars[0]), empty0 = smem_u32(&bars[MAX_STAGES]);
    const uint32_t done = smem_u32(&bars[2 * MAX_STAGES]);

    if (threadIdx.x == 0) {
        for (int s = 0; s < stages; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        mbar_init(done, 1);
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(mw) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(&mx) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(&tmem_base)),
                     "r"(p.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            int issued = 0;
            for (int i = 0; i < nk; ++i) {
                const int s = i % stages;
                const uint32_t ph = (uint32_t)(i / stages) & 1u;
                if (!mbar_wait(empty0 + 8 * s, ph ^ 1u, &abort_flag, p.status)) break;
                mbar_expect_tx(full0 + 8 * s, A_BYTES + b_bytes);
                tma_load_2d(a_base + s * A_BYTES, mw, (kb0 + i) * BK, row0, full0 + 8 * s);
                tma_load_2d(b_base + s * b_bytes, &mx, (kb0 + i) * BK, n0, full0 + 8 * s);
                issued = i + 1;
            }
            if (abort_flag) {
                // let the copies still in flight land before the CTA exits
                volatile int never = 0;
                for (int i = (issued > stages ? issued - stages : 0); i < issued; ++i)
                    mbar_wait(full0 + 8 * (i % stages), (uint32_t)(i / stages) & 1u, &never,
                              p.status);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = instr_desc(p.BN);
            for (int i = 0; i < nk; ++i) {
                const int s = i % stages;
                const uint32_t ph = (uint32_t)(i / stages) & 1u;
                if (!mbar_wait(full0 + 8 * s, ph, &abort_flag, p.status)) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint64_t ad = smem_desc(a_base + s * A_BYTES);
                const uint64_t bd = smem_desc(b_base + s * b_bytes);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                    mma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (i | kk) != 0);
                mma_commit(empty0 + 8 * s);
            }
            mma_commit(done);   // arrives once every MMA issued above has completed
            // after an abort the epilogue may skip its wait: the tensor memory is
            // freed only once every MMA issued here has completed
            volatile int never = 0;
            mbar_wait(done, 0, &never, p.status);
        }
        __syncwarp();
    }

    // ---- epilogue -----------------------------------------------------------
    const bool ok = mbar_wait(done, 0, &abort_flag, p.status) && !abort_flag;
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int row = warp * 32 + lane;
    const int o_local = row0 + row;
    const bool row_ok = o_local < p.seg_rows[seg];
    const int o = p.seg_out[seg] + o_local;
    const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
    const int M = p.M;

    if (p.splits == 1) {
        for (int c0 = 0; c0 < p.BN; c0 += 16) {
            uint32_t r[16];
            tmem_ld16(taddr + c0, r);
            if (ok && row_ok) {
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const int m = n0 + c0 + j;
                    if (m < M) {
                        float *y = p.Y + (size_t)m * p.ldy + o;
                        const float v = __uint_as_float(r[j]);
                        *y = p.epi == EPI_ADD ? *y + v : v;
                    }
                }
            }
        }
    } else {
        const int tile_id = blockIdx.x * p.n_tiles_n + ntile;
        const size_t tile_elems = (size_t)p.BN * BM;
        float *part = p.ws + ((size_t)tile_id * p.splits + split) * tile_elems;
        for (int c0 = 0; c0 < p.BN; c0 += 16) {
            uint32_t r[16];
            tmem_ld16(taddr + c0, r);
#pragma unroll
            for (int j = 0; j < 16; ++j) part[(size_t)(c0 + j) * BM + row] = __uint_as_float(r[j]);
        }
        __threadfence();
        __syncthreads();
        if (threadIdx.x == 0) {
            const int prev = atomicAdd(&p.counters[tile_id], 1);
            is_last = prev == p.splits - 1;
        }
        __syncthreads();
        if (is_last) {
            __threadfence();
            const float *tb = p.ws + (size_t)tile_id * p.splits * tile_elems;
            for (int c = 0; c < p.BN; ++c) {
                const int m = n0 + c;
                if (m >= M) break;
                float v = 0.f;
                for (int s = 0; s < p.splits; ++s)
                    v += __ldcg(tb + (size_t)s * tile_elems + (size_t)c * BM + row);
                if (ok && row_ok) {
                    float *y = p.Y + (size_t)m * p.ldy + o;
                    *y = p.epi == EPI_ADD ? *y + v : v;
                }
            }
            if (threadIdx.x == 0) p.counters[tile_id] = 0;
        }
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(p.tmem_cols)
                     : "memory");
    }
}

// ---------------------------------------------------------------------------
// Persistent stream-K variant (the context GEMM).
//
// The work is the list of (tile, K-block) units, tile-major; CTA c of G takes
// units [c*U/G, (c+1)*U/G), so every CTA streams about the same number of
// weight bytes through one continuously running TMA -> MMA pipeline, across
// tile boundaries. Roles (192 threads): warp 0 lane 0 issues TMA, warp 1
// allocates TMEM and its lane 0 issues the MMAs, warps 2-5 drain the
// accumulators. Two TMEM accumulators let the epilogue of one tile overlap the
// MMAs of the next. A tile whose K range is cut between CTAs ("pieces") is
// fixed up through the workspace: each piece is written to its CTA's slot (a
// CTA has at most two cut tiles, its first and its last), and the CTA that
// takes the tile's last ticket sums the pieces in CTA order (deterministic)
// and applies the epilogue. No CTA ever waits on another.
// ---------------------------------------------------------------------------
constexpr int P_THREADS = 192;
constexpr int P_MAX_STAGES = 12;
constexpr int P_MAX_PIECES = 128;   // pieces of one cut tile (CTAs sharing it)

struct PkParams {
    int n_seg;
    int seg_tiles[3];
    int seg_rows[3];
    int seg_out[3];
    int M, kblocks, BN, n_tiles_n, stages, acc_stride, tmem_cols, grid;
    long long units;        // stream-K units: T_sk tiles x K-blocks
    int T_sk, dp_rounds;    // stream-K tiles; whole-tile rounds of G tiles after them
    const bf16 *wpacked;    // pre-packed weights (tile-contiguous, pre-swizzled)
    float *Y;
    int ldy, epi;
    float *ws;
    int *counters;
    int *status;
    bf16 *act;              // EPI_SWIGLU (glu-packed gate/up): act [M][F] split bf16
    int F;
    uint32_t stg_off;       // EPI_SWIGLU: byte offset of the 16 KB staging tile
    int has_lo;             // X is a split pair: its lo plane comes through the second map
    long lo;                // lo-plane offset of act (elements)
    unsigned long long *stamp;   // launch stamps (entry, wait, exit ns) or null
};

// silu(g) * u, the SwiGLU product of the fused epilogues.
__device__ __forceinline__ float swiglu_fused(float g, float u) {
    return __fdividef(g, 1.f + __expf(-g)) * u;
}

// CTA owning unit u under the balanced partition u0(c) = floor(c * U / G).
__device__ __forceinline__ int owner_cta(long long u, long long U, int G) {
    return (int)(((u + 1) * (long long)G - 1) / U);
}

// The work items of one CTA, in order: its share of the stream-K tiles
// [0, T_sk) (a contiguous range of (tile, K-block) units, cut at tile
// boundaries), then its whole data-parallel tiles T_sk + cta + j*G.
struct ItemIter {
    long long u, u1;
    int KB, T_sk, G, cta, dp_j, dp_rounds;
    __device__ bool next(int &t, int &kb_b, int &kb_e) {
        if (u < u1) {
            t = (int)(u / KB);
            kb_b = (int)(u - (long long)t * KB);
            kb_e = (int)min((long long)KB, kb_b + (u1 - u));
            u += kb_e - kb_b;
            return true;
        }
        if (dp_j < dp_rounds) {
            t = T_sk + cta + dp_j * G;
            kb_b = 0;
            kb_e = KB;
            ++dp_j;
            return true;
        }
        return false;
    }
};

__global__ void __launch_bounds__(P_THREADS, 1)
    gemm_persist_kernel(const __grid_constant__ CUtensorMap mx, const __grid_constant__ CUtensorMap mxl,
                        const PkParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[2 * P_MAX_STAGES + 5];
    __shared__ uint32_t tmem_base;
    __shared__ volatile int abort_flag;
    __shared__ int s_reduce;
    __shared__ int s_slot[P_MAX_PIECES];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int cta = blockIdx.x;
    const long long U = p.units;                      // stream-K units
    const long long u0 = (long long)cta * U / p.grid, u1 = (long long)(cta + 1) * U / p.grid;
    const int KB = p.kblocks, stages = p.stages, BN = p.BN;
    const bool has_lo = p.has_lo != 0;
    const uint32_t b_bytes = (uint32_t)BN * BK * 2;           // one plane of a token stage
    const uint32_t bs_bytes = has_lo ? 2 * b_bytes : b_bytes;  // hi, then lo
    const ItemIter items0{u0, u1, KB, p.T_sk, p.grid, cta, 0, p.dp_rounds};

    const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
    const uint32_t a_base = sbase, b_base = sbase + stages * A_BYTES;
    const uint32_t full0 = smem_u32(&bars[0]), empty0 = smem_u32(&bars[P_MAX_STAGES]);
    const uint32_t accf0 = smem_u32(&bars[2 * P_MAX_STAGES]);
    const uint32_t acce0 = smem_u32(&bars[2 * P_MAX_STAGES + 2]);
    const uint32_t drain = smem_u32(&bars[2 * P_MAX_STAGES + 4]);

    if (threadIdx.x == 0) {
        stamp_min(p.stamp, 0);
        for (int s = 0; s < stages; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(accf0 + 8 * a, 1);
            mbar_init(acce0 + 8 * a, 128);
        }
        mbar_init(drain, 1);
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(&tmem_base)),
                     "r"(p.tmem_cols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;

    // (tile) -> weight segment, weight rows, token rows
    auto tile_geom = [&](int t, int &seg, int &row0, int &n0) {
        const int wt = t / p.n_tiles_n, nt = t - wt * p.n_tiles_n;
        int w = wt;
        seg = 0;
        while (seg < p.n_seg - 1 && w >= p.seg_tiles[seg]) {
            w -= p.seg_tiles[seg];
            ++seg;
        }
        row0 = w * BM;
        n0 = nt * BN;
    };
    const size_t blk_elems = A_BYTES / 2;

    if (warp == 0) {
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(&mx) : "memory");
            if (has_lo) asm volatile("prefetch.tensormap [%0];" ::"l"(&mxl) : "memory");
            // Weights never depend on the previous kernel: the first stages'
            // weight blocks are requested before waiting for it.
            int n_pre = 0;
            {
                ItemIter it = items0;
                int t, kb_b, kb_e;
                while (n_pre < stages && it.next(t, kb_b, kb_e)) {
                    const bf16 *w = p.wpacked + ((size_t)(t / p.n_tiles_n) * KB + kb_b) * blk_elems;
                    for (int kb = kb_b; kb < kb_e && n_pre < stages; ++kb, ++n_pre, w += blk_elems) {
                        mbar_expect_tx(full0 + 8 * n_pre, A_BYTES + bs_bytes);
                        bulk_load(a_base + n_pre * A_BYTES, w, A_BYTES, full0 + 8 * n_pre);
                    }
                }
            }
            pdl_wait();
            stamp_min(p.stamp, 1);
            pdl_trigger();
            ItemIter it = items0;
            int t, kb_b, kb_e, s = 0, i = 0;
            uint32_t ph = 0;
            bool stop = false;
            while (!stop && it.next(t, kb_b, kb_e)) {
                int seg, row0, n0;
                tile_geom(t, seg, row0, n0);
                const bf16 *w = p.wpacked + ((size_t)(t / p.n_tiles_n) * KB + kb_b) * blk_elems;
                for (int kb = kb_b; kb < kb_e; ++kb, ++i, w += blk_elems) {
                    if (i >= n_pre) {
                        if (!mbar_wait(empty0 + 8 * s, ph ^ 1u, &abort_flag, p.status)) {
                            stop = true;
                            break;
                        }
                        mbar_expect_tx(full0 + 8 * s, A_BYTES + bs_bytes);
                        bulk_load(a_base + s * A_BYTES, w, A_BYTES, full0 + 8 * s);
                    }
                    tma_load_2d(b_base + s * bs_bytes, &mx, kb * BK, n0, full0 + 8 * s);
                    if (has_lo) tma_load_2d(b_base + s * bs_bytes + b_bytes, &mxl, kb * BK, n0, full0 + 8 * s);
                    if (++s == stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            if (abort_flag) {
                volatile int never = 0;
                for (int j = (i > stages ? i - stages : 0); j < i; ++j)
                    mbar_wait(full0 + 8 * (j % stages), (uint32_t)(j / stages) & 1u, &never,
                              p.status);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        pdl_wait();
        if (lane == 0) {
            const uint32_t idesc = instr_desc(BN);
            ItemIter it = items0;
            int t, kb_b, kb_e, s = 0;
            uint32_t ph = 0;
            for (int item = 0; !abort_flag && it.next(t, kb_b, kb_e); ++item) {
                const int a = item & 1;
                if (!mbar_wait(acce0 + 8 * a, (uint32_t)((item >> 1) & 1) ^ 1u, &abort_flag,
                               p.status))
                    break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t acc = tmem + a * p.acc_stride;
                for (int j = 0; j < kb_e - kb_b; ++j) {
                    if (!mbar_wait(full0 + 8 * s, ph, &abort_flag, p.status)) break;
                    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                    const uint64_t ad = smem_desc(a_base + s * A_BYTES);
                    const uint64_t bd = smem_desc(b_base + s * bs_bytes);
                    const uint64_t bl = smem_desc(b_base + s * bs_bytes + b_bytes);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        mma_bf16(acc, ad + 2 * kk, bd + 2 * kk, idesc, (j != 0) || (kk != 0));
                        if (has_lo) mma_bf16(acc, ad + 2 * kk, bl + 2 * kk, idesc, 1u);
                    }
                    mma_commit(empty0 + 8 * s);
                    if (++s == stages) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
                mma_commit(accf0 + 8 * a);
            }
            // every MMA issued above completes before the CTA frees its TMEM
            mma_commit(drain);
            volatile int never = 0;
            mbar_wait(drain, 0, &never, p.status);
        }
        __syncwarp();
    } else {
        // epilogue warps: TMEM lane quarter (warp % 4)
        pdl_wait();
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int et = threadIdx.x - 64;     // 0..127
        ItemIter it = items0;
        int t, kb_b, kb_e;
        for (int item = 0; it.next(t, kb_b, kb_e); ++item) {
            const int a = item & 1;
            const bool ok = mbar_wait(accf0 + 8 * a, (uint32_t)(item >> 1) & 1u, &abort_flag,
                                      p.status) && !abort_flag;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            int seg, row0, n0;
            tile_geom(t, seg, row0, n0);
            const int o_local = row0 + row;
            const bool row_ok = ok && o_local < p.seg_rows[seg];
            const int o = p.seg_out[seg] + o_local;
            const bool whole = kb_b == 0 && kb_e == KB;
            const uint32_t taddr = tmem + a * p.acc_stride + ((uint32_t)(q * 32) << 16);
            // a CTA cuts at most two stream-K tiles: its first item and its last
            const int slot = 2 * cta + (item == 0 ? 0 : 1);
            float *part = p.ws + (size_t)slot * BN * BM;
            const bool add = p.epi == EPI_ADD;
            const bool glu = p.epi == EPI_SWIGLU;
            float *stg = reinterpret_cast<float *>(smem_raw + p.stg_off);   // [32 columns][128 rows]
            for (int g0 = 0; g0 < BN; g0 += 32) {
                // up to 32 accumulator columns with one TMEM round trip
                const int gw = min(32, BN - g0);
                uint32_t r[32];
                tmem_ld_cols(taddr + g0, r, gw);
                if (whole && glu) {
                    // gate row i and up row 64 + i of the tile sit in different
                    // warps: exchange through shared memory, then thread (i, h)
                    // writes act[m][64 t + i] for the columns of half h
                    asm volatile("bar.sync 1, 128;" ::: "memory");
#pragma unroll
                    for (int j = 0; j < 32; ++j) stg[j * BM + row] = __uint_as_float(r[j]);
                    asm volatile("bar.sync 1, 128;" ::: "memory");
                    const int i = et & 63, h = et >> 6;
                    const int jo = (row0 >> 1) + i;
                    if (ok && jo < p.F) {
#pragma unroll 4
                        for (int c = 16 * h; c < 16 * h + 16; ++c) {
                            const int m = n0 + g0 + c;
                            if (c < gw && m < p.M)
                                Split<bf16>::store(p.act + (size_t)m * p.F + jo, p.lo,
                                                   swiglu_fused(stg[c * BM + i], stg[c * BM + 64 + i]));
                        }
                    }
                } else if (!whole) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < gw) part[(size_t)(g0 + j) * BM + row] = __uint_as_float(r[j]);
                } else if (row_ok) {
                    float *yb = p.Y + (size_t)(n0 + g0) * p.ldy + o;
                    const int mlim = p.M - (n0 + g0);
                    if (add) {               // residual: every load in flight, then the stores
                        float yin[32];
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            yin[j] = (j < gw && j < mlim) ? yb[(size_t)j * p.ldy] : 0.f;
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < gw && j < mlim) yb[(size_t)j * p.ldy] = yin[j] + __uint_as_float(r[j]);
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            if (j < gw && j < mlim) yb[(size_t)j * p.ldy] = __uint_as_float(r[j]);
                    }
                }
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(acce0 + 8 * a) : "memory");
            if (whole) continue;
            // ticket for the cut tile; the last piece reduces all pieces in CTA order
            __threadfence();
            asm volatile("bar.sync 1, 128;" ::: "memory");
            const int c_first = owner_cta((long long)t * KB, U, p.grid);
            const int c_last = owner_cta((long long)(t + 1) * KB - 1, U, p.grid);
            const int np = c_last - c_first + 1;
            if (et == 0) {
                const int prev = atomicAdd(&p.counters[t], 1);
                s_reduce = prev == np - 1;
            }
            if (et < np && et < P_MAX_PIECES) {
                const int cc = c_first + et;
                const long long cu0 = (long long)cc * U / p.grid;
                s_slot[et] = 2 * cc + (cu0 >= (long long)t * KB ? 0 : 1);
            }
            asm volatile("bar.sync 1, 128;" ::: "memory");
            if (!s_reduce) continue;
            if (np > P_MAX_PIECES) {
                set_status(p.status, ST_RANGE);
                continue;
            }
            __threadfence();
            // flat float4 view of the [BN][128] pieces; 16 float4 loads in flight per thread
            const int n4 = BN * BM / 4;
            const size_t piece4 = (size_t)BN * BM / 4;
            const float4 *ws4 = reinterpret_cast<const float4 *>(p.ws);
            for (int base4 = et; base4 < n4; base4 += 4 * 128) {
                float4 acc[4];
#pragma unroll
                for (int g = 0; g < 4; ++g) acc[g] = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int i0 = 0; i0 < np; i0 += 4) {
                    float4 v[4][4];
#pragma unroll
                    for (int pi = 0; pi < 4; ++pi) {
                        const bool have = i0 + pi < np;
                        const float4 *src = ws4 + (size_t)s_slot[have ? i0 + pi : 0] * piece4;
#pragma unroll
                        for (int g = 0; g < 4; ++g) {
                            const int e4 = base4 + g * 128;
                            v[pi][g] = (have && e4 < n4) ? __ldcg(src + e4)
                                                         : make_float4(0.f, 0.f, 0.f, 0.f);
                        }
                    }
#pragma unroll
                    for (int pi = 0; pi < 4; ++pi)
#pragma unroll
                        for (int g = 0; g < 4; ++g) {
                            acc[g].x += v[pi][g].x; acc[g].y += v[pi][g].y;
                            acc[g].z += v[pi][g].z; acc[g].w += v[pi][g].w;
                        }
                }
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const int e4 = base4 + g * 128;
                    if (p.epi == EPI_SWIGLU) {
                        // lane l < 16 holds gate rows 4l..4l+3 of a column, lane
                        // l + 16 the matching up rows (e4 % 32 is the lane; the
                        // branch conditions below are uniform over the warp)
                        float4 up;
                        up.x = __shfl_xor_sync(0xffffffffu, acc[g].x, 16);
                        up.y = __shfl_xor_sync(0xffffffffu, acc[g].y, 16);
                        up.z = __shfl_xor_sync(0xffffffffu, acc[g].z, 16);
                        up.w = __shfl_xor_sync(0xffffffffu, acc[g].w, 16);
                        if (e4 >= n4) continue;
                        const int col = (e4 * 4) / BM, r4 = (e4 * 4) - col * BM;
                        const int m = n0 + col;
                        const int jo = (row0 >> 1) + r4;
                        if (m >= p.M || !ok || r4 >= 64 || jo >= p.F) continue;
                        bf16 *dst = p.act + (size_t)m * p.F + jo;     // F % 4 == 0: 8-byte aligned
                        Split<bf16>::store4(dst, p.lo,
                                            make_float4(swiglu_fused(acc[g].x, up.x), swiglu_fused(acc[g].y, up.y),
                                                        swiglu_fused(acc[g].z, up.z), swiglu_fused(acc[g].w, up.w)));
                        continue;
                    }
                    if (e4 >= n4) continue;
                    const int col = (e4 * 4) / BM, r4 = (e4 * 4) - col * BM;
                    const int m = n0 + col;
                    if (m >= p.M || !ok) continue;
                    float *y = p.Y + (size_t)m * p.ldy + p.seg_out[seg] + row0 + r4;
                    if (row0 + r4 + 4 <= p.seg_rows[seg] &&
                        ((reinterpret_cast<uintptr_t>(y) & 15u) == 0)) {      // one 16-byte access
                        float4 out = acc[g];
                        if (p.epi == EPI_ADD) {
                            const float4 yi = *reinterpret_cast<const float4 *>(y);
                            out.x += yi.x; out.y += yi.y; out.z += yi.z; out.w += yi.w;
                        }
                        *reinterpret_cast<float4 *>(y) = out;
                    } else {
                        const float vv[4] = {acc[g].x, acc[g].y, acc[g].z, acc[g].w};
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            if (row0 + r4 + e < p.seg_rows[seg]) {
                                if (p.epi == EPI_ADD) y[e] = y[e] + vv[e];
                                else y[e] = vv[e];
                            }
                    }
                }
            }
            if (et == 0) p.counters[t] = 0;
        }
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0) stamp_max(p.stamp, 2);
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(p.tmem_cols)
                     : "memory");
    }
}

// ---------------------------------------------------------------------------
// Split-K with a cluster reduction (decode shapes, M <= 128 token rows).
//
// One CTA per (weight tile, token tile, K-split); the s K-splits of a tile are
// one thread-block cluster. Each CTA streams its K range (pre-packed weight
// blocks by cp.async.bulk before the previous kernel ends, token blocks by
// TMA), accumulates in TMEM, and, with s > 1, leaves its fp32 partial in its
// own shared memory; after a cluster barrier each CTA sums one slice of the
// tile over all s partials through distributed shared memory, in rank order
// (deterministic), and writes it. At most two CTAs share an SM, so every
// launch of the decode step is a single wave.
// ---------------------------------------------------------------------------
constexpr int C_THREADS = 128;
constexpr int C_STAGES = 4;

struct CkParams {
    int n_seg;
    int seg_tiles[3];
    int seg_rows[3];
    int seg_out[3];
    int M, kblocks, BN, n_tiles_n, splits, tmem_cols;
    int stages;             // ring depth (<= C_STAGES)
    int has_lo;             // X is a split pair: its lo plane comes through the second map
    const bf16 *wpacked;
    float *Y;
    int ldy, epi;
    int *status;
    GemmFused fx;           // EPI_SWIGLU / EPI_ROPE_KV operands
    GemmNorm nout, nin;     // folded RMSNorm: producer / consumer side (ss null: off)
    unsigned long long *stamp;   // launch stamps (entry, wait, exit ns) or null
};

__device__ __forceinline__ void c_cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t c_cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t c_mapa(uint32_t local, uint32_t rank) {
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(local), "r"(rank));
    return a;
}

// Where a CTA finds the S partials of the token columns it owns, [c_lo,
// c_hi) = [rank * BN / S, (rank + 1) * BN / S): its own partial ([BN][128]
// fp32, all columns) and, for S > 1, the other ranks' slices of its columns,
// pushed into its receive buffer by bulk copies (slot q < rank ? q : q - 1,
// `span` columns each).
struct PartSrc {
    const float *own, *recv;
    int rank, S, c_lo, c_hi, span;
    // shared-window address of a float4 (read with ld.shared)
    __device__ __forceinline__ uint32_t at(int q, int col, int row) const {
        const float *b = q == rank ? own + col * BM : recv + ((q < rank ? q : q - 1) * span + (col - c_lo)) * BM;
        return (uint32_t)__cvta_generic_to_shared(b + row);
    }
};

__device__ __forceinline__ float4 lds4(uint32_t a) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "r"(a));
    return v;
}
__device__ __forceinline__ float lds1(const float *p) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"((uint32_t)__cvta_generic_to_shared(p)));
    return v;
}

// Sums, in rank order, of the S partials' float4 at K (column, row) places
// (all in this CTA's shared memory); every load is issued before the first sum.
template <int K>
__device__ __forceinline__ void c_part_sums(const PartSrc &ps, const int (&col)[K], const int (&row)[K],
                                            const bool (&use)[K], float4 (&out)[K]) {
    if (ps.S == 1) {                 // one partial: plain loads (no unrolled rank loop)
#pragma unroll
        for (int k = 0; k < K; ++k) out[k] = use[k] ? lds4(ps.at(0, col[k], row[k])) : make_float4(0.f, 0.f, 0.f, 0.f);
        return;
    }
    float4 v[K][8];
#pragma unroll
    for (int q = 0; q < 8; ++q) {
        if (q >= ps.S) break;
#pragma unroll
        for (int k = 0; k < K; ++k)
            if (use[k]) v[k][q] = lds4(ps.at(q, col[k], row[k]));
    }
#pragma unroll
    for (int k = 0; k < K; ++k) {
        float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int q = 0; q < 8; ++q)
            if (q < ps.S && use[k]) {
                a.x += v[k][q].x; a.y += v[k][q].y; a.z += v[k][q].z; a.w += v[k][q].w;
            }
        out[k] = a;
    }
}

// The fused epilogues read the tile's S partials ([BN][128] fp32 in each
// cluster CTA's shared memory at part_s) and take this CTA's rank share of the
// BN * 16 groups of four rows of one token; the partials are summed in rank
// order, as in the plain reduction. Each thread handles two groups per pass,
// with every load of both issued before either is used, so that a pass costs
// about one round trip to distributed shared memory and one to global memory.

// SwiGLU (glu-packed tile: rows 0-63 gate, 64-127 up):
// act[m][64 t + i] = bf16(silu(g) * u), scaled first by the folded-norm 1/rms.
__device__ __forceinline__ void c_epi_swiglu(const CkParams &p, const PartSrc &ps, bool ok, int wt, int n0,
                                             const float *rinv) {
    // the parameters the loop uses, read once before its stores
    bf16 *const act = p.fx.act;
    const int F = p.fx.F, M = p.M;
    const long lo = p.fx.lo;
    const int n = (ps.c_hi - ps.c_lo) * 16;         // groups of this CTA's columns
    auto emit = [&](float4 a, float4 b, int c, int j) {
        const int m = n0 + c;
        if (!ok || m >= M || j >= F) return;          // F % 4 == 0: whole groups
        if (rinv) {
            const float sc = lds1(rinv + c);
            a.x *= sc; a.y *= sc; a.z *= sc; a.w *= sc;
            b.x *= sc; b.y *= sc; b.z *= sc; b.w *= sc;
        }
        const float o0 = __fdividef(a.x, 1.f + __expf(-a.x)) * b.x;
        const float o1 = __fdividef(a.y, 1.f + __expf(-a.y)) * b.y;
        const float o2 = __fdividef(a.z, 1.f + __expf(-a.z)) * b.z;
        const float o3 = __fdividef(a.w, 1.f + __expf(-a.w)) * b.w;
        Split<bf16>::store4(act + (size_t)m * F + j, lo, make_float4(o0, o1, o2, o3));
    };
    for (int e0 = threadIdx.x; e0 < n; e0 += 2 * C_THREADS) {
        int col[4], row[4];
        bool use[4];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int e = e0 + u * C_THREADS;
            col[2 * u] = col[2 * u + 1] = ps.c_lo + (e >> 4);
            row[2 * u] = (e & 15) << 2;
            row[2 * u + 1] = row[2 * u] + 64;
            use[2 * u] = use[2 * u + 1] = e < n;
        }
        float4 v[4];
        c_part_sums<4>(ps, col, row, use, v);
#pragma unroll
        for (int u = 0; u < 2; ++u)
            if (use[2 * u]) emit(v[2 * u], v[2 * u + 1], col[2 * u], wt * 64 + row[2 * u]);
    }
}

// Global operands of the first EPI_PRE groups (RoPE) or columns (norm) of a
// thread are requested before the split-K exchange, so that their round trip
// overlaps it; later ones (large column shares only) are loaded in the loop.
constexpr int EPI_PRE = 4;

struct RopePre {
    RowDesc d[EPI_PRE];
    float4 c01[EPI_PRE], c23[EPI_PRE];
};

// RoPE + K/V placement (tile of wq;wk;wv rows, hd | 128): rotate-half pairs
// (i, i + hd/2) of one head; q rotated into q_out [M][H], k rotated and v into
// kdst / vdst [B][nh][slots][hd] at the row's slot. Row descriptors come from
// shared memory (loaded while the MMAs ran).
struct RopeGeom {
    int hd, lh, half, lhd, n;
    __device__ __forceinline__ RopeGeom(int hd_, const PartSrc &ps)
        : hd(hd_), lh(hd_ == 128 ? 6 : 5), half(1 << lh), lhd(lh + 1), n((ps.c_hi - ps.c_lo) * 16) {}
    // group e of this CTA's columns: token column and first row of the pair
    __device__ __forceinline__ void at(const PartSrc &ps, int e, int &c, int &r) const {
        c = ps.c_lo + (e >> 4);
        const int p4 = (e & 15) << 2;
        r = ((p4 >> lh) << lhd) | (p4 & (half - 1));
    }
};

// the rotation-table entries (cos, sin of 4 consecutive frequencies) of one group
__device__ __forceinline__ void c_rope_tab(const CkParams &p, const RopeGeom &g, int pos, int row0, int r,
                                           float4 &c01, float4 &c23) {
    if (pos < 0 || pos >= p.fx.max_pos) {
        set_status(p.status, ST_RANGE);
        pos = 0;
    }
    const int i = (row0 + r) & (g.hd - 1);
    const float4 *cs = reinterpret_cast<const float4 *>(p.fx.rope_tab + (size_t)pos * g.half + i);
    c01 = cs[0];
    c23 = cs[1];
}

__device__ __forceinline__ void c_rope_pre(const CkParams &p, const PartSrc &ps, bool ok, int seg, int row0,
                                           int n0, int rows_here, const RowDesc *srow, RopePre &pre) {
    const RopeGeom g(p.fx.hd, ps);
#pragma unroll
    for (int k = 0; k < EPI_PRE; ++k) {
        const int e = threadIdx.x + k * C_THREADS;
        if (e >= g.n) break;
        int c, r;
        g.at(ps, e, c, r);
        pre.d[k] = srow[c];
        if (ok && seg < 2 && n0 + c < p.M && r < rows_here)
            c_rope_tab(p, g, pre.d[k].pos, row0, r, pre.c01[k], pre.c23[k]);
    }
}

__device__ __forceinline__ void c_epi_rope(const CkParams &p, const PartSrc &ps, bool ok, int seg, int row0,
                                           int n0, int rows_here, const float *rinv, const RowDesc *srow,
                                           const RopePre &pre) {
    const RopeGeom g(p.fx.hd, ps);
    const int slots = p.fx.slots, nh = p.fx.nh, M = p.M, hd = g.hd, half = g.half;
    bf16 *const qo = p.fx.q_out, *const kvd = seg == 1 ? p.fx.kdst : p.fx.vdst;
    const long lo = p.fx.lo;
    int *const status = p.status;
    for (int k = 0;; ++k) {
        const int e = threadIdx.x + k * C_THREADS;
        if (e >= g.n) break;
        int c, r;
        g.at(ps, e, c, r);
        const int m = n0 + c;
        if (!ok || m >= M || r >= rows_here) continue;
        RowDesc d;
        float4 c01, c23;
        if (k < EPI_PRE) {
#pragma unroll
            for (int j = 0; j < EPI_PRE; ++j)       // static indices only
                if (j == k) { d = pre.d[j]; c01 = pre.c01[j]; c23 = pre.c23[j]; }
        } else {
            d = srow[c];
            if (seg < 2) c_rope_tab(p, g, d.pos, row0, r, c01, c23);
        }
        const int col[2] = {c, c}, row[2] = {r, r + half};
        const bool use[2] = {true, true};
        float4 v[2];
        c_part_sums<2>(ps, col, row, use, v);
        float4 a = v[0], b = v[1];
        if (rinv) {
            const float sc = lds1(rinv + c);
            a.x *= sc; a.y *= sc; a.z *= sc; a.w *= sc;
            b.x *= sc; b.y *= sc; b.z *= sc; b.w *= sc;
        }
        const int o = row0 + r, h = o >> g.lhd, i = o & (hd - 1);
        if (seg < 2) {
            const float x0 = a.x, x1 = a.y, x2 = a.z, x3 = a.w;
            a.x = x0 * c01.x - b.x * c01.y; b.x = b.x * c01.x + x0 * c01.y;
            a.y = x1 * c01.z - b.y * c01.w; b.y = b.y * c01.z + x1 * c01.w;
            a.z = x2 * c23.x - b.z * c23.y; b.z = b.z * c23.x + x2 * c23.y;
            a.w = x3 * c23.z - b.w * c23.w; b.w = b.w * c23.z + x3 * c23.w;
        }
        bf16 *dst;
        if (seg == 0) {
            dst = qo + (size_t)m * (nh * hd) + o;
        } else {
            if (d.dst >= slots) set_status(status, ST_RANGE);
            if (d.dst < 0 || d.dst >= slots) continue;
            dst = kvd + ((size_t)(d.req * nh + h) * slots + d.dst) * hd + i;
        }
        Split<bf16>::store4(dst, lo, a);
        Split<bf16>::store4(dst + half, lo, b);
    }
}

// Residual rows of the first EPI_PRE columns of a warp (folded-norm producer
// with accumulation), requested before the exchange.
__device__ __forceinline__ void c_norm_pre(const CkParams &p, const PartSrc &ps, bool ok, int o_base,
                                           int rows_here, int n0, float4 (&yv)[EPI_PRE]) {
    const int warp = threadIdx.x >> 5, r4 = (threadIdx.x & 31) * 4;
    if (p.epi != EPI_ADD || r4 + 4 > rows_here) return;
#pragma unroll
    for (int k = 0; k < EPI_PRE; ++k) {
        const int c = ps.c_lo + warp + k * (C_THREADS / 32);
        if (ok && c < ps.c_hi && n0 + c < p.M)
            yv[k] = *reinterpret_cast<const float4 *>(p.Y + (size_t)(n0 + c) * p.ldy + o_base + r4);
    }
}

// Producer side of a folded RMSNorm: this CTA's token columns, one warp per
// column (lane = 4 consecutive weight rows): the S partials summed in rank
// order, the residual added, then Y (fp32), xg = bf16(y * g) and the column's
// sum of squares over the tile's rows (a warp reduction in a fixed order) into
// ss[m][tile].
__device__ __forceinline__ void c_reduce_norm(const CkParams &p, const PartSrc &ps, bool ok, int tile, int o_base,
                                              int rows_here, int n0, const float4 (&yv)[EPI_PRE]) {
    constexpr int NW = C_THREADS / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool add = p.epi == EPI_ADD;
    const int r4 = lane * 4;
    const bool full = r4 + 4 <= rows_here;
    float g4[4] = {0.f, 0.f, 0.f, 0.f};
    if (full) {
        const uint2 gw = *reinterpret_cast<const uint2 *>(p.nout.g + o_base + r4);
        const __nv_bfloat162 g01 = *reinterpret_cast<const __nv_bfloat162 *>(&gw.x);
        const __nv_bfloat162 g23 = *reinterpret_cast<const __nv_bfloat162 *>(&gw.y);
        g4[0] = __low2float(g01); g4[1] = __high2float(g01);
        g4[2] = __low2float(g23); g4[3] = __high2float(g23);
    }
    float *const Y = p.Y;
    bf16 *const XG = p.nout.xg;
    const int ldy = p.ldy, M = p.M;
    const long xlo = p.nout.lo;
    float *const ssd = p.nout.ss;
    const int ssld = p.nout.ld;
    const bf16 *const gn = p.nout.g;
    for (int k = 0;; ++k) {
        const int c = ps.c_lo + warp + k * NW;
        if (c >= ps.c_hi) break;                         // warp-uniform
        const int col[1] = {c}, row[1] = {r4};
        const bool use[1] = {true};
        float4 v[1];
        c_part_sums<1>(ps, col, row, use, v);
        float a[4] = {v[0].x, v[0].y, v[0].z, v[0].w};
        const int m = n0 + c;
        const bool live = ok && m < M;                   // warp-uniform
        float ss = 0.f;
        if (live) {
            float *y = Y + (size_t)m * ldy + o_base + r4;
            bf16 *xg = XG + (size_t)m * ldy + o_base + r4;
            if (full) {
                if (add) {
                    float4 yi;
                    if (k < EPI_PRE) {
#pragma unroll
                        for (int j = 0; j < EPI_PRE; ++j)
                            if (j == k) yi = yv[j];
                    } else {
                        yi = *reinterpret_cast<const float4 *>(y);
                    }
                    a[0] += yi.x; a[1] += yi.y; a[2] += yi.z; a[3] += yi.w;
                }
                *reinterpret_cast<float4 *>(y) = make_float4(a[0], a[1], a[2], a[3]);
                Split<bf16>::store4(xg, xlo, make_float4(a[0] * g4[0], a[1] * g4[1], a[2] * g4[2], a[3] * g4[3]));
                ss = a[0] * a[0] + a[1] * a[1] + a[2] * a[2] + a[3] * a[3];
            } else {
                const bf16 *g = gn + o_base + r4;
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (r4 + e < rows_here) {
                        const float ye = add ? y[e] + a[e] : a[e];
                        y[e] = ye;
                        Split<bf16>::store(xg + e, xlo, ye * __bfloat162float(g[e]));
                        ss += ye * ye;
                    }
            }
        }
        ss = warp_sum(ss);
        if (live && lane == 0) ssd[(size_t)m * ssld + tile] = ss;
    }
}

template <bool PAIR>
__global__ void __launch_bounds__(C_THREADS)
    gemm_cluster_kernel(const __grid_constant__ CUtensorMap mx, const __grid_constant__ CUtensorMap mxl,
                        const __grid_constant__ CUtensorMap mw, const CkParams p) {
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[2 * C_STAGES + 3];
    __shared__ uint32_t tmem_base;
    __shared__ volatile int abort_flag;
    __shared__ float s_rinv[128];     // folded RMSNorm (consumer): 1/rms of each token column
    __shared__ RowDesc s_rows[128];   // EPI_ROPE_KV: the token columns' row descriptors

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int wt = blockIdx.x, seg = 0;
    while (seg < p.n_seg - 1 && wt >= p.seg_tiles[seg]) {
        wt -= p.seg_tiles[seg];
        ++seg;
    }
    const int row0 = wt * BM;
    const int n0 = blockIdx.y * p.BN;
    const int split = blockIdx.z, S = p.splits;
    const int KB = p.kblocks;
    const int kb0 = (int)((long long)split * KB / S), kb1 = (int)((long long)(split + 1) * KB / S);
    const int nk = kb1 - kb0;
    const int BN = p.BN;
    const int stages = p.stages;
    const bool has_lo = p.has_lo != 0;
    // Two-SM mode (one K split only): CTAs 2j and 2j+1 run one M = 256 tile;
    // each holds its own weight rows and half of the token columns.
    constexpr bool pair = PAIR;
    const uint32_t half = pair ? (blockIdx.x & 1u) : 0u;       // 1: the odd CTA of a pair
    const int BNs = pair ? BN / 2 : BN;                        // token columns in this CTA's stages
    const uint32_t b_bytes = (uint32_t)BNs * BK * 2;         // one plane of a token stage
    const uint32_t bs_bytes = has_lo ? 2 * b_bytes : b_bytes; // hi, then lo
    const size_t blk_elems = A_BYTES / 2;
    const bf16 *wblk = p.wpacked + ((size_t)blockIdx.x * KB + kb0) * blk_elems;

    const uint32_t sbase = (smem_u32(smem_raw) + 1023u) & ~1023u;
    const uint32_t a_base = sbase, b_base = sbase + stages * A_BYTES;
    const uint32_t full0 = smem_u32(&bars[0]), empty0 = smem_u32(&bars[C_STAGES]);
    const uint32_t done = smem_u32(&bars[2 * C_STAGES]);
    const uint32_t recv_bar = smem_u32(&bars[2 * C_STAGES + 1]);   // the other ranks' slices have landed
    const uint32_t pexit = smem_u32(&bars[2 * C_STAGES + 2]);      // (pair) the other CTA is done with its TMEM

    if (threadIdx.x == 0) {
        stamp_min(p.stamp, 0);
        for (int s = 0; s < stages; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        mbar_init(done, 1);
        mbar_init(recv_bar, 1);
        mbar_init(pexit, 1);
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        if constexpr (pair) {   // both CTAs of the pair allocate together (the same columns in each)
            asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(&tmem_base)),
                         "r"(p.tmem_cols)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
        } else {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                             smem_u32(&tmem_base)),
                         "r"(p.tmem_cols)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
        }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;
    const uint32_t my_rank = pair ? c_cluster_rank() : 0u;
    const uint32_t lead_rank = my_rank & ~1u;                 // (pair) the even CTA
    const uint16_t pair_mask = (uint16_t)(3u << lead_rank);
    // where this CTA's copies complete: its own barriers, or (pair) the even CTA's
    const uint32_t sig0 = pair ? c_mapa(full0, lead_rank) : full0;
    const uint32_t stage_tx = (pair ? 2u : 1u) * (A_BYTES + bs_bytes);
    // (pair) both CTAs' barriers are initialised before either signals the other's
    if constexpr (pair) c_cluster_sync();

    if (warp == 0) {
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(&mx) : "memory");
            if (has_lo) asm volatile("prefetch.tensormap [%0];" ::"l"(&mxl) : "memory");
            if (pair) asm volatile("prefetch.tensormap [%0];" ::"l"(&mw) : "memory");
            // the weight block of pipeline step i: a bulk copy, or (pair) a tensor
            // copy of its 128 rows that completes on the even CTA's barrier
            auto load_w = [&](int i, int st) {
                if (!pair || half == 0) mbar_expect_tx(full0 + 8 * st, stage_tx);
                if constexpr (pair)
                    tma_load_2d_pair(a_base + st * A_BYTES, &mw, 0, (int)(((size_t)blockIdx.x * KB + kb0 + i) * BM),
                                     sig0 + 8 * st);
                else
                    bulk_load(a_base + st * A_BYTES, wblk + (size_t)i * blk_elems, A_BYTES, full0 + 8 * st);
            };
            // weights first (they never depend on the previous kernel), then wait
            const int n_pre = min(stages, nk);
            for (int j = 0; j < n_pre; ++j) load_w(j, j);
            pdl_wait();
            stamp_min(p.stamp, 1);
            pdl_trigger();
            int s = 0;
            uint32_t ph = 0;
            int i = 0;
            for (; i < nk; ++i) {
                if (i >= n_pre) {
                    if (!mbar_wait(empty0 + 8 * s, ph ^ 1u, &abort_flag, p.status)) break;
                    load_w(i, s);
                }
                if constexpr (pair) {
                    const int ny = n0 + (int)half * BNs;
                    tma_load_2d_pair(b_base + s * bs_bytes, &mx, (kb0 + i) * BK, ny, sig0 + 8 * s);
                    if (has_lo) tma_load_2d_pair(b_base + s * bs_bytes + b_bytes, &mxl, (kb0 + i) * BK, ny, sig0 + 8 * s);
                } else {
                    tma_load_2d(b_base + s * bs_bytes, &mx, (kb0 + i) * BK, n0, full0 + 8 * s);
                    if (has_lo) tma_load_2d(b_base + s * bs_bytes + b_bytes, &mxl, (kb0 + i) * BK, n0, full0 + 8 * s);
                }
                if (++s == stages) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            if (abort_flag && (!pair || half == 0)) {   // (pair: the even CTA's barriers count both CTAs' copies)
                volatile int never = 0;
                for (int j = (i > stages ? i - stages : 0); j < i; ++j)
                    mbar_wait(full0 + 8 * (j % stages), (uint32_t)(j / stages) & 1u, &never, p.status);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        pdl_wait();
        if (lane == 0 && (!pair || half == 0)) {      // (pair: the even CTA issues for both)
            const uint32_t idesc = instr_desc(BN, pair ? 2 * BM : BM);
            int s = 0;
            uint32_t ph = 0;
            for (int i = 0; i < nk; ++i) {
                if (pair ? !mbar_wait_cluster(full0 + 8 * s, ph, &abort_flag, p.status)
                         : !mbar_wait(full0 + 8 * s, ph, &abort_flag, p.status))
                    break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint64_t ad = smem_desc(a_base + s * A_BYTES);
                const uint64_t bd = smem_desc(b_base + s * bs_bytes);
                const uint64_t bl = smem_desc(b_base + s * bs_bytes + b_bytes);
                if constexpr (pair) {
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        mma_bf16_pair(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (i != 0) || (kk != 0));
                        if (has_lo) mma_bf16_pair(tmem, ad + 2 * kk, bl + 2 * kk, idesc, 1u);
                    }
                    mma_commit_pair(empty0 + 8 * s, pair_mask);
                } else {
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        mma_bf16(tmem, ad + 2 * kk, bd + 2 * kk, idesc, (i != 0) || (kk != 0));
                        if (has_lo) mma_bf16(tmem, ad + 2 * kk, bl + 2 * kk, idesc, 1u);
                    }
                    mma_commit(empty0 + 8 * s);
                }
                if (++s == stages) {
                    s = 0;
                    ph ^= 1u;
                }
            }
            if constexpr (pair) mma_commit_pair(done, pair_mask);
            else mma_commit(done);
            volatile int never = 0;     // (as gemm_tc_kernel: no MMA outlives the CTA's TMEM)
            mbar_wait(done, 0, &never, p.status);
        }
        __syncwarp();
    } else {
        pdl_wait();
        // idle during the main loop: the row scales of a folded RMSNorm
        if (p.nin.ss)
            for (int t = threadIdx.x - 64; t < p.BN; t += C_THREADS - 64) {
                const int m = n0 + t;
                float sum = 0.f;
                if (m < p.M)
                    for (int j = 0; j < p.nin.parts; ++j) sum += p.nin.ss[(size_t)m * p.nin.ld + j];
                s_rinv[t] = rsqrtf(sum / (float)p.nin.H + p.nin.eps);
            }
        if (p.epi == EPI_ROPE_KV)
            for (int t = threadIdx.x - 64; t < p.BN; t += C_THREADS - 64) {
                const int m = n0 + t;
                s_rows[t] = m < p.M ? p.fx.rows[m] : RowDesc{0, 0, 0, -1};
            }
    }

    // ---- epilogue: all 4 warps, TMEM lane quarter = warp -------------------
    const bool ok = mbar_wait(done, 0, &abort_flag, p.status) && !abort_flag;
    // K split over the cluster: this CTA's MMAs are done, so its ring may now
    // receive the other ranks' slices. It arrives on the cluster barrier here
    // and waits on it only after storing its own partial, which hides the
    // barrier's round trip behind that store.
    if (S > 1) {
        __syncwarp();
        asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
    }
    pdl_wait();                       // (every thread) before reading Y, rows or the table
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const int row = warp * 32 + lane;
    const uint32_t taddr = tmem + ((uint32_t)(warp * 32) << 16);
    const bool add = p.epi == EPI_ADD;
    const int rows_here = p.seg_rows[seg] - row0;           // valid weight rows in this tile
    const int o_base = p.seg_out[seg] + row0;
    const bool paired = p.epi >= EPI_SWIGLU;
    const bool norm_out = p.nout.ss != nullptr;
    if (S == 1 && !paired && !norm_out) {
        for (int g0 = 0; g0 < BN; g0 += 32) {
            const int gw = min(32, BN - g0);
            uint32_t r[32];
            tmem_ld_cols(taddr + g0, r, gw);
            if (ok && row < rows_here) {
                float *yb = p.Y + (size_t)(n0 + g0) * p.ldy + o_base + row;
                const int mlim = p.M - (n0 + g0);
                if (add) {
                    float yin[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        yin[j] = (j < gw && j < mlim) ? yb[(size_t)j * p.ldy] : 0.f;
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < gw && j < mlim) yb[(size_t)j * p.ldy] = yin[j] + __uint_as_float(r[j]);
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (j < gw && j < mlim) yb[(size_t)j * p.ldy] = __uint_as_float(r[j]);
                }
            }
        }
    } else {
        // partial [BN][128] fp32 in this CTA's (now idle) stage memory
        float *part = reinterpret_cast<float *>(smem_raw + (sbase - smem_u32(smem_raw)));
        for (int g0 = 0; g0 < BN; g0 += 32) {
            const int gw = min(32, BN - g0);
            uint32_t r[32];
            tmem_ld_cols(taddr + g0, r, gw);
#pragma unroll
            for (int j = 0; j < 32; ++j)
                if (j < gw) part[(g0 + j) * BM + row] = __uint_as_float(r[j]);
        }
        // Split-K reduction, push style: after a cluster barrier (every rank's
        // MMAs are done, so every rank's stage memory is free), each rank sends
        // every other rank the slice of its partial that holds that rank's
        // columns, by bulk copies into the receiver's buffer that complete on the
        // receiver's mbarrier; each rank then reduces its own columns from its
        // own shared memory, in rank order.
        const uint32_t rank = S > 1 ? c_cluster_rank() : 0u;
        const int span = (BN + S - 1) / S;
        PartSrc ps;
        ps.own = part;
        ps.recv = part + BN * BM;
        ps.rank = (int)rank;
        ps.S = S;
        ps.c_lo = (int)rank * BN / S;
        ps.c_hi = ((int)rank + 1) * BN / S;
        ps.span = span;
        bool okr = ok;
        __syncthreads();                 // the staged row descriptors and the partial, for every warp
        RopePre rpre;
        float4 yv[EPI_PRE];
        // the global operands of the first groups are requested after the
        // cluster barrier, so that they arrive while the slices are exchanged
        auto pre_loads = [&]() {
            if (paired && p.epi == EPI_ROPE_KV) c_rope_pre(p, ps, ok, seg, row0, n0, rows_here, s_rows, rpre);
            if (norm_out) c_norm_pre(p, ps, ok, o_base, rows_here, n0, yv);
        };
        if (S > 1) {
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");    // part, for the bulk copies
            asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
            if (threadIdx.x == 0) {
                mbar_expect_tx(recv_bar, (uint32_t)((S - 1) * (ps.c_hi - ps.c_lo) * BM * 4));
                for (int t = 0; t < S; ++t) {
                    const int t_lo = t * BN / S, t_hi = (t + 1) * BN / S;
                    if (t == (int)rank || t_hi == t_lo) continue;
                    const int slot = (int)rank < t ? (int)rank : (int)rank - 1;
                    const uint32_t src = smem_u32(part + t_lo * BM);
                    const uint32_t dst = c_mapa(smem_u32(ps.recv + slot * span * BM), (uint32_t)t);
                    asm volatile(
                        "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                            dst),
                        "r"(src), "r"((uint32_t)((t_hi - t_lo) * BM * 4)), "r"(c_mapa(recv_bar, (uint32_t)t))
                        : "memory");
                }
                asm volatile("cp.async.bulk.commit_group;" ::: "memory");
            }
            pre_loads();
            okr = mbar_wait(recv_bar, 0, &abort_flag, p.status) && ok;
        } else {
            pre_loads();
        }
        if (p.epi == EPI_SWIGLU)
            c_epi_swiglu(p, ps, okr, wt, n0, p.nin.ss ? s_rinv : nullptr);
        else if (paired)
            c_epi_rope(p, ps, okr, seg, row0, n0, rows_here, p.nin.ss ? s_rinv : nullptr, s_rows, rpre);
        else if (norm_out)
            c_reduce_norm(p, ps, okr, wt, o_base, rows_here, n0, yv);
        else {
            // plain reduction of this CTA's columns, float4 = 4 consecutive weight rows of one token
            const int n = (ps.c_hi - ps.c_lo) * (BM / 4);
            for (int e0 = threadIdx.x; e0 < n; e0 += 2 * C_THREADS) {
                int col[2], row[2];
                bool use[2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int e = e0 + u * C_THREADS;
                    col[u] = ps.c_lo + e / (BM / 4);
                    row[u] = (e % (BM / 4)) * 4;
                    use[u] = e < n;
                }
                float4 v[2];
                c_part_sums<2>(ps, col, row, use, v);
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int m = n0 + col[u], r4 = row[u];
                    if (!use[u] || !okr || m >= p.M) continue;
                    float4 acc = v[u];
                    float *y = p.Y + (size_t)m * p.ldy + o_base + r4;
                    if (r4 + 4 <= rows_here && ((reinterpret_cast<uintptr_t>(y) & 15u) == 0)) {
                        if (add) {
                            const float4 yi = *reinterpret_cast<const float4 *>(y);
                            acc.x += yi.x; acc.y += yi.y; acc.z += yi.z; acc.w += yi.w;
                        }
                        *reinterpret_cast<float4 *>(y) = acc;
                    } else {
                        const float vv[4] = {acc.x, acc.y, acc.z, acc.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e)
                            if (r4 + e < rows_here) {
                                if (add) y[e] = y[e] + vv[e];
                                else y[e] = vv[e];
                            }
                    }
                }
            }
        }
        // this CTA's outgoing copies have read its partial before it exits
        if (S > 1 && threadIdx.x == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0) stamp_max(p.stamp, 2);
    if constexpr (pair) {
        // the pair frees its tensor memory together, once both CTAs have read
        // theirs (and, for the odd CTA, once the even one has seen every copy land)
        if (warp == 1) {
            if (lane == 0) {
                mbar_arrive_remote(c_mapa(pexit, my_rank ^ 1u));
                volatile int never = 0;
                mbar_wait_cluster(pexit, 0, &never, p.status);
            }
            __syncwarp();
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                         "r"(p.tmem_cols)
                         : "memory");
        }
    } else if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(p.tmem_cols)
                     : "memory");
    }
}

// One 16 KB packed block per CTA: rows row0..row0+127 of the block's segment,
// columns kb*64 .. kb*64+63, written in the swizzled shared-memory order.
__global__ void pack_kernel(GemmW W, int K, int KB, uint8_t *dst) {
    const long long blk = blockIdx.x;
    const int wt = (int)(blk / KB), kb = (int)(blk - (long long)wt * KB);
    int seg = 0, w = wt;
    while (seg < W.nseg - 1 && w >= (W.rows[seg] + BM - 1) / BM) {
        w -= (W.rows[seg] + BM - 1) / BM;
        ++seg;
    }
    const bf16 *src = static_cast<const bf16 *>(W.w[seg]);
    const int rows = W.rows[seg], row0 = w * BM;
    uint8_t *out = dst + blk * (long long)A_BYTES;
    for (int q = threadIdx.x; q < BM * 8; q += blockDim.x) {
        const int r = q >> 3, c = q & 7;
        const int row = row0 + r, k = kb * BK + c * 8;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (row < rows && k + 8 <= K) v = *reinterpret_cast<const uint4 *>(src + (size_t)row * K + k);
        *reinterpret_cast<uint4 *>(out + r * 128 + ((c ^ (r & 7)) << 4)) = v;
    }
}

// Glu-packed gate/up: block (t, kb) takes gate rows 64t.. into its rows 0..63
// and up rows 64t.. into rows 64..127 (rows past F are 0).
__global__ void pack_glu_kernel(const bf16 *gate, const bf16 *up, int F, int K, int KB, uint8_t *dst) {
    const long long blk = blockIdx.x;
    const int t = (int)(blk / KB), kb = (int)(blk - (long long)t * KB);
    uint8_t *out = dst + blk * (long long)A_BYTES;
    for (int q = threadIdx.x; q < BM * 8; q += blockDim.x) {
        const int r = q >> 3, c = q & 7;
        const int frow = t * 64 + (r & 63), k = kb * BK + c * 8;
        const bf16 *src = r < 64 ? gate : up;
        uint4 v = make_uint4(0, 0, 0, 0);
        if (frow < F && k + 8 <= K) v = *reinterpret_cast<const uint4 *>(src + (size_t)frow * K + k);
        *reinterpret_cast<uint4 *>(out + r * 128 + ((c ^ (r & 7)) << 4)) = v;
    }
}

// Records a host-detected problem in the device status word, in stream order.
__global__ void flag_kernel(int *status, int code) { set_status(status, code); }

struct MapKey {
    const void *ptr;
    long rows, cols, ld, box_rows;
    bool operator==(const MapKey &o) const {
        return ptr == o.ptr && rows == o.rows && cols == o.cols && ld == o.ld &&
               box_rows == o.box_rows;
    }
};
struct MapKeyHash {
    size_t operator()(const MapKey &k) const {
        size_t h = std::hash<const void *>()(k.ptr);
        h ^= std::hash<long>()(k.rows * 1315423911L + k.cols * 2654435761L + k.ld * 97 + k.box_rows);
        return h;
    }
};

}  // namespace

constexpr int MAX_STAMPS = 2048;   // GEMM launches per stamping window
constexpr int MAX_XSTAMPS = 512;   // other stamped launches (attention) per window, slots after the GEMMs'
constexpr int ALL_STAMPS = MAX_STAMPS + MAX_XSTAMPS;

// Sums of the closed stamping windows (device memory).
struct StampAcc {
    unsigned long long span_ns;   // sum over launches of exit - entry
    unsigned long long crit_ns;   // sum over launches of exit - wait
    unsigned long long launches, windows;
    double bytes, wbytes;         // algorithmic bytes of those launches
    double flops, mma_flops;      // 2 M O K of those launches; as issued (x2 for split operands)
    double pre_bytes;             // weight bytes requested before the wait on the previous kernel
};

__global__ void stamp_init_kernel(unsigned long long *st, int n, StampAcc *acc, unsigned long long *slot_acc) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        st[3 * i] = ~0ull;
        st[3 * i + 1] = ~0ull;
        st[3 * i + 2] = 0ull;
        slot_acc[3 * i] = slot_acc[3 * i + 1] = slot_acc[3 * i + 2] = 0ull;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) *acc = StampAcc{0, 0, 0, 0, 0.0, 0.0, 0.0, 0.0, 0.0};
}

// A stamp's spans: exit - max(wait, entry) and exit - entry (0, 0 if unused).
__device__ __forceinline__ bool stamp_spans(const unsigned long long *st, unsigned long long &crit,
                                            unsigned long long &span) {
    const unsigned long long e0 = st[0], w0 = st[1], e1 = st[2];
    if (e0 == ~0ull || e1 < e0) return false;
    span = e1 - e0;
    crit = e1 - (w0 <= e1 ? (w0 > e0 ? w0 : e0) : e0);
    return true;
}

// Closes a window of n GEMM launches and xn other launches: adds the GEMMs'
// spans to acc, every launch's spans to its slot's sums in slot_acc, and
// clears the slots for the next window (one block; runs after the window's
// launches).
__global__ void stamp_collect_kernel(unsigned long long *st, int n, int xn, double bytes, double wbytes, double flops,
                                     double mma_flops, double pre_bytes, StampAcc *acc, unsigned long long *slot_acc) {
    __shared__ unsigned long long s_span, s_crit, s_cnt;
    if (threadIdx.x == 0) s_span = s_crit = s_cnt = 0;
    __syncthreads();
    unsigned long long span = 0, crit = 0, cnt = 0;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        unsigned long long c1, s1;
        if (stamp_spans(st + 3 * i, c1, s1)) {
            span += s1;
            crit += c1;
            ++cnt;
            slot_acc[3 * i] += c1;
            slot_acc[3 * i + 1] += s1;
            slot_acc[3 * i + 2] += 1;
        }
        st[3 * i] = ~0ull;
        st[3 * i + 1] = ~0ull;
        st[3 * i + 2] = 0ull;
    }
    for (int j = threadIdx.x; j < xn; j += blockDim.x) {
        const int i = MAX_STAMPS + j;
        unsigned long long c1, s1;
        if (stamp_spans(st + 3 * i, c1, s1)) {
            slot_acc[3 * i] += c1;
            slot_acc[3 * i + 1] += s1;
            slot_acc[3 * i + 2] += 1;
        }
        st[3 * i] = ~0ull;
        st[3 * i + 1] = ~0ull;
        st[3 * i + 2] = 0ull;
    }
    atomicAdd(&s_span, span);
    atomicAdd(&s_crit, crit);
    atomicAdd(&s_cnt, cnt);
    __syncthreads();
    if (threadIdx.x == 0) {
        acc->span_ns += s_span;
        acc->crit_ns += s_crit;
        acc->launches += s_cnt;
        acc->windows += 1;
        acc->bytes += bytes;
        acc->wbytes += wbytes;
        acc->flops += flops;
        acc->mma_flops += mma_flops;
        acc->pre_bytes += pre_bytes;
    }
}

struct GemmPlan {
    float *ws = nullptr;
    int *counters = nullptr;
    int num_sms = 148;
    PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    std::unordered_map<MapKey, CUtensorMap, MapKeyHash> maps;
    bool smem_set = false;
    bool cluster_attr_set = false;
    bool profile = false;
    std::vector<cudaEvent_t> ev;
    size_t ev_used = 0;
    double prof_bytes = 0.0, prof_wbytes = 0.0, prof_flops = 0.0, prof_mma = 0.0, prof_pre = 0.0;
    // launch stamps: one slot of 3 per launch of a stamping window
    bool stamp_mode = false, stamp_active = false;
    int stamp_next = 0, xstamp_next = 0, cur_slot = -1;
    double stamp_bytes = 0.0, stamp_wbytes = 0.0, stamp_flops = 0.0, stamp_mma = 0.0, stamp_pre = 0.0;
    unsigned long long *stamps = nullptr;
    StampAcc *stamp_acc = nullptr;
    // per slot: sums of exit - wait, exit - entry and the stamped launches
    // ([ALL_STAMPS][3]); what each slot of the last closed window held
    unsigned long long *slot_acc = nullptr;
    std::vector<GemmSlot> slot_info = std::vector<GemmSlot>(ALL_STAMPS);
    int slot_n = 0, xslot_n = 0;
};

bool gemm_plan_create(GemmPlan **out, int, int, int, int) {
    GemmPlan *p = new GemmPlan();
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, dev);
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn) {
        delete p;
        return false;
    }
    p->encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    if (cudaMalloc(&p->ws, WS_BYTES) != cudaSuccess ||
        cudaMalloc(&p->counters, sizeof(int) * N_COUNTERS) != cudaSuccess ||
        cudaMalloc(&p->stamps, sizeof(unsigned long long) * 3 * ALL_STAMPS) != cudaSuccess ||
        cudaMalloc(&p->slot_acc, sizeof(unsigned long long) * 3 * ALL_STAMPS) != cudaSuccess ||
        cudaMalloc(&p->stamp_acc, sizeof(StampAcc)) != cudaSuccess) {
        gemm_plan_destroy(p);
        return false;
    }
    cudaMemset(p->counters, 0, sizeof(int) * N_COUNTERS);
    *out = p;
    return true;
}

void gemm_plan_destroy(GemmPlan *p) {
    if (!p) return;
    if (p->ws) cudaFree(p->ws);
    if (p->counters) cudaFree(p->counters);
    if (p->stamps) cudaFree(p->stamps);
    if (p->stamp_acc) cudaFree(p->stamp_acc);
    if (p->slot_acc) cudaFree(p->slot_acc);
    for (cudaEvent_t e : p->ev) cudaEventDestroy(e);
    delete p;
}

bool gemm_profile_enable(GemmPlan *p, int mode) {
    p->profile = mode == 1;
    p->stamp_mode = mode == 2;
    p->stamp_active = false;
    p->ev_used = 0;
    p->prof_bytes = p->prof_wbytes = p->prof_flops = p->prof_mma = p->prof_pre = 0.0;
    if (p->stamp_mode) {
        stamp_init_kernel<<<8, 256>>>(p->stamps, ALL_STAMPS, p->stamp_acc, p->slot_acc);
        if (cudaDeviceSynchronize() != cudaSuccess) return false;
    }
    return true;
}

bool gemm_profile_on(const GemmPlan *p) { return p->profile; }
bool gemm_stamp_on(const GemmPlan *p) { return p->stamp_mode; }

void gemm_stamp_begin(GemmPlan *p) {
    if (!p->stamp_mode) return;
    p->stamp_active = true;
    p->stamp_next = 0;
    p->xstamp_next = 0;
    p->cur_slot = -1;
    p->stamp_bytes = p->stamp_wbytes = p->stamp_flops = p->stamp_mma = p->stamp_pre = 0.0;
}

void gemm_stamp_end(GemmPlan *p, cudaStream_t s) {
    if (!p->stamp_active) return;
    p->stamp_active = false;
    p->slot_n = p->stamp_next;
    p->xslot_n = p->xstamp_next;
    stamp_collect_kernel<<<1, 256, 0, s>>>(p->stamps, p->stamp_next, p->xstamp_next, p->stamp_bytes, p->stamp_wbytes,
                                           p->stamp_flops, p->stamp_mma, p->stamp_pre, p->stamp_acc, p->slot_acc);
    note_launch();
}

// The stamp slot of the next launch (null outside a window or when full).
static unsigned long long *stamp_slot(GemmPlan *p) {
    if (!p->stamp_active || p->stamp_next >= MAX_STAMPS) return nullptr;
    p->cur_slot = p->stamp_next;
    return p->stamps + 3 * (p->stamp_next++);
}

unsigned long long *gemm_stamp_external(GemmPlan *p, int kind, int rows, int outputs, int inner) {
    if (!p || !p->stamp_active || p->xstamp_next >= MAX_XSTAMPS) return nullptr;
    const int i = MAX_STAMPS + p->xstamp_next++;
    p->slot_info[i] = GemmSlot{kind, rows, outputs, inner, 0, 0.0, 0.0, 0.0};
    return p->stamps + 3 * i;
}

int gemm_profile_slots(GemmPlan *p, GemmSlot *out, int max) {
    if (!p->stamp_mode) return 0;
    std::vector<unsigned long long> acc(3 * (size_t)ALL_STAMPS);
    cudaDeviceSynchronize();
    if (cudaMemcpy(acc.data(), p->slot_acc, acc.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost) !=
        cudaSuccess)
        return -1;
    cudaMemset(p->slot_acc, 0, acc.size() * sizeof(unsigned long long));
    int n = 0;
    auto put = [&](int i) {
        if (n >= max) return;
        GemmSlot g = p->slot_info[i];
        g.launches = (long)acc[3 * i + 2];
        g.critical_ms = acc[3 * i] * 1e-6;
        g.ms = acc[3 * i + 1] * 1e-6;
        out[n++] = g;
    };
    for (int i = 0; i < p->slot_n; ++i) put(i);
    for (int j = 0; j < p->xslot_n; ++j) put(MAX_STAMPS + j);
    return n;
}

// Algorithmic bytes and flops of a launch of M token rows x O outputs x K for
// the open profile (events or stamps); nb = 2 for split token operands (two
// MMAs per tile); pre = weight bytes its CTAs request before they wait for
// the previous kernel.
static void account(GemmPlan *p, double weight_bytes, double total_bytes, int M, int O, int K, int nb,
                    double pre) {
    const double fl = 2.0 * M * O * K;
    if (p->cur_slot >= 0) {          // the launch that just took a stamp slot
        p->slot_info[p->cur_slot] = GemmSlot{0, M, O, K, 0, total_bytes, 0.0, 0.0};
        p->cur_slot = -1;
    }
    if (p->profile) {
        p->prof_wbytes += weight_bytes;
        p->prof_bytes += total_bytes;
        p->prof_flops += fl;
        p->prof_mma += fl * nb;
        p->prof_pre += pre;
    }
    if (p->stamp_active) {
        p->stamp_wbytes += weight_bytes;
        p->stamp_bytes += total_bytes;
        p->stamp_flops += fl;
        p->stamp_mma += fl * nb;
        p->stamp_pre += pre;
    }
}

GemmProfile gemm_profile_read(GemmPlan *p) {
    GemmProfile r{};
    if (p->stamp_mode) {
        StampAcc a{};
        cudaDeviceSynchronize();
        cudaMemcpy(&a, p->stamp_acc, sizeof a, cudaMemcpyDeviceToHost);
        cudaMemset(p->stamp_acc, 0, sizeof a);
        r.launches = (long)a.launches;
        r.ms = a.span_ns * 1e-6;
        r.critical_ms = a.crit_ns * 1e-6;
        r.windows = (long)a.windows;
        r.bytes = a.bytes;
        r.weight_bytes = a.wbytes;
        r.flops = a.flops;
        r.mma_flops = a.mma_flops;
        r.prefetch_bytes = a.pre_bytes;
        return r;
    }
    r.bytes = p->prof_bytes;
    r.weight_bytes = p->prof_wbytes;
    r.flops = p->prof_flops;
    r.mma_flops = p->prof_mma;
    r.prefetch_bytes = p->prof_pre;
    for (size_t i = 0; i + 1 < p->ev_used; i += 2) {
        float ms = 0.f;
        cudaEventSynchronize(p->ev[i + 1]);
        if (cudaEventElapsedTime(&ms, p->ev[i], p->ev[i + 1]) == cudaSuccess) r.ms += ms;
        r.launches += 1;
    }
    p->ev_used = 0;
    p->prof_bytes = p->prof_wbytes = p->prof_flops = p->prof_mma = p->prof_pre = 0.0;
    return r;
}

static const CUtensorMap *get_map(GemmPlan *p, const void *ptr, long rows, long cols, long ld,
                                  long box_rows, int *status) {
    MapKey key{ptr, rows, cols, ld, box_rows};
    auto it = p->maps.find(key);
    if (it != p->maps.end()) return &it->second;
    CUtensorMap m;
    memset(&m, 0, sizeof m);
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = p->encode(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims,
                           strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) {
        fprintf(stderr, "msd: cuTensorMapEncodeTiled failed (%d) rows=%ld cols=%ld ld=%ld\n", (int)r,
                rows, cols, ld);
        return nullptr;
    }
    return &p->maps.emplace(key, m).first->second;
}

// Tensor map over a packed weight buffer as rows of 64 bf16 (blocks of 128 rows
// are the 16 KB pipeline blocks, already in shared-memory order: no swizzle).
static const CUtensorMap *get_wmap(GemmPlan *p, const void *packed, long rows) {
    MapKey key{packed, rows, BK, -1, BM};
    auto it = p->maps.find(key);
    if (it != p->maps.end()) return &it->second;
    CUtensorMap m;
    memset(&m, 0, sizeof m);
    cuuint64_t dims[2] = {(cuuint64_t)BK, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)BK * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)BM};
    cuuint32_t estr[2] = {1, 1};
    if (p->encode(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(packed), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
        fprintf(stderr, "msd: cuTensorMapEncodeTiled failed for packed weights (%ld rows)\n", rows);
        return nullptr;
    }
    return &p->maps.emplace(key, m).first->second;
}

size_t gemm_pack_bytes(const GemmW &W, int K) {
    long long tiles = 0;
    for (int i = 0; i < W.nseg; ++i) tiles += (W.rows[i] + BM - 1) / BM;
    return (size_t)tiles * ((K + BK - 1) / BK) * A_BYTES;
}

void gemm_pack(const GemmW &W, int K, void *dst, cudaStream_t s) {
    const long long blocks = (long long)(gemm_pack_bytes(W, K) / A_BYTES);
    if (blocks <= 0) return;
    pack_kernel<<<(unsigned)blocks, 256, 0, s>>>(W, K, (K + BK - 1) / BK, static_cast<uint8_t *>(dst));
    note_launch();
}

size_t gemm_pack_glu_bytes(int F, int K) {
    return (size_t)((F + 63) / 64) * ((K + BK - 1) / BK) * A_BYTES;
}

void gemm_pack_glu(const void *gate, const void *up, int F, int K, void *dst, cudaStream_t s) {
    const long long blocks = (long long)(gemm_pack_glu_bytes(F, K) / A_BYTES);
    if (blocks <= 0) return;
    pack_glu_kernel<<<(unsigned)blocks, 256, 0, s>>>(static_cast<const bf16 *>(gate),
                                                      static_cast<const bf16 *>(up), F, K,
                                                      (K + BK - 1) / BK, static_cast<uint8_t *>(dst));
    note_launch();
}

// Launch of the cluster split-K kernel: s K-splits per tile (a cluster), chosen
// so that tiles * s fills the CTAs the SMs hold at once, s <= 8 and >= 2
// K-blocks each. Two CTAs share an SM when three stages fit in half of its
// shared memory (token tiles of up to 64 split rows), otherwise one with up to
// four stages; the split count keeps every split's partial slices within the
// stage memory they reuse.
static void gemm_cluster(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W,
                         int tiles, int BN, int kblocks, float *Y, int ldy, int epi, int *status,
                         cudaStream_t s, int O, const GemmFused *fx = nullptr,
                         const GemmNorm *nout = nullptr, const GemmNorm *nin = nullptr) {
    CkParams ck;
    memset(&ck, 0, sizeof ck);
    if (fx) ck.fx = *fx;
    if (nout) ck.nout = *nout;
    if (nin) ck.nin = *nin;
    ck.n_seg = W.nseg;
    int out_off = 0;
    for (int i = 0; i < W.nseg; ++i) {
        ck.seg_rows[i] = W.rows[i];
        ck.seg_tiles[i] = (W.rows[i] + BM - 1) / BM;
        ck.seg_out[i] = out_off;
        out_off += W.rows[i];
    }
    const int nb = X_lo ? 2 : 1;
    size_t stage = A_BYTES + (size_t)nb * BN * BK * 2;
    constexpr size_t HALF_SM = 104u * 1024u, FULL_SM = 200u * 1024u;
    const int per_sm = 3 * stage <= HALF_SM ? 2 : 1;
    int stages = (int)((per_sm == 2 ? HALF_SM : FULL_SM) / stage);
    stages = std::max(2, std::min(stages, C_STAGES));
    int S = (per_sm * p->num_sms) / tiles;
    S = std::max(1, std::min(S, 8));
    while (S > 1 && kblocks / S < 2) --S;
    // own partial [BN][128] fp32 plus the other ranks' slices of this rank's columns
    while (S > 1 && (size_t)BN * BM * 4 + (size_t)(S - 1) * ((BN + S - 1) / S) * BM * 4 > stages * stage) --S;
    // Two-SM tiles for unsplit launches whose token stage is as large as the
    // weight block (split token rows, 32 or more): each CTA of a pair holds
    // half the token columns, so the ring gets a fourth stage.
    const bool pair = S == 1 && nb == 2 && BN >= 32 && tiles % 2 == 0 && per_sm == 2;
    const int BNs = pair ? BN / 2 : BN;
    if (pair) {
        stage = A_BYTES + (size_t)nb * BNs * BK * 2;
        stages = std::max(2, std::min((int)(HALF_SM / stage), C_STAGES));
    }
    ck.M = M;
    ck.kblocks = kblocks;
    ck.BN = BN;
    ck.n_tiles_n = 1;
    ck.splits = S;
    ck.stages = stages;
    ck.has_lo = X_lo ? 1 : 0;
    ck.tmem_cols = BN <= 32 ? 32 : (BN <= 64 ? 64 : 128);
    ck.wpacked = static_cast<const bf16 *>(W.packed);
    ck.Y = Y;
    ck.ldy = ldy;
    ck.epi = epi;
    ck.status = status;
    const CUtensorMap *mx = get_map(p, X, M, K, ldx, BNs, status);
    ck.stamp = stamp_slot(p);
    const CUtensorMap *mxl = X_lo ? get_map(p, X_lo, M, K, ldx, BNs, status) : mx;
    const CUtensorMap *mw = pair ? get_wmap(p, W.packed, (long)tiles * kblocks * BM) : mx;
    if (!mx || !mxl || !mw) return;
    const size_t smem = 1024 + (size_t)stages * stage;
    if (!p->cluster_attr_set) {
        cudaFuncSetAttribute(gemm_cluster_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(1024 + FULL_SM));
        cudaFuncSetAttribute(gemm_cluster_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(1024 + FULL_SM));
        p->cluster_attr_set = true;
    }
    const bool prof = p->profile;
    if (prof) {
        while (p->ev.size() < p->ev_used + 2) {
            cudaEvent_t e;
            cudaEventCreate(&e);
            p->ev.push_back(e);
        }
        cudaEventRecord(p->ev[p->ev_used], s);
    }
    cudaLaunchConfig_t lc;
    memset(&lc, 0, sizeof lc);
    lc.gridDim = dim3((unsigned)tiles, 1, (unsigned)S);
    lc.blockDim = dim3(C_THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = pair ? 2u : 1u;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = (unsigned)S;
    lc.attrs = at;
    lc.numAttrs = 2;
    if ((pair ? cudaLaunchKernelEx(&lc, gemm_cluster_kernel<true>, *mx, *mxl, *mw, ck)
              : cudaLaunchKernelEx(&lc, gemm_cluster_kernel<false>, *mx, *mxl, *mw, ck)) != cudaSuccess) {
        cudaGetLastError();
        flag_kernel<<<1, 1, 0, s>>>(status, ST_RANGE);
        fprintf(stderr, "msd: cluster GEMM launch failed (M=%d K=%d O=%d S=%d)\n", M, K, O, S);
    }
    note_launch();
    if (prof) {
        cudaEventRecord(p->ev[p->ev_used + 1], s);
        p->ev_used += 2;
    }
    const double wb = (double)O * K * 2.0;
    double yb = (double)M * O * 4.0 * (epi == EPI_ADD ? 2 : 1);
    if (epi == EPI_SWIGLU) yb = (double)M * fx->F * 2.0 * nb;
    if (epi == EPI_ROPE_KV) yb = (double)M * O * 2.0 * nb;
    double pre = 0.0;      // the blocks each split requests before its wait (padded rows included)
    for (int z = 0; z < S; ++z)
        pre += (double)tiles * std::min(stages, (int)((long long)(z + 1) * kblocks / S - (long long)z * kblocks / S)) *
               A_BYTES;
    account(p, wb, wb + (double)M * K * 2.0 * nb + yb, M, O, K, nb, std::min(pre, wb));
}

// The persistent stream-K GEMM (many token rows). fx: EPI_SWIGLU writes
// act = silu(g) * u from glu-packed gate/up weights instead of Y.
static void gemm_persist(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W,
                         int O, float *Y, int ldy, int epi, const GemmFused *fx, int *status, cudaStream_t s);

bool gemm_bf16_fused(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W,
                     int O, const GemmFused &fx, int *status, cudaStream_t s, const GemmNorm *norm_in) {
    if (M <= 0 || !W.packed || W.nseg < 1) return false;
    if (fx.epi == EPI_SWIGLU && (W.nseg != 1 || W.rows[0] != glu_rows(fx.F) || fx.F % 4)) return false;
    if (M > 128) {
        // many token rows: the persistent GEMM with SwiGLU fused into its
        // epilogue (RoPE/KV stays a separate kernel there: fused, its
        // per-column gathers outlasted the main loop, measured slower)
        if (fx.epi != EPI_SWIGLU || norm_in || !fx.act) return false;
        gemm_persist(p, X, X_lo, ldx, M, K, W, O, nullptr, 0, EPI_SWIGLU, &fx, status, s);
        return true;
    }
    if (fx.epi == EPI_ROPE_KV &&
        (W.nseg != 3 || (fx.hd != 64 && fx.hd != 128) || fx.nh * fx.hd != W.rows[0] ||
         W.rows[1] != W.rows[0] || W.rows[2] != W.rows[0]))
        return false;
    if (fx.epi != EPI_SWIGLU && fx.epi != EPI_ROPE_KV) return false;
    int tiles = 0;
    for (int i = 0; i < W.nseg; ++i) tiles += (W.rows[i] + BM - 1) / BM;
    const int BN = ((M + 15) / 16) * 16;
    if (norm_in && (!norm_in->ss || norm_in->parts <= 0 || norm_in->parts > norm_in->ld || BN > 128))
        return false;
    gemm_cluster(p, X, X_lo, ldx, M, K, W, tiles, BN, (K + BK - 1) / BK, nullptr, 0, fx.epi, status, s, O, &fx,
                 nullptr, norm_in);
    return true;
}

bool gemm_bf16(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W, int O,
               float *Y, int ldy, int epi, int *status, cudaStream_t s, const GemmNorm *norm_out) {
    if (M <= 0 || O <= 0) return true;
    if (norm_out && (M > 128 || !W.packed || W.nseg != 1 || !norm_out->ss || !norm_out->xg || !norm_out->g ||
                     (O + BM - 1) / BM > norm_out->ld || O % 4 || ldy % 4))
        return false;
    if (M <= 128 && W.packed) {
        int tiles = 0;
        for (int i = 0; i < W.nseg; ++i) tiles += (W.rows[i] + BM - 1) / BM;
        gemm_cluster(p, X, X_lo, ldx, M, K, W, tiles, ((M + 15) / 16) * 16, (K + BK - 1) / BK, Y, ldy, epi,
                     status, s, O, nullptr, norm_out);
        return true;
    }
    gemm_persist(p, X, X_lo, ldx, M, K, W, O, Y, ldy, epi, nullptr, status, s);
    return true;
}

static void gemm_persist(GemmPlan *p, const bf16 *X, const bf16 *X_lo, int ldx, int M, int K, const GemmW &W,
                         int O, float *Y, int ldy, int epi, const GemmFused *fx, int *status, cudaStream_t s) {
    const bool glu = fx && fx->epi == EPI_SWIGLU;
    PkParams pk;
    memset(&pk, 0, sizeof pk);
    pk.n_seg = W.nseg;
    int tiles = 0, out_off = 0;
    for (int i = 0; i < W.nseg; ++i) {
        pk.seg_rows[i] = W.rows[i];
        pk.seg_tiles[i] = (W.rows[i] + BM - 1) / BM;
        pk.seg_out[i] = out_off;
        out_off += W.rows[i];
        tiles += pk.seg_tiles[i];
    }
    const int nb = X_lo ? 2 : 1;
    // the fused SwiGLU epilogue takes 16 KB of staging from the ring's budget
    const uint32_t stg_bytes = glu ? 32u * BM * 4u : 0u;
    constexpr uint32_t BUDGET = 208u * 1024u;
    // token tiles: the widest (fewest tiles, most weight reuse) that keeps three
    // stages in shared memory; five stages measured best on decode shapes
    int nt = (M + 255) / 256, BN = 0;
    for (;; ++nt) {
        BN = ((M + nt - 1) / nt + 15) / 16 * 16;
        const uint32_t st = A_BYTES + (uint32_t)nb * BN * BK * 2;
        if (3u * st + stg_bytes <= BUDGET || BN <= 16) break;
    }
    const int kblocks = (K + BK - 1) / BK;
    const uint32_t stage_bytes = A_BYTES + (uint32_t)nb * BN * BK * 2;
    int stages = (int)((BUDGET - stg_bytes) / stage_bytes);
    stages = stages < 2 ? 2 : (stages > 5 ? 5 : stages);
    const size_t smem = 1024 + (size_t)stages * stage_bytes + stg_bytes;
    const long long tiles_total = (long long)tiles * nt;
    const long long all_units = tiles_total * kblocks;
    // one CTA per SM, at least 4 K-blocks each
    long long G = all_units / 4;
    if (G > p->num_sms) G = p->num_sms;
    if (G < 1) G = 1;
    // whole tiles in rounds of G, the remainder split stream-K across all CTAs
    // (its fix-ups overlap the whole tiles that follow). A remainder of a few
    // short-K tiles would cut each into more than eight pieces, summed by one
    // CTA: there one round of whole tiles joins it (every tile in two or three
    // pieces, fixed up at the end). Measured on the 960-row verify GEMMs: O
    // (K = 4096) 89 -> 75 us; down (K = 11008) 106 -> 140 us and the SwiGLU
    // launches slower, so those keep the rounds.
    int dp_rounds = (int)(tiles_total / G);
    int T_sk = (int)(tiles_total - (long long)dp_rounds * G);
    if (T_sk > 0 && dp_rounds > 0 && G > 8LL * T_sk && kblocks <= 64 && !glu) {
        --dp_rounds;
        T_sk += (int)G;
    }
    const long long units = (long long)T_sk * kblocks;
    const size_t ws_need = 2ull * G * BN * BM * sizeof(float);
    if (ws_need > WS_BYTES || tiles_total > N_COUNTERS) {
        flag_kernel<<<1, 1, 0, s>>>(status, ST_RANGE);
        fprintf(stderr, "msd: GEMM shape M=%d K=%d O=%d exceeds the workspace\n", M, K, O);
        return;
    }
    int acc = 32;
    while (acc < BN) acc <<= 1;
    pk.M = M;
    pk.kblocks = kblocks;
    pk.BN = BN;
    pk.n_tiles_n = nt;
    pk.stages = stages;
    pk.acc_stride = acc;
    pk.tmem_cols = 2 * acc;
    pk.grid = (int)G;
    pk.units = units;
    pk.T_sk = T_sk;
    pk.dp_rounds = dp_rounds;
    pk.Y = Y;
    pk.ldy = ldy;
    pk.epi = epi;
    pk.ws = p->ws;
    pk.counters = p->counters;
    pk.status = status;
    pk.wpacked = static_cast<const bf16 *>(W.packed);
    pk.has_lo = X_lo ? 1 : 0;
    if (glu) {
        pk.epi = EPI_SWIGLU;
        pk.act = fx->act;
        pk.F = fx->F;
        pk.lo = fx->lo;
        pk.stg_off = (uint32_t)(1024 + (size_t)stages * stage_bytes);
    }
    if (!W.packed) {
        flag_kernel<<<1, 1, 0, s>>>(status, ST_RANGE);
        fprintf(stderr, "msd: GEMM weights were not packed\n");
        return;
    }
    const CUtensorMap *mx = get_map(p, X, M, K, ldx, BN, status);
    const CUtensorMap *mxl = X_lo ? get_map(p, X_lo, M, K, ldx, BN, status) : mx;
    if (!mx || !mxl) return;
    pk.stamp = stamp_slot(p);
    if (!p->smem_set) {
        cudaFuncSetAttribute(gemm_persist_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(BUDGET + 1024));
        p->smem_set = true;
    }
    const bool prof = p->profile;
    if (prof) {
        while (p->ev.size() < p->ev_used + 2) {
            cudaEvent_t e;
            cudaEventCreate(&e);
            p->ev.push_back(e);
        }
        cudaEventRecord(p->ev[p->ev_used], s);
    }
    // Programmatic dependent launch: the kernel may start while the previous
    // kernel on the stream finishes; it waits (griddepcontrol.wait) before
    // touching anything but weights.
    cudaLaunchConfig_t lc;
    memset(&lc, 0, sizeof lc);
    lc.gridDim = dim3((unsigned)G);
    lc.blockDim = dim3(P_THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = at;
    lc.numAttrs = 1;
    cudaLaunchKernelEx(&lc, gemm_persist_kernel, *mx, *mxl, pk);
    note_launch();
    if (prof) {
        cudaEventRecord(p->ev[p->ev_used + 1], s);
        p->ev_used += 2;
    }
    const double wb = (double)O * K * 2.0;
    account(p, wb, wb + (double)M * K * 2.0 * nb +
                       (glu ? (double)M * fx->F * 2.0 * nb : (double)M * O * 4.0 * (epi == EPI_ADD ? 2 : 1)),
            M, O, K, nb, std::min(wb, (double)G * std::min<long long>(stages, all_units / G) * A_BYTES));
}

}  // namespace msd

// ---------------------------------------------------------------------------
// Allocation-free GEMM entry point (msd_linear_noalloc in include/msd.h).
//
// Some callers cannot call cudaMalloc: a host program whose device memory is
// entirely owned by its own pool allocator, code that runs where an allocation
// would synchronise the device or is not permitted, or a plug-in that is handed
// buffers but no allocator. For them the split-K scratch of the tensor-core
// GEMM lives in one file-scope device array, loaded with the library and held
// by every GPU that loads it until the process exits.
//
// Layout of the array: a status word (padded to 256 bytes), NOALLOC_COUNTERS
// int tile tickets, then the fp32 split-K partials (NOALLOC_PARTIAL_BYTES). In
// host code the array's name is only a host-side stand-in; the device address
// comes from cudaGetSymbolAddress, taken once per device (with that device
// current) on the first call made on it. Every call shares the array and it
// keeps the last call's contents: the tickets are cleared on the caller's
// stream before each launch that uses them, and calls that overlap on the GPU
// race on the array. The split-K choice is limited to what the array holds, so
// a shape that would split further on the context GEMM runs with fewer splits
// (none at worst) instead of being refused.
// ---------------------------------------------------------------------------
namespace msd {
namespace {
constexpr size_t NOALLOC_STATUS_BYTES = 256;
constexpr int NOALLOC_COUNTERS = 4096;
constexpr size_t NOALLOC_PARTIAL_BYTES = 16ull << 20;
constexpr size_t NOALLOC_BYTES = NOALLOC_STATUS_BYTES + NOALLOC_COUNTERS * sizeof(int) + NOALLOC_PARTIAL_BYTES;
constexpr int NOALLOC_MAX_DEVICES = 64;
constexpr size_t NOALLOC_MAX_MAPS = 256;   // cached weight tensor maps per process
constexpr long NOALLOC_MAX_ROWS = 65535L * 256;   // token-tile grid dimension limit
}  // namespace

static __device__ __align__(256) unsigned char g_noalloc_scratch[NOALLOC_BYTES];

namespace {
struct NoAllocDevice {
    bool ready = false;
    unsigned char *scratch = nullptr;   // device address of g_noalloc_scratch
    int num_sms = 0;
    int status_host = 0;                // last value read back from the status word
};
std::mutex g_noalloc_mu;
NoAllocDevice g_noalloc_dev[NOALLOC_MAX_DEVICES];
GemmPlan g_noalloc_maps;                // host-side tensor-map cache only (no device memory)

// One-time set-up of the current device (caller holds g_noalloc_mu).
bool noalloc_setup(int dev) {
    NoAllocDevice &d = g_noalloc_dev[dev];
    if (d.ready) return true;
    void *ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_noalloc_scratch) != cudaSuccess || !ptr) return false;
    if (cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
    if (cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024 + 1024) !=
        cudaSuccess)
        return false;
    if (!g_noalloc_maps.encode) {
        cudaDriverEntryPointQueryResult q;
        void *fn = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !fn)
            return false;
        g_noalloc_maps.encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    d.scratch = static_cast<unsigned char *>(ptr);
    d.ready = true;
    return true;
}

// Tensor map of an activation operand: encoded on every call (a host-only
// computation), so the cache holds weight maps alone.
bool encode_x_map(const void *x, long rows, long cols, long ld, long box_rows, CUtensorMap *m) {
    memset(m, 0, sizeof *m);
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return g_noalloc_maps.encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(x), dims, strides, box,
                                 estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}
}  // namespace

// Device address of the no-alloc status word on the current device (set-up
// included); null if the set-up failed.
int *noalloc_status_word() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= NOALLOC_MAX_DEVICES) return nullptr;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!noalloc_setup(dev)) return nullptr;
    return reinterpret_cast<int *>(g_noalloc_dev[dev].scratch);
}

// Test hook of the bounded waits: one CTA waits on an mbarrier that nothing
// arrives at, through the same bounded wait as the GEMM kernels, gives up
// after limit_ns and records ST_TIMEOUT in *status. No copy or MMA is in
// flight while it waits.
__global__ void wait_probe_kernel(int *status, unsigned long long limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ volatile int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        mbar_wait(smem_u32(&bar), 0, &abort_flag, status, limit_ns);
    }
}

bool launch_wait_probe(int *status, long long limit_ns, cudaStream_t s) {
    wait_probe_kernel<<<1, 32, 0, s>>>(status, (unsigned long long)limit_ns);
    note_launch();
    return cudaGetLastError() == cudaSuccess;
}

}  // namespace msd

extern "C" msd_status msd_linear_noalloc(const void *x, int32_t ldx, int32_t m, int32_t k,
                                         const void *w, int32_t o, float *y, int32_t ldy,
                                         int32_t accumulate, void *stream) {
    using namespace msd;
    constexpr msd_status OK = MSD_OK, INVALID = MSD_ERR_INVALID, CAPACITY = MSD_ERR_CAPACITY,
                         CUDA_ERR = MSD_ERR_CUDA, DEVICE = MSD_ERR_DEVICE;
    if (!x || !w || !y || m <= 0 || k <= 0 || o <= 0 || ldx < k || ldy < o) return INVALID;
    if (ldx % 8 || k % 8) return INVALID;
    if ((long)m > NOALLOC_MAX_ROWS) return CAPACITY;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= NOALLOC_MAX_DEVICES) return CUDA_ERR;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!noalloc_setup(dev)) return CUDA_ERR;
    NoAllocDevice &d = g_noalloc_dev[dev];
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int *status = reinterpret_cast<int *>(d.scratch);
    // The status word left by earlier launches on this device (a bounded wait
    // that ran out): read back into pageable host memory, so the copy returns
    // once the work queued before it on `stream` has finished; a set word is
    // cleared and reported once.
    if (cudaMemcpyAsync(&d.status_host, status, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return CUDA_ERR;
    if (cudaStreamSynchronize(s) != cudaSuccess) return CUDA_ERR;
    if (d.status_host != 0) {
        d.status_host = 0;
        if (cudaMemsetAsync(status, 0, sizeof(int), s) != cudaSuccess) return CUDA_ERR;
        return DEVICE;
    }
    // The same tile shape and stages as the context GEMM; the split-K choice is
    // limited to what the array holds.
    const int M = m, K = k, O = o;
    const int tiles = (O + BM - 1) / BM;
    const int nt = (M + 255) / 256;
    int BN = (M + nt - 1) / nt;
    BN = ((BN + 15) / 16) * 16;
    const int kblocks = (K + BK - 1) / BK;
    const uint32_t stage_bytes = A_BYTES + (uint32_t)BN * BK * 2;
    const int ctas_per_sm = BN <= 128 ? 2 : 1;
    int stages = (int)((ctas_per_sm == 2 ? 100u * 1024u : 200u * 1024u) / stage_bytes);
    stages = stages < 2 ? 2 : (stages > MAX_STAGES ? MAX_STAGES : stages);
    const size_t smem = 1024 + (size_t)stages * stage_bytes;
    const long base = (long)tiles * nt;
    const long slots = (long)d.num_sms * ctas_per_sm;
    const size_t tile_bytes = (size_t)BN * BM * sizeof(float);
    int best_s = 1;
    double best = 1e30;
    for (int sp = 1; sp <= 16 && sp <= kblocks; ++sp) {
        const int kps = (kblocks + sp - 1) / sp;
        const int se = (kblocks + kps - 1) / kps;
        if (se > 1 && ((size_t)base * se * tile_bytes > NOALLOC_PARTIAL_BYTES || base > NOALLOC_COUNTERS))
            continue;
        const long waves = (base * se + slots - 1) / slots;
        const double cost = (double)waves * kps + (se > 1 ? 2.0 : 0.0);
        if (cost < best - 1e-9) { best = cost; best_s = se; }
    }
    const int kps = (kblocks + best_s - 1) / best_s;
    const int splits = (kblocks + kps - 1) / kps;

    TcParams tp;
    memset(&tp, 0, sizeof tp);
    tp.n_seg = 1;
    tp.seg_tiles[0] = tiles;
    tp.seg_rows[0] = O;
    tp.seg_out[0] = 0;
    tp.M = M;
    tp.kblocks = kblocks;
    tp.splits = splits;
    tp.kb_per_split = kps;
    tp.BN = BN;
    tp.n_tiles_n = nt;
    tp.stages = stages;
    tp.tmem_cols = BN <= 32 ? 32 : (BN <= 64 ? 64 : (BN <= 128 ? 128 : 256));
    tp.Y = y;
    tp.ldy = ldy;
    tp.epi = accumulate ? EPI_ADD : EPI_STORE;
    tp.counters = reinterpret_cast<int *>(d.scratch + NOALLOC_STATUS_BYTES);
    tp.ws = reinterpret_cast<float *>(d.scratch + NOALLOC_STATUS_BYTES + NOALLOC_COUNTERS * sizeof(int));
    tp.status = status;
    if (g_noalloc_maps.maps.size() >= NOALLOC_MAX_MAPS) g_noalloc_maps.maps.clear();
    const CUtensorMap *mw = get_map(&g_noalloc_maps, w, O, K, K, BM, nullptr);
    CUtensorMap mx;
    if (!mw || !encode_x_map(x, M, K, ldx, BN, &mx)) return INVALID;
    if (splits > 1 && cudaMemsetAsync(tp.counters, 0, sizeof(int) * base, s) != cudaSuccess)
        return CUDA_ERR;
    gemm_tc_kernel<<<dim3(tiles, nt, splits), THREADS, smem, s>>>(*mw, *mw, *mw, mx, tp);
    note_launch();
    return cudaGetLastError() == cudaSuccess ? OK : CUDA_ERR;
}
