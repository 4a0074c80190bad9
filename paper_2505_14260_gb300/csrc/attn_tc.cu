// Tree-masked attention on the 5th-generation tensor cores (bf16 contexts).
//
// Every operand is a split bf16 pair (hi + lo, common.cuh), so both products
// run as three tcgen05.mma each into one fp32 accumulator in tensor memory:
//   S = Q K^T  as  Qh Kh + Ql Kh + Qh Kl
//   O += P V   as  Ph Vh + Pl Vh + Ph Vl
// (the dropped lo*lo terms are 2^-18 of the product), which keeps the
// attention as precise as an fp32 evaluation.
//
// A CTA takes 64 query rows of one request and one head (the MMA's M = 64)
// and one range of keys (a split). Roles (320 threads):
//   warp 0 lane 0   TMA: K and V tiles of 64 keys (hi and lo planes, 128-byte
//                   swizzle) into a three-stage shared-memory ring
//   warp 1          allocates tensor memory; lane 0 issues the MMAs
//   warps 2-9       two per TMEM lane quarter (an M = 64 accumulator keeps
//                   rows 16q .. 16q+15 in lanes 0-15 of quarter q), each
//                   taking half of a tile's keys and of O's columns: load the
//                   query rows into TMEM, then per key tile read S, mask it
//                   (prefix length, tree bitmask), run the online softmax in
//                   base 2 and write P (hi, lo) back over S as the A operand
//                   of the P V product
// Q and P are A operands read from tensor memory (P of a tile's keys 32h ..
// 32h+31 written over those keys' S columns, hi pairs then lo pairs, by the
// warps that read them), so shared memory holds only the K/V ring; S is
// double-buffered so the Q K^T of tile j+1 overlaps the softmax of tile j. O stays in TMEM; a row's running maximum is moved (and O
// and the row sum rescaled) only when a tile's maximum exceeds it by more than
// 2^8, so P <= 256.
//
// Visible keys of a row (Sec. 3.2: a candidate is conditioned on its prefix
// only): cache positions [0, plen) of its request, and tree slots whose bit is
// set in its mask. The live prefix is cut into splits of whole key tiles (their
// count a function of the launch's shape, so a result depends on L alone), the
// last split also taking the tree slots; the splits
// of a (row tile, head) form a thread-block cluster and combine their
// partials (O, max, sum) through distributed shared memory in split order:
// deterministic. Every mbarrier wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <unordered_map>

#include "attn_tc.h"

namespace msd {

namespace {

constexpr int ROWS = 64;          // query rows per CTA (MMA M)
constexpr int KT = 64;            // keys per tile (N of Q K^T, K of P V)
constexpr int THREADS = 320;      // warp 0 TMA, warp 1 MMA, warps 2-9 softmax
constexpr int STAGES = 3;
constexpr int MAX_SPLITS = 9;     // splits of a (row tile, head) = cluster size
constexpr int ORDER_MAX = 64;     // request blocks a launch can reorder
constexpr unsigned long long ATTN_TIMEOUT_NS = 2000000000ull;
constexpr float RESCALE_LOG2 = 8.f;

template <int HD>
struct Lay {
    static constexpr int NB = HD / 64;                    // 64-column boxes of a row
    static constexpr uint32_t BOX = KT * 128;             // [64 rows][64 bf16] = 8 KB
    static constexpr uint32_t TILE = NB * BOX;            // one plane of a K or V tile
    static constexpr uint32_t STAGE = 4 * TILE;           // K hi, K lo, V hi, V lo
    // tensor-memory columns: Q hi, Q lo (bf16 pairs), two S/P buffers, O
    static constexpr uint32_t T_QH = 0, T_QL = HD / 2, T_S = HD, T_O = HD + 2 * KT;
    static constexpr uint32_t T_COLS = T_O + HD <= 256 ? 256 : 512;
    static constexpr int LD = HD + 4;                     // fp32 partial row stride (floats)
};

struct AttnTcParams {
    const bf16 *q;
    const RowDesc *rows;
    const uint64_t *mask;
    bf16 *out;
    long lo;                  // lo planes of q and out (elements); K/V: lo_rows rows on
    int lo_rows;
    int *status;
    int R, rows_per_req, tiles_per_req, nh, cache_slots, tree_slots, mask_words;
    int nsplit, has_tree;     // splits of the live prefix; the tree keys follow in the last one
    int cache_early;          // cache K/V may be requested before the wait (not written by the previous kernel)
    float scale_log2;
    unsigned long long *stamp;   // profiling: earliest entry, earliest return from the wait, latest exit (ns)
    int n_order;              // > 0: row-tile blocks launch in this order (longest request first)
    uint8_t order[ORDER_MAX];
};

__device__ __forceinline__ uint32_t su32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ unsigned long long gtime() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ bool bar_try(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        "selp.b32 %0, 1, 0, p;\n}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: gives up when *abort is set by another thread, or after the
// limit (then sets *abort and records ST_TIMEOUT).
__device__ bool bar_wait(uint32_t bar, uint32_t parity, volatile int *abort, int *status) {
    if (bar_try(bar, parity)) return true;
    const unsigned long long t0 = gtime();
    while (!bar_try(bar, parity)) {
        if (*abort) return false;
        if (gtime() - t0 > ATTN_TIMEOUT_NS) {
            *abort = 1;
            set_status(status, ST_TIMEOUT);
            return false;
        }
    }
    return true;
}

__device__ __forceinline__ void bar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}
__device__ __forceinline__ void bar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void bar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void tma2d(uint32_t dst, const CUtensorMap *m, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(m), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// Shared-memory matrix descriptor (sm100 version 1, 128-byte swizzle): start
// address, leading byte offset (MN-major: the stride between 64-element
// atoms along M/N) and stride byte offset (the stride between 8-row groups).
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor, kind::f16: fp32 accumulate, bf16 A and B, A
// K-major, B K-major (b_mn = 0) or MN-major (1).
__device__ __forceinline__ uint32_t idesc(int M, int N, int b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)b_mn << 16) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}

// D (+)= A B^T with A read from tensor memory and B from shared memory.
__device__ __forceinline__ void mma_ts(uint32_t d, uint32_t a, uint64_t b, uint32_t id, uint32_t acc) {
    asm volatile(
        "{\n.reg .pred p;\nsetp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}" ::"r"(d),
        "r"(a), "l"(b), "r"(id), "r"(acc));
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// 32 columns of this warp's lanes, waited for in the same asm statement: the
// compiler sees the registers defined only once the data has landed.
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


// Stores of 32 / 16 columns, waited for in the same asm statement, so the
// source registers are not reused before the tensor memory has taken them.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t *r) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n"
        "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
        "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
        "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t *r) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};\n"
        "tcgen05.wait::st.sync.aligned;" ::"r"(taddr),
        "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
        "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
        : "memory");
}

// Barrier of the two softmax warps that share TMEM lane quarter q (named
// barrier 1 + q, 64 threads; no other warp joins it): they exchange their
// rows' tile maxima and sums through shared memory. The warp reconverges
// first: the barrier's aligned form needs every lane of a warp to reach it
// together.
__device__ __forceinline__ void softmax_sync(int quarter) {
    __syncwarp();
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    asm volatile("barrier.sync.aligned %0, 64;" ::"r"(1 + quarter) : "memory");
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// 2^x (the SFU approximation; 2^-inf = 0)
__device__ __forceinline__ float ex2_fast(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ uint32_t dsmem_addr(uint32_t local, int rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}

// (no memory clobber: the partials are read only between two cluster
// barriers, themselves compiler barriers, so the loads may overlap)
__device__ __forceinline__ float2 dsmem_ld_f2(uint32_t a) {
    float2 v;
    asm volatile("ld.shared::cluster.v2.f32 {%0,%1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(a));
    return v;
}

__device__ __forceinline__ float4 dsmem_ld_f4(uint32_t a) {
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(a));
    return v;
}

// hi and lo bf16 pairs of two fp32 values (element 2c in the low half).
__device__ __forceinline__ void split_pair(float a, float b, uint32_t &hi, uint32_t &lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    const __nv_bfloat162 l = __floats2bfloat162_rn(a - __low2float(h), b - __high2float(h));
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}

template <int HD>
__global__ void __launch_bounds__(THREADS, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap mkc, const __grid_constant__ CUtensorMap mvc,
                   const __grid_constant__ CUtensorMap mkt, const __grid_constant__ CUtensorMap mvt,
                   const AttnTcParams p) {
    using L = Lay<HD>;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[2 * STAGES + 8];
    __shared__ uint32_t tmem_base;
    __shared__ int s_pmax;
    __shared__ volatile int abort_flag;
    __shared__ float s_xmax[6 * ROWS];     // tile maxima [tile parity][half][row], then row sums [half][row]

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0 && p.stamp) atomicMin(p.stamp, gtime());
    // heads vary fastest in the launch order, then row tiles, request blocks in
    // p.order (the CTAs of the longest requests start first)
    const int h = blockIdx.x, tile = blockIdx.y, split = blockIdx.z;
    const int pos = tile / p.tiles_per_req;
    const int blk = p.n_order > 0 ? (int)p.order[pos] : pos;
    const int r0 = blk * p.rows_per_req + (tile - pos * p.tiles_per_req) * ROWS;
    const int r_end = min(r0 + ROWS, (blk + 1) * p.rows_per_req);
    const int H = p.nh * HD;

    const uint32_t base = (su32(smem_raw) + 1023u) & ~1023u;
    const uint32_t full0 = su32(&bars[0]), empty0 = su32(&bars[STAGES]);
    const uint32_t s_full0 = su32(&bars[2 * STAGES]), p_full0 = su32(&bars[2 * STAGES + 2]);
    const uint32_t o_ready = su32(&bars[2 * STAGES + 4]), q_ready = su32(&bars[2 * STAGES + 5]);
    const uint32_t drain = su32(&bars[2 * STAGES + 6]);

    // softmax threads: warps 2-9 read TMEM lane quarter q = warp & 3, whose
    // lanes 0-15 hold rows 16q .. 16q+15 of the M = 64 accumulators
    const bool smx = warp >= 2;
    const int quarter = warp & 3;
    const int row_local = 16 * quarter + lane;
    const int row = r0 + row_local;
    const bool valid = smx && lane < 16 && row < r_end;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            bar_init(full0 + 8 * s, 1);
            bar_init(empty0 + 8 * s, 1);
        }
        for (int b = 0; b < 2; ++b) {
            bar_init(s_full0 + 8 * b, 1);
            bar_init(p_full0 + 8 * b, 256);
        }
        bar_init(o_ready, 1);
        bar_init(q_ready, 256);
        bar_init(drain, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        s_pmax = 0;
        abort_flag = 0;
        asm volatile("prefetch.tensormap [%0];" ::"l"(&mkc) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(&mvc) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(su32(&tmem_base)),
                     "r"(L::T_COLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    __syncthreads();
    // Before the wait: the row descriptors (written by set-up kernels at least
    // two launches back) and, unless the previous kernel wrote into it, the
    // cache K/V. The previous kernel's q and tree K/V are read after the wait.
    const int req = p.rows[r0].req;
    const int plen = valid ? p.rows[row].plen : 0;
    if (valid) atomicMax(&s_pmax, plen);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;

    // Key range of this split. The request's live prefix is cut into nsplit
    // equal runs of whole 64-key tiles (nsplit depends only on the launch's
    // shape, so a result depends on L alone); the last split, whose run is the
    // shortest, takes the tree keys after its cache keys.
    const int live = min(s_pmax, p.cache_slots);
    const int per_split = ((live + KT - 1) / KT + p.nsplit - 1) / p.nsplit * KT;
    const int k_lo = split * per_split, k_hi = min(k_lo + per_split, live);
    const int nc = k_hi > k_lo ? (k_hi - k_lo + KT - 1) / KT : 0;      // cache tiles
    const bool has_tree_tiles = p.has_tree && split == p.nsplit - 1;
    const int ntiles = nc + (has_tree_tiles ? (p.tree_slots + KT - 1) / KT : 0);
    const int row_base_c = (req * p.nh + h) * p.cache_slots;
    const int row_base_t = (req * p.nh + h) * p.tree_slots;

    auto issue = [&](int i) {
        const int s = i % STAGES;
        const uint32_t bar = full0 + 8 * s;
        const uint32_t kd = base + s * L::STAGE;
        bar_expect_tx(bar, L::STAGE);
        const bool cache = i < nc;
        const CUtensorMap *mk = cache ? &mkc : &mkt, *mv = cache ? &mvc : &mvt;
        const int y = cache ? row_base_c + k_lo + i * KT : row_base_t + (i - nc) * KT;
#pragma unroll
        for (int b = 0; b < L::NB; ++b) {
            tma2d(kd + b * L::BOX, mk, b * 64, y, bar);
            tma2d(kd + L::TILE + b * L::BOX, mk, b * 64, y + p.lo_rows, bar);
            tma2d(kd + 2 * L::TILE + b * L::BOX, mv, b * 64, y, bar);
            tma2d(kd + 3 * L::TILE + b * L::BOX, mv, b * 64, y + p.lo_rows, bar);
        }
    };
    // the cache tiles of the first stages may go out before the wait; tree
    // K/V is the previous kernel's output
    const int n_pre = min(STAGES, ntiles);
    const int n_early = p.cache_early ? min(n_pre, nc) : 0;
    if (threadIdx.x == 0)
        for (int i = 0; i < n_early; ++i) issue(i);
    wait_prior();
    if (threadIdx.x == 0 && p.stamp) atomicMin(p.stamp + 1, gtime());
    allow_dependents();

    // TMEM addresses of this warp's lane quarter
    const uint32_t tq = tmem + ((uint32_t)(32 * quarter) << 16);

    if (warp == 0) {
        // ---- producer ------------------------------------------------------
        if (lane == 0) {
            for (int i = n_early; i < n_pre; ++i) issue(i);
            int i = n_pre;
            for (; i < ntiles; ++i) {
                const int s = i % STAGES;
                if (!bar_wait(empty0 + 8 * s, (uint32_t)(i / STAGES - 1) & 1u, &abort_flag, p.status)) break;
                issue(i);
            }
            if (abort_flag) {       // the copies still in flight land before the CTA exits
                volatile int never = 0;
                for (int j = (i > STAGES ? i - STAGES : 0); j < i; ++j)
                    bar_wait(full0 + 8 * (j % STAGES), (uint32_t)(j / STAGES) & 1u, &never, p.status);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---- MMA issue -----------------------------------------------------
        if (lane == 0 && ntiles > 0) {
            const uint32_t id_qk = idesc(ROWS, KT, 0), id_pv = idesc(ROWS, HD, 1);
            auto qk = [&](int t) -> bool {
                const int s = t % STAGES;
                if (!bar_wait(full0 + 8 * s, (uint32_t)(t / STAGES) & 1u, &abort_flag, p.status)) return false;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t kd = base + s * L::STAGE;
                const uint32_t sd = tmem + L::T_S + (t & 1) * KT;
#pragma unroll
                for (int kk = 0; kk < HD / 16; ++kk) {
                    const uint32_t ko = (kk >> 2) * L::BOX + (kk & 3) * 32;
                    const uint64_t kh = sdesc(kd + ko, 16, 1024), kl = sdesc(kd + L::TILE + ko, 16, 1024);
                    mma_ts(sd, tmem + L::T_QH + kk * 8, kh, id_qk, kk > 0);
                    mma_ts(sd, tmem + L::T_QL + kk * 8, kh, id_qk, 1u);
                    mma_ts(sd, tmem + L::T_QH + kk * 8, kl, id_qk, 1u);
                }
                mma_commit(s_full0 + 8 * (t & 1));
                return true;
            };
            bool ok = bar_wait(q_ready, 0, &abort_flag, p.status);
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            if (ok) ok = qk(0);
            if (ok && ntiles > 1) ok = qk(1);
            for (int j = 0; ok && j < ntiles; ++j) {
                if (!bar_wait(p_full0 + 8 * (j & 1), (uint32_t)(j >> 1) & 1u, &abort_flag, p.status)) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t vd = base + (j % STAGES) * L::STAGE + 2 * L::TILE;
                // P of keys 32h .. 32h+31 sits in S columns 32h .. 32h+31: hi pairs
                // in the first 16, lo pairs in the next 16
                const uint32_t pd = tmem + L::T_S + (j & 1) * KT;
#pragma unroll
                for (int kk = 0; kk < KT / 16; ++kk) {
                    const uint32_t ph = pd + (kk >> 1) * 32 + (kk & 1) * 8, pl = ph + 16;
                    const uint64_t vh = sdesc(vd + kk * 2048, L::BOX, 1024);
                    const uint64_t vl = sdesc(vd + L::TILE + kk * 2048, L::BOX, 1024);
                    mma_ts(tmem + L::T_O, ph, vh, id_pv, (j > 0) || (kk > 0));
                    mma_ts(tmem + L::T_O, pl, vh, id_pv, 1u);
                    mma_ts(tmem + L::T_O, ph, vl, id_pv, 1u);
                }
                mma_commit(empty0 + 8 * (j % STAGES));
                mma_commit(o_ready);
                if (j + 2 < ntiles) ok = qk(j + 2);
            }
            // no MMA outlives the CTA's tensor memory
            mma_commit(drain);
            volatile int never = 0;
            bar_wait(drain, 0, &never, p.status);
        }
        __syncwarp();
    }

    // ---- softmax warps ----------------------------------------------------
    // Two warps share each TMEM lane quarter and take half of every tile's keys
    // (half 0: keys 0-31, half 1: keys 32-63) and half of O's columns; the two
    // halves of a row exchange their tile maxima through shared memory, so both
    // keep the same reference maximum. A failed (timed-out) wait makes a warp
    // skip the work of the remaining tiles but not the CTA barriers, so the
    // warps stay in step.
    auto wwait = [&](uint32_t bar, uint32_t parity) {
        const bool r = bar_wait(bar, parity, &abort_flag, p.status);
        return __all_sync(0xffffffffu, r);
    };
    const int hf = (warp - 2) >> 2;                   // column half of a softmax warp
    constexpr int OH = HD / 2;                        // O columns per half
    uint32_t o_acc[OH];                               // this half of the row's O (fp32 bits)
    float m_used = -INFINITY, l_sum = 0.f;
    bool dead = false;
    if (smx) {
        // query row (hi, lo) into tensor memory, the A operand of Q K^T: this
        // half's HD/4 bf16 pairs of each plane
        {
            const uint4 *qh = reinterpret_cast<const uint4 *>(p.q + (size_t)row * H + h * HD);
            const uint4 *ql = reinterpret_cast<const uint4 *>(p.q + p.lo + (size_t)row * H + h * HD);
            uint32_t rh[HD / 4], rl[HD / 4];
#pragma unroll
            for (int u = 0; u < HD / 16; ++u) {
                const int g = hf * (HD / 16) + u;            // uint4 index in the row
                const uint4 a4 = valid ? qh[g] : make_uint4(0, 0, 0, 0);
                const uint4 b4 = valid && p.lo ? ql[g] : make_uint4(0, 0, 0, 0);
                rh[4 * u] = a4.x; rh[4 * u + 1] = a4.y; rh[4 * u + 2] = a4.z; rh[4 * u + 3] = a4.w;
                rl[4 * u] = b4.x; rl[4 * u + 1] = b4.y; rl[4 * u + 2] = b4.z; rl[4 * u + 3] = b4.w;
            }
#pragma unroll
            for (int c0 = 0; c0 < HD / 4; c0 += 16) {
                tmem_st16(tq + L::T_QH + hf * (HD / 4) + c0, rh + c0);
                tmem_st16(tq + L::T_QL + hf * (HD / 4) + c0, rl + c0);
            }
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            bar_arrive(q_ready);
        }
        const uint64_t *mrow = (has_tree_tiles && valid) ? p.mask + (size_t)row * p.mask_words : nullptr;
        const int klim = valid ? min(k_hi, plen) : 0;        // cache keys visible by position
        const int tlim = valid ? p.tree_slots : 0;           // tree keys: by the ancestor mask
        for (int j = 0; j < ntiles; ++j) {
            if (!dead && !wwait(s_full0 + 8 * (j & 1), (uint32_t)(j >> 1) & 1u)) dead = true;
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t sd = tq + L::T_S + (j & 1) * KT;
            uint32_t sr[32];
            tmem_ld32(sd + 32 * hf, sr);
            const bool tree_tile = j >= nc;
            const int key0 = (tree_tile ? (j - nc) * KT : k_lo + j * KT) + 32 * hf;
            const int lim = (tree_tile ? tlim : klim) - key0;   // columns c < lim are inside the range
            uint32_t bits = 0xffffffffu;
            if (tree_tile) {
                const int w = j - nc;                           // one mask word per 64 tree keys
                bits = (mrow && w < p.mask_words) ? (uint32_t)(mrow[w] >> (32 * hf)) : 0u;
            }
            float v[32];
            float mx = -INFINITY;
#pragma unroll
            for (int c = 0; c < 32; ++c) {
                const bool vis = c < lim && ((bits >> c) & 1u);
                v[c] = vis ? __uint_as_float(sr[c]) * p.scale_log2 : -INFINITY;
                mx = fmaxf(mx, v[c]);
            }
            // the row's tile maximum over both halves
            float *xm = s_xmax + ((j & 1) * 2 + hf) * ROWS;
            if (lane < 16) xm[row_local] = mx;
            softmax_sync(quarter);
            if (lane < 16) mx = fmaxf(mx, s_xmax[((j & 1) * 2 + (hf ^ 1)) * ROWS + row_local]);
            // move the reference maximum only when the tile's exceeds it by > 2^8
            // (and O already holds visible keys: otherwise O is exactly 0). The
            // rescale waits for P V of tile j-1 on o_ready: the completed Q K^T of
            // tile j implies P V of tile j-2, so the barrier is at most one phase
            // behind and its parity names the phase.
            const bool need = m_used != -INFINITY && mx > m_used + RESCALE_LOG2;
            if (__any_sync(0xffffffffu, need)) {
                if (!dead && !wwait(o_ready, (uint32_t)(j - 1) & 1u)) dead = true;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const float f = need ? ex2_fast(m_used - mx) : 1.f;
#pragma unroll
                for (int c0 = 0; c0 < OH; c0 += 32) {
                    uint32_t r[32];
                    tmem_ld32(tq + L::T_O + hf * OH + c0, r);
#pragma unroll
                    for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * f);
                    tmem_st32(tq + L::T_O + hf * OH + c0, r);
                }
                l_sum *= f;
                if (need) m_used = mx;
            }
            if (m_used == -INFINITY) m_used = mx;
            const float use = m_used == -INFINITY ? 0.f : m_used;
            float rs = 0.f;
            uint32_t ph[16], pl[16];
#pragma unroll
            for (int c = 0; c < 32; c += 2) {
                const float e0 = ex2_fast(v[c] - use), e1 = ex2_fast(v[c + 1] - use);
                rs += e0 + e1;
                split_pair(e0, e1, ph[c / 2], pl[c / 2]);
            }
            l_sum += rs;
            tmem_st16(sd + 32 * hf, ph);                  // over this half's own S columns:
            tmem_st16(sd + 32 * hf + 16, pl);             // hi pairs, then lo pairs
            asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
            bar_arrive(p_full0 + 8 * (j & 1));
        }
        // every MMA of the split has completed (the drain barrier completes once,
        // after the last P V; o_ready's parity could not tell its last phase from
        // the one two phases back)
        if (!dead && ntiles > 0 && !wwait(drain, 0u)) dead = true;
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        if (ntiles > 0) {
#pragma unroll
            for (int c0 = 0; c0 < OH; c0 += 32) tmem_ld32(tq + L::T_O + hf * OH + c0, o_acc + c0);
        } else {
#pragma unroll
            for (int c = 0; c < OH; ++c) o_acc[c] = 0u;
        }
        // the row's sum over both halves
        if (lane < 16) s_xmax[(4 + hf) * ROWS + row_local] = l_sum;
        softmax_sync(quarter);
        if (lane < 16) l_sum += s_xmax[(4 + (hf ^ 1)) * ROWS + row_local];
    }
    const bool ok = !dead && !abort_flag;

    const int nsplit = p.nsplit;
    if (nsplit == 1) {
        if (valid && ok) {
            const float inv = l_sum > 0.f ? 1.f / l_sum : 0.f;
            bf16 *dst = p.out + (size_t)row * H + h * HD + hf * OH;
#pragma unroll
            for (int c = 0; c < OH; c += 4)
                Split<bf16>::store4(dst + c, p.lo,
                                    make_float4(__uint_as_float(o_acc[c]) * inv, __uint_as_float(o_acc[c + 1]) * inv,
                                                __uint_as_float(o_acc[c + 2]) * inv,
                                                __uint_as_float(o_acc[c + 3]) * inv));
        }
    } else {
        // Several splits: this (row tile, head)'s CTAs form one cluster. Each
        // leaves its partial (unnormalised O, reference max m, sum l) in its own
        // shared memory (the K/V ring is idle now); after a cluster barrier every
        // CTA combines a slice of the rows, reading all partials through
        // distributed shared memory in rank order, and writes them out.
        float *s_o = reinterpret_cast<float *>(smem_raw + (base - su32(smem_raw)));   // [64][LD]
        float *s_ml = s_o + ROWS * L::LD;                                             // [64][2]
        __syncthreads();                  // every TMA into the ring has landed and been used
        if (smx && lane < 16) {
            const bool live = valid && ok;
#pragma unroll
            for (int c = 0; c < OH; c += 4)
                *reinterpret_cast<float4 *>(s_o + row_local * L::LD + hf * OH + c) =
                    live ? make_float4(__uint_as_float(o_acc[c]), __uint_as_float(o_acc[c + 1]),
                                       __uint_as_float(o_acc[c + 2]), __uint_as_float(o_acc[c + 3]))
                         : make_float4(0.f, 0.f, 0.f, 0.f);
            if (hf == 0)
                *reinterpret_cast<float2 *>(s_ml + row_local * 2) =
                    live ? make_float2(m_used, l_sum) : make_float2(-INFINITY, 0.f);
        }
        cluster_sync();
        const uint32_t rank = cluster_rank();
        const int nrows = r_end - r0;
        const int per = (nrows + nsplit - 1) / nsplit;
        const int row_lo = (int)rank * per, row_hi = min(nrows, row_lo + per);
        const uint32_t o_local = su32(s_o), ml_local = su32(s_ml);
        // a half-warp per row (16 lanes, HD/64 float4 each): every row of the
        // slice in one pass at the decode shapes
        constexpr int C4 = HD / 4, NHALF = THREADS / 16, PER_LANE = C4 / 16;
        const int hl = lane & 15;
        for (int r2 = row_lo + (threadIdx.x >> 4); r2 - (int)(lane >> 4) < row_hi; r2 += NHALF) {
            const bool live = r2 < row_hi;
            const int rr = live ? r2 : row_lo;
            float2 ml = make_float2(-INFINITY, 0.f);
            if (live && hl < nsplit) ml = dsmem_ld_f2(dsmem_addr(ml_local + rr * 8, hl));
            float4 v[MAX_SPLITS][PER_LANE];
#pragma unroll
            for (int sp = 0; sp < MAX_SPLITS; ++sp)
#pragma unroll
                for (int e = 0; e < PER_LANE; ++e)
                    if (live && sp < nsplit)
                        v[sp][e] = dsmem_ld_f4(dsmem_addr(o_local + (rr * L::LD + 4 * (hl + 16 * e)) * 4, sp));
            // lane sp of the half holds split sp's (m, l); shuffles within the
            // half give the max and the sum
            float M = ml.x;
#pragma unroll
            for (int o = 8; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o, 16));
            const float w = (hl < nsplit && M != -INFINITY) ? exp2f(ml.x - M) : 0.f;
            // the normaliser summed in split order (empty splits add exact zeros),
            // so a launch's result never depends on how many empty splits it has
            const float wl = w * ml.y;
            float den = 0.f;
#pragma unroll
            for (int sp = 0; sp < MAX_SPLITS; ++sp) {
                const float t = __shfl_sync(0xffffffffu, wl, sp, 16);
                if (sp < nsplit) den += t;
            }
            const float inv = den > 0.f ? 1.f / den : 0.f;
            const float wn = w * inv;
            float wsp[MAX_SPLITS];
#pragma unroll
            for (int sp = 0; sp < MAX_SPLITS; ++sp) wsp[sp] = __shfl_sync(0xffffffffu, wn, sp, 16);
            if (live && !abort_flag) {
#pragma unroll
                for (int e = 0; e < PER_LANE; ++e) {
                    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int sp = 0; sp < MAX_SPLITS; ++sp)
                        if (sp < nsplit) {
                            acc.x += wsp[sp] * v[sp][e].x; acc.y += wsp[sp] * v[sp][e].y;
                            acc.z += wsp[sp] * v[sp][e].z; acc.w += wsp[sp] * v[sp][e].w;
                        }
                    Split<bf16>::store4(p.out + (size_t)(r0 + rr) * H + h * HD + 4 * (hl + 16 * e), p.lo, acc);
                }
            }
        }
        cluster_sync();                    // partials stay readable until all are done
    }

    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (threadIdx.x == 0 && p.stamp) atomicMax(p.stamp + 2, gtime());
    if (warp == 1) {
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(L::T_COLS)
                     : "memory");
    }
}

struct MapKey {
    const void *ptr;
    long rows;
    bool operator==(const MapKey &o) const { return ptr == o.ptr && rows == o.rows; }
};
struct MapKeyHash {
    size_t operator()(const MapKey &k) const {
        return std::hash<const void *>()(k.ptr) ^ std::hash<long>()(k.rows * 2654435761L);
    }
};

}  // namespace

struct AttnTcPlan {
    int num_sms = 148;
    PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    std::unordered_map<MapKey, CUtensorMap, MapKeyHash> maps;
    bool attr_set = false;
};

bool attn_tc_plan_create(AttnTcPlan **out) {
    AttnTcPlan *p = new AttnTcPlan();
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&p->num_sms, cudaDevAttrMultiProcessorCount, dev);
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn) {
        delete p;
        return false;
    }
    p->encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    *out = p;
    return true;
}

void attn_tc_plan_destroy(AttnTcPlan *p) { delete p; }

// Tensor map over `rows` rows of hd bf16 (boxes of 64 rows x 64 columns).
static const CUtensorMap *kv_map(AttnTcPlan *p, const void *ptr, long rows, int hd) {
    MapKey key{ptr, rows};
    auto it = p->maps.find(key);
    if (it != p->maps.end()) return &it->second;
    CUtensorMap m;
    memset(&m, 0, sizeof m);
    cuuint64_t dims[2] = {(cuuint64_t)hd, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)hd * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)KT};
    cuuint32_t estr[2] = {1, 1};
    if (p->encode(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return nullptr;
    return &p->maps.emplace(key, m).first->second;
}

bool launch_attention_tc(AttnTcPlan *p, const AttnArgs<bf16> &a, int B, int rows_per_req, const int *order,
                         int *status, cudaStream_t s, unsigned long long *stamp) {
    if (a.R <= 0) return true;
    if (a.hd != 64 && a.hd != 128) return false;
    if (a.lo % a.hd) return false;
    const int tiles_per_req = (rows_per_req + ROWS - 1) / ROWS;
    const int n_blocks = a.R / rows_per_req;
    const int row_tiles = n_blocks * tiles_per_req;
    if (row_tiles > 65535 || a.nh > 65535) return false;   // grid (heads, row tiles, splits)
    const long base = (long)row_tiles * a.nh;
    const int has_tree = a.mask != nullptr;
    // One CTA fills an SM: as many splits per (row tile, head) as keep the
    // launch within one wave (a function of the launch's shape alone).
    const int nsplit = (int)std::max<long>(1, std::min<long>(MAX_SPLITS, p->num_sms / base));
    const long lo_rows = a.lo / a.hd;
    const long kc_rows = (long)B * a.nh * a.cache_slots + lo_rows;
    const CUtensorMap *mkc = kv_map(p, a.cache_k, kc_rows, a.hd);
    const CUtensorMap *mvc = kv_map(p, a.cache_v, kc_rows, a.hd);
    const CUtensorMap *mkt = mkc, *mvt = mvc;
    if (has_tree) {
        const long kt_rows = (long)B * a.nh * a.tree_slots + lo_rows;
        mkt = kv_map(p, a.tree_k, kt_rows, a.hd);
        mvt = kv_map(p, a.tree_v, kt_rows, a.hd);
    }
    if (!mkc || !mvc || !mkt || !mvt) return false;
    AttnTcParams tp;
    memset(&tp, 0, sizeof tp);
    tp.q = a.q;
    tp.rows = a.rows;
    tp.mask = a.mask;
    tp.out = a.out;
    tp.lo = a.lo;
    tp.lo_rows = (int)lo_rows;
    tp.status = status;
    tp.R = a.R;
    tp.rows_per_req = rows_per_req;
    tp.tiles_per_req = tiles_per_req;
    tp.nh = a.nh;
    tp.cache_slots = a.cache_slots;
    tp.tree_slots = a.tree_slots;
    tp.mask_words = a.mask_words;
    tp.has_tree = has_tree;
    tp.nsplit = nsplit;
    tp.cache_early = a.cache_fresh ? 0 : 1;
    tp.scale_log2 = a.scale * 1.4426950408889634f;
    tp.stamp = stamp;
    if (order && n_blocks > 1 && n_blocks <= ORDER_MAX) {
        // the kernel indexes rows through it: only a permutation is taken
        uint64_t seen = 0;
        for (int i = 0; i < n_blocks; ++i) {
            if (order[i] < 0 || order[i] >= n_blocks || (seen >> order[i] & 1)) return false;
            seen |= 1ull << order[i];
            tp.order[i] = (uint8_t)order[i];
        }
        tp.n_order = n_blocks;
    }
    const size_t smem = 1024 + (a.hd == 128 ? (size_t)STAGES * Lay<128>::STAGE : (size_t)STAGES * Lay<64>::STAGE);
    if (!p->attr_set) {
        cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(1024 + STAGES * Lay<128>::STAGE));
        cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(1024 + STAGES * Lay<64>::STAGE));
        cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        p->attr_set = true;
    }
    // the splits of one (row tile, head) run as one cluster (z = splits)
    cudaLaunchConfig_t lc;
    memset(&lc, 0, sizeof lc);
    lc.gridDim = dim3(a.nh, row_tiles, nsplit);
    lc.blockDim = dim3(THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    // Plain stream order behind the previous kernel (no programmatic
    // serialisation: its CTAs could not start before that kernel's CTAs left
    // the SMs anyway, and its griddepcontrol.wait then returned 3-4 us after
    // their exit where a plain launch starts 1.3 us after it); the kernel still
    // releases its own dependents early.
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 1;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = nsplit;
    lc.attrs = at;
    lc.numAttrs = 1;
    cudaError_t e = a.hd == 128 ? cudaLaunchKernelEx(&lc, attn_tc_kernel<128>, *mkc, *mvc, *mkt, *mvt, tp)
                                : cudaLaunchKernelEx(&lc, attn_tc_kernel<64>, *mkc, *mvc, *mkt, *mvt, tp);
    note_launch();
    if (e != cudaSuccess) return false;
    return true;
}

}  // namespace msd
