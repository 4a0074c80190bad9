// Tree-masked attention on the tensor cores for the bf16 path.
//
// A CTA (8 warps) takes 64 query rows of one request and one head: warps g and
// g + 4 own rows 16g .. 16g + 15, and split every key tile between them (keys
// 0-31 and 32-63), each with its own online-softmax state; the two halves merge
// once, after the CTA's last tile. Keys come in tiles of 64, staged by TMA (two
// 64x64 boxes per tile for head_dim 128, 128-byte swizzle) into a ring of
// shared-memory stages completed on mbarriers. Per tile and warp: S = Q K^T
// over its 32 keys with mma.sync m16n8k16 (bf16, fp32 accumulate), masking, an
// online softmax in base 2 (row max and sum across the 4 lanes of a quad with
// shuffles), and O += P V (P re-packed from the S accumulators as the A
// operand, V read with ldmatrix.trans).
//
// Visible keys of a row (Sec. 3.2: a candidate is conditioned on its prefix
// only): cache positions [0, plen) of its request, and tree slots whose bit is
// set in its mask. The cache range is split across CTAs (z < nsplit_cache);
// the tree part is one more split. With more than one split, every CTA writes
// unnormalised partials (O, running max, running sum) to a workspace and the
// last CTA of a (row tile, head) combines them in split order (deterministic),
// then resets its ticket. All mbarrier waits are bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstring>
#include <unordered_map>

#include "attn_tc.h"

namespace msd {

namespace {

constexpr int ROWS = 64;          // query rows per CTA
constexpr int KT = 64;            // keys per tile
constexpr int THREADS = 256;      // 8 warps: 4 row groups x 2 key halves
// row stride (floats) of the fp32 partials in shared memory: padded so that the
// 8 rows a warp writes at once fall in different banks
template <int HD> constexpr int PART_LD = HD + 8;
constexpr int MAX_STAGES = 3;
constexpr int CACHE_SPLITS = 8;   // cache splits of a decode launch (capacity-derived chunk)
constexpr int MAX_SPLITS = CACHE_SPLITS + 1;   // + the tree split = cluster size
constexpr unsigned long long ATTN_TIMEOUT_NS = 2000000000ull;

struct AttnTcParams {
    const bf16 *q;
    const RowDesc *rows;
    const uint64_t *mask;
    bf16 *out;
    int *status;
    int R, rows_per_req, tiles_per_req, nh, cache_slots, tree_slots, mask_words;
    int nsplit_cache, has_tree, chunk, stages;
    int cache_early;          // cache K/V may be requested before the wait (not written by the previous kernel)
    float scale_log2;
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

__device__ bool bar_wait(uint32_t bar, uint32_t parity, int *status) {
    if (bar_try(bar, parity)) return true;
    const unsigned long long t0 = gtime();
    while (!bar_try(bar, parity)) {
        if (gtime() - t0 > ATTN_TIMEOUT_NS) {
            set_status(status, ST_TIMEOUT);
            return false;
        }
    }
    return true;
}

__device__ __forceinline__ void tma2d(uint32_t dst, const CUtensorMap *m, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(m), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// Byte address of 16-byte chunk `c` of row `row` in a [64][HD] bf16 tile
// stored as HD/64 boxes of [64 rows][128 B] with the 128-byte swizzle.
__device__ __forceinline__ uint32_t swz(uint32_t base, int row, int c) {
    return base + (c >> 3) * 8192 + row * 128 + (((c & 7) ^ (row & 7)) << 4);
}

__device__ __forceinline__ void ldsm4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                      uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm4t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                       uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}

__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\nbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t dsmem_addr(uint32_t local, int rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}

__device__ __forceinline__ float dsmem_ld_f32(uint32_t a) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
    return v;
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

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

template <int HD>
__global__ void __launch_bounds__(THREADS, 2)
    attn_tc_kernel(const __grid_constant__ CUtensorMap mkc, const __grid_constant__ CUtensorMap mvc,
                   const __grid_constant__ CUtensorMap mkt, const __grid_constant__ CUtensorMap mvt,
                   const AttnTcParams p) {
    constexpr int NB = HD / 64;                   // 64-wide boxes per row
    constexpr int TILE_BYTES = KT * HD * 2;       // one K (or V) tile
    constexpr int NT_O = HD / 8;                  // O n-tiles per warp
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t bars[MAX_STAGES];
    __shared__ int s_pmax;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = warp & 3, half = warp >> 2;     // row group, key half of each tile
    const int tile = blockIdx.x, h = blockIdx.y, split = blockIdx.z;
    const int blk = tile / p.tiles_per_req;
    const int r0 = blk * p.rows_per_req + (tile - blk * p.tiles_per_req) * ROWS;
    const int r_end = min(r0 + ROWS, (blk + 1) * p.rows_per_req);
    const bool is_tree = p.has_tree && split == p.nsplit_cache;
    const int H = p.nh * HD;

    const uint32_t base = (su32(smem_raw) + 1023u) & ~1023u;
    const uint32_t q_s = base;                             // [64][HD]
    const uint32_t kv_s = base + ROWS * HD * 2;            // STAGES x (K tile, V tile)

    if (threadIdx.x == 0) {
        for (int s = 0; s < p.stages; ++s)
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(su32(&bars[s])), "r"(1));
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        s_pmax = 0;
        asm volatile("prefetch.tensormap [%0];" ::"l"(&mkc) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(&mvc) : "memory");
    }
    __syncthreads();
    // Before the wait: the row descriptors (written by set-up kernels at least
    // two launches back) and, unless the previous kernel wrote into it, the
    // cache K/V. The previous kernel's q and tree K/V are read after the wait.
    const int req = p.rows[r0].req;

    // Rows of this thread: A = lane/4, B = lane/4 + 8 of the warp's 16.
    const int ra = r0 + grp * 16 + (lane >> 2), rb = ra + 8;
    const bool va = ra < r_end, vb = rb < r_end;
    const int plen_a = va ? p.rows[ra].plen : 0, plen_b = vb ? p.rows[rb].plen : 0;
    atomicMax(&s_pmax, max(plen_a, plen_b));
    __syncthreads();

    // Key range of this split.
    int k_lo, k_hi, row_base;
    const CUtensorMap *mk, *mv;
    if (is_tree) {
        k_lo = 0;
        k_hi = p.tree_slots;
        row_base = (req * p.nh + h) * p.tree_slots;
        mk = &mkt;
        mv = &mvt;
    } else {
        k_lo = split * p.chunk;
        k_hi = min(k_lo + p.chunk, min(s_pmax, p.cache_slots));
        row_base = (req * p.nh + h) * p.cache_slots;
        mk = &mkc;
        mv = &mvc;
    }
    const int ntiles = k_hi > k_lo ? (k_hi - k_lo + KT - 1) / KT : 0;
    const uint32_t stage_bytes = 2 * TILE_BYTES;

    const int stages = p.stages;
    auto issue = [&](int i) {
        const int s = i % stages;
        const uint32_t bar = su32(&bars[s]);
        const uint32_t kd = kv_s + s * stage_bytes, vd = kd + TILE_BYTES;
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar),
                     "r"(stage_bytes)
                     : "memory");
        const int y = row_base + k_lo + i * KT;
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            tma2d(kd + b * 8192, mk, b * 64, y, bar);
            tma2d(vd + b * 8192, mv, b * 64, y, bar);
        }
    };
    // K/V tiles in flight first, then the Q tile (all its loads issued before
    // the first shared-memory store); rows past the request's rows are zero.
    const bool early = !is_tree && p.cache_early;
    if (threadIdx.x == 0 && early)
        for (int i = 0; i < min(stages, ntiles); ++i) issue(i);
    wait_prior();
    allow_dependents();
    if (threadIdx.x == 0 && !early)
        for (int i = 0; i < min(stages, ntiles); ++i) issue(i);
    {
        constexpr int QV = ROWS * HD / 8 / THREADS;   // 16-byte pieces per thread
        uint4 qv[QV];
#pragma unroll
        for (int j = 0; j < QV; ++j) {
            const int i = threadIdx.x + j * THREADS;
            const int row = i / (HD / 8), c = i - row * (HD / 8);
            qv[j] = r0 + row < r_end
                        ? __ldg(reinterpret_cast<const uint4 *>(p.q + (size_t)(r0 + row) * H + h * HD + c * 8))
                        : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int j = 0; j < QV; ++j) {
            const int i = threadIdx.x + j * THREADS;
            const int row = i / (HD / 8), c = i - row * (HD / 8);
            asm volatile("st.shared.v4.b32 [%0], {%1,%2,%3,%4};" ::"r"(swz(q_s, row, c)), "r"(qv[j].x),
                         "r"(qv[j].y), "r"(qv[j].z), "r"(qv[j].w)
                         : "memory");
        }
    }
    __syncthreads();

    // Q fragments of the warp's 16 rows are re-read from shared memory per tile
    // (ldmatrix), which keeps two 8-warp CTAs' registers on an SM.
    const int q_row = grp * 16 + ((lane >> 3) & 1) * 8 + (lane & 7);

    // Tree-mask words of the two rows (tree split only).
    const uint64_t *mask_a = (is_tree && va) ? p.mask + (size_t)ra * p.mask_words : nullptr;
    const uint64_t *mask_b = (is_tree && vb) ? p.mask + (size_t)rb * p.mask_words : nullptr;

    float o[NT_O][4];
#pragma unroll
    for (int j = 0; j < NT_O; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float m_a = -INFINITY, m_b = -INFINITY, l_a = 0.f, l_b = 0.f;
    bool ok = true;

    for (int i = 0; i < ntiles; ++i) {
        const int s = i % stages;
        if (!bar_wait(su32(&bars[s]), (uint32_t)(i / stages) & 1u, p.status)) ok = false;
        const uint32_t ks = kv_s + s * stage_bytes, vs = ks + TILE_BYTES;
        const int key0 = k_lo + i * KT;

        // this warp's 32 keys of the tile: kh .. kh + 31
        const int kh = half * 32;
        float sc[4][4];
#pragma unroll
        for (int j = 0; j < 4; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
            uint32_t qf[4];
            ldsm4(swz(q_s, q_row, 2 * kk + (lane >> 4)), qf[0], qf[1], qf[2], qf[3]);
#pragma unroll
            for (int np = 0; np < 2; ++np) {
                const int m = lane >> 3;
                const int key = kh + np * 16 + (m >> 1) * 8 + (lane & 7);
                uint32_t b0, b1, b2, b3;
                ldsm4(swz(ks, key, 2 * kk + (m & 1)), b0, b1, b2, b3);
                mma16816(sc[2 * np], qf, b0, b1);
                mma16816(sc[2 * np + 1], qf, b2, b3);
            }
        }
        // mask + scale (base-2 logits)
        uint64_t wa = 0, wb = 0;
        if (is_tree) {
            const int w = key0 >> 6;
            if (mask_a && w < p.mask_words) wa = mask_a[w];
            if (mask_b && w < p.mask_words) wb = mask_b[w];
        }
        float mx_a = -INFINITY, mx_b = -INFINITY;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int kl = kh + 8 * j + 2 * (lane & 3) + (e & 1);
                const int key = key0 + kl;
                bool vis;
                if (is_tree) {
                    const uint64_t wd = e < 2 ? wa : wb;
                    vis = key < k_hi && ((wd >> (key & 63)) & 1ull);
                } else {
                    vis = key < k_hi && key < (e < 2 ? plen_a : plen_b);
                }
                const float v = vis ? sc[j][e] * p.scale_log2 : -INFINITY;
                sc[j][e] = v;
                if (e < 2) mx_a = fmaxf(mx_a, v); else mx_b = fmaxf(mx_b, v);
            }
        }
        mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 1));
        mx_a = fmaxf(mx_a, __shfl_xor_sync(0xffffffffu, mx_a, 2));
        mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 1));
        mx_b = fmaxf(mx_b, __shfl_xor_sync(0xffffffffu, mx_b, 2));
        const float mn_a = fmaxf(m_a, mx_a), mn_b = fmaxf(m_b, mx_b);
        const float use_a = mn_a == -INFINITY ? 0.f : mn_a, use_b = mn_b == -INFINITY ? 0.f : mn_b;
        const float cf_a = exp2f(m_a - use_a), cf_b = exp2f(m_b - use_b);
        m_a = mn_a;
        m_b = mn_b;
        float rs_a = 0.f, rs_b = 0.f;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            sc[j][0] = exp2f(sc[j][0] - use_a);
            sc[j][1] = exp2f(sc[j][1] - use_a);
            sc[j][2] = exp2f(sc[j][2] - use_b);
            sc[j][3] = exp2f(sc[j][3] - use_b);
            rs_a += sc[j][0] + sc[j][1];
            rs_b += sc[j][2] + sc[j][3];
        }
        l_a = l_a * cf_a + rs_a;
        l_b = l_b * cf_b + rs_b;
#pragma unroll
        for (int j = 0; j < NT_O; ++j) {
            o[j][0] *= cf_a; o[j][1] *= cf_a;
            o[j][2] *= cf_b; o[j][3] *= cf_b;
        }
        // O += P V over the warp's 32 keys
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            uint32_t pa[4];
            pa[0] = pack_bf16(sc[2 * kk][0], sc[2 * kk][1]);
            pa[1] = pack_bf16(sc[2 * kk][2], sc[2 * kk][3]);
            pa[2] = pack_bf16(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
            pa[3] = pack_bf16(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
            for (int dp = 0; dp < HD / 16; ++dp) {
                const int m = lane >> 3;
                const int key = kh + kk * 16 + (m & 1) * 8 + (lane & 7);
                uint32_t b0, b1, b2, b3;
                ldsm4t(swz(vs, key, 2 * dp + (m >> 1)), b0, b1, b2, b3);
                mma16816(o[2 * dp], pa, b0, b1);
                mma16816(o[2 * dp + 1], pa, b2, b3);
            }
        }
        __syncthreads();                              // every warp is done with stage s
        if (threadIdx.x == 0 && i + stages < ntiles) issue(i + stages);
    }

    l_a += __shfl_xor_sync(0xffffffffu, l_a, 1);
    l_a += __shfl_xor_sync(0xffffffffu, l_a, 2);
    l_b += __shfl_xor_sync(0xffffffffu, l_b, 1);
    l_b += __shfl_xor_sync(0xffffffffu, l_b, 2);

    // Merge the two key halves of each row group: the upper warps leave (O, m,
    // l) in shared memory (the K/V stages are idle now), the lower warps fold
    // them into theirs; the result is left in the same place for the cluster
    // combine below.
    const int col0 = 2 * (lane & 3);
    __syncthreads();
    constexpr int LD = PART_LD<HD>;
    float *s_o = reinterpret_cast<float *>(smem_raw + (kv_s - su32(smem_raw)));   // [64][LD]
    float *s_ml = s_o + ROWS * LD;                                               // [64][2]
    const int la = grp * 16 + (lane >> 2), lb = la + 8;
    if (half == 1) {
#pragma unroll
        for (int j = 0; j < NT_O; ++j) {
            const int c = 8 * j + col0;
            *reinterpret_cast<float2 *>(s_o + la * LD + c) = make_float2(o[j][0], o[j][1]);
            *reinterpret_cast<float2 *>(s_o + lb * LD + c) = make_float2(o[j][2], o[j][3]);
        }
        if ((lane & 3) == 0) {
            *reinterpret_cast<float2 *>(s_ml + la * 2) = make_float2(m_a, l_a);
            *reinterpret_cast<float2 *>(s_ml + lb * 2) = make_float2(m_b, l_b);
        }
    }
    __syncthreads();
    if (half == 0) {
        const float2 ua = *reinterpret_cast<const float2 *>(s_ml + la * 2);
        const float2 ub = *reinterpret_cast<const float2 *>(s_ml + lb * 2);
        const float Ma = fmaxf(m_a, ua.x), Mb = fmaxf(m_b, ub.x);
        const float ba = Ma == -INFINITY ? 0.f : Ma, bb = Mb == -INFINITY ? 0.f : Mb;
        const float c0a = exp2f(m_a - ba), c1a = exp2f(ua.x - ba);
        const float c0b = exp2f(m_b - bb), c1b = exp2f(ub.x - bb);
#pragma unroll
        for (int j = 0; j < NT_O; ++j) {
            const int c = 8 * j + col0;
            const float2 xa = *reinterpret_cast<const float2 *>(s_o + la * LD + c);
            const float2 xb = *reinterpret_cast<const float2 *>(s_o + lb * LD + c);
            o[j][0] = o[j][0] * c0a + xa.x * c1a;
            o[j][1] = o[j][1] * c0a + xa.y * c1a;
            o[j][2] = o[j][2] * c0b + xb.x * c1b;
            o[j][3] = o[j][3] * c0b + xb.y * c1b;
        }
        l_a = l_a * c0a + ua.y * c1a;
        l_b = l_b * c0b + ub.y * c1b;
        m_a = Ma;
        m_b = Mb;
    }

    const int nsplit = p.nsplit_cache + p.has_tree;
    if (nsplit == 1) {
        if (half == 1) return;
        const float ia = l_a > 0.f ? 1.f / l_a : 0.f, ib = l_b > 0.f ? 1.f / l_b : 0.f;
#pragma unroll
        for (int j = 0; j < NT_O; ++j) {
            const int col = h * HD + 8 * j + col0;
            if (va && ok)
                *reinterpret_cast<uint32_t *>(p.out + (size_t)ra * H + col) =
                    pack_bf16(o[j][0] * ia, o[j][1] * ia);
            if (vb && ok)
                *reinterpret_cast<uint32_t *>(p.out + (size_t)rb * H + col) =
                    pack_bf16(o[j][2] * ib, o[j][3] * ib);
        }
        return;
    }

    // Several splits: this (row tile, head)'s CTAs form one thread-block
    // cluster. Each leaves its partial (unnormalised O, running max m, running
    // sum l) in its own shared memory; after a cluster barrier every CTA
    // combines a slice of the rows, reading all partials through distributed
    // shared memory in rank order (deterministic), and writes them out.
    __syncwarp();                      // the quad's reads of s_ml above are done
    if (half == 0) {
#pragma unroll
        for (int j = 0; j < NT_O; ++j) {
            const int c = 8 * j + col0;
            *reinterpret_cast<float2 *>(s_o + la * LD + c) = make_float2(o[j][0], o[j][1]);
            *reinterpret_cast<float2 *>(s_o + lb * LD + c) = make_float2(o[j][2], o[j][3]);
        }
        if ((lane & 3) == 0) {
            *reinterpret_cast<float2 *>(s_ml + la * 2) = make_float2(m_a, l_a);
            *reinterpret_cast<float2 *>(s_ml + lb * 2) = make_float2(m_b, l_b);
        }
    }
    cluster_sync();
    const uint32_t rank = cluster_rank();
    const int nrows = r_end - r0;
    const int per = (nrows + nsplit - 1) / nsplit;
    const int row_lo = (int)rank * per, row_hi = min(nrows, row_lo + per);
    const uint32_t o_local = su32(s_o), ml_local = su32(s_ml);
    constexpr int C4 = HD / 4, NWARP = THREADS / 32;
    // a warp combines two of the CTA's rows per pass, every partial load of
    // both (max and sum of each split, then its O) issued before any is used
    for (int rr0 = row_lo + warp; rr0 < row_hi; rr0 += 2 * NWARP) {
        const int rr[2] = {rr0, rr0 + NWARP};
        const bool has[2] = {true, rr0 + NWARP < row_hi};
        float2 ml[2];
        float4 v[2][MAX_SPLITS];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            ml[u] = make_float2(-INFINITY, 0.f);
            if (has[u] && lane < nsplit) ml[u] = dsmem_ld_f2(dsmem_addr(ml_local + rr[u] * 8, lane));
        }
#pragma unroll
        for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int sp = 0; sp < MAX_SPLITS; ++sp)
                if (has[u] && lane < C4 && sp < nsplit)
                    v[u][sp] = dsmem_ld_f4(dsmem_addr(o_local + (rr[u] * LD + 4 * lane) * 4, sp));
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            if (!has[u]) continue;                         // warp-uniform
            // lane sp holds split sp's (m, l); warp shuffles give the max and the sum
            const float M = warp_max(ml[u].x);
            const float w = (lane < nsplit && M != -INFINITY) ? exp2f(ml[u].x - M) : 0.f;
            const float den = warp_sum(w * ml[u].y);
            const float inv = den > 0.f ? 1.f / den : 0.f;
            const float wn = w * inv;
            float wsp[MAX_SPLITS];
#pragma unroll
            for (int sp = 0; sp < MAX_SPLITS; ++sp) wsp[sp] = __shfl_sync(0xffffffffu, wn, sp);
            if (lane < C4) {
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int sp = 0; sp < MAX_SPLITS; ++sp)
                    if (sp < nsplit) {
                        acc.x += wsp[sp] * v[u][sp].x; acc.y += wsp[sp] * v[u][sp].y;
                        acc.z += wsp[sp] * v[u][sp].z; acc.w += wsp[sp] * v[u][sp].w;
                    }
                uint2 packed;
                packed.x = pack_bf16(acc.x, acc.y);
                packed.y = pack_bf16(acc.z, acc.w);
                if (ok)
                    *reinterpret_cast<uint2 *>(p.out + (size_t)(r0 + rr[u]) * H + h * HD + 4 * lane) = packed;
            }
        }
    }
    cluster_sync();                                    // partials stay readable until all are done
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
    int chunk_tiles = 1;       // keys per cache split / 64: fixed per context
    PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    std::unordered_map<MapKey, CUtensorMap, MapKeyHash> maps;
    bool attr_set = false;
};

bool attn_tc_plan_create(AttnTcPlan **out, int max_keys) {
    AttnTcPlan *p = new AttnTcPlan();
    // The cache range is cut at fixed multiples of chunk_tiles * 64 keys, a
    // function of the capacity only, so results never depend on how many
    // (possibly empty) splits a launch covers; with the tree split a launch
    // has at most MAX_SPLITS CTAs per cluster.
    const int tiles = (max_keys + KT - 1) / KT;
    // At most CACHE_SPLITS cache splits (+ the tree split): one cluster of <= 9
    // two-stage CTAs per (row tile, head), two CTAs per SM, so a decode launch
    // is one wave at any prefix length.
    p->chunk_tiles = std::max(2, (tiles + CACHE_SPLITS - 1) / CACHE_SPLITS);
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
    *out = p;
    return true;
}

void attn_tc_plan_destroy(AttnTcPlan *p) { delete p; }

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
    if (p->encode(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides, box,
                  estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return nullptr;
    return &p->maps.emplace(key, m).first->second;
}

bool launch_attention_tc(AttnTcPlan *p, const AttnArgs<bf16> &a, int B, int rows_per_req,
                         int p_bound, int *status, cudaStream_t s) {
    if (a.R <= 0) return true;
    if (a.hd != 64 && a.hd != 128) return false;
    const int tiles_per_req = (rows_per_req + ROWS - 1) / ROWS;
    const int n_blocks = a.R / rows_per_req;
    const int row_tiles = n_blocks * tiles_per_req;
    const long base = (long)row_tiles * a.nh;
    const int has_tree = a.mask != nullptr;
    const int pb = std::max(1, std::min(p_bound, a.cache_slots));
    const int cache_tiles = (pb + KT - 1) / KT;
    // enough (row tile, head) CTAs already: one split over the whole range;
    // otherwise fixed-size splits (the count only covers [0, p_bound))
    const int chunk_tiles = base >= p->num_sms ? cache_tiles : p->chunk_tiles;
    const int nsplit = (cache_tiles + chunk_tiles - 1) / chunk_tiles;
    const int tot = nsplit + has_tree;
    if (tot > MAX_SPLITS) return false;
    const long kc_rows = (long)B * a.nh * a.cache_slots;
    const CUtensorMap *mkc = kv_map(p, a.cache_k, kc_rows, a.hd);
    const CUtensorMap *mvc = kv_map(p, a.cache_v, kc_rows, a.hd);
    const CUtensorMap *mkt = mkc, *mvt = mvc;
    if (has_tree) {
        const long kt_rows = (long)B * a.nh * a.tree_slots;
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
    tp.status = status;
    tp.R = a.R;
    tp.rows_per_req = rows_per_req;
    tp.tiles_per_req = tiles_per_req;
    tp.nh = a.nh;
    tp.cache_slots = a.cache_slots;
    tp.tree_slots = a.tree_slots;
    tp.mask_words = a.mask_words;
    tp.nsplit_cache = nsplit;
    tp.has_tree = has_tree;
    tp.chunk = chunk_tiles * KT;
    // two stages keep two CTAs on an SM; three only where a split holds more
    // than two tiles and the CTAs fit on the SMs at one per SM
    tp.stages = (chunk_tiles <= 2 || (long)row_tiles * a.nh * (nsplit + has_tree) > p->num_sms) ? 2 : MAX_STAGES;
    tp.cache_early = a.cache_fresh ? 0 : 1;
    tp.scale_log2 = a.scale * 1.4426950408889634f;
    const size_t smem = 1024 + (size_t)ROWS * a.hd * 2 + (size_t)tp.stages * 2 * KT * a.hd * 2;
    if (!p->attr_set) {
        cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             1024 + ROWS * 128 * 2 + MAX_STAGES * 2 * KT * 128 * 2);
        cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             1024 + ROWS * 64 * 2 + MAX_STAGES * 2 * KT * 64 * 2);
        cudaFuncSetAttribute(attn_tc_kernel<128>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        cudaFuncSetAttribute(attn_tc_kernel<64>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        p->attr_set = true;
    }
    // the splits of one (row tile, head) run as one cluster (z = splits)
    cudaLaunchConfig_t lc;
    memset(&lc, 0, sizeof lc);
    lc.gridDim = dim3(row_tiles, a.nh, tot);
    lc.blockDim = dim3(THREADS);
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = 1;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = tot;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = at;
    lc.numAttrs = 2;
    cudaError_t e = a.hd == 128
                        ? cudaLaunchKernelEx(&lc, attn_tc_kernel<128>, *mkc, *mvc, *mkt, *mvt, tp)
                        : cudaLaunchKernelEx(&lc, attn_tc_kernel<64>, *mkc, *mvc, *mkt, *mvt, tp);
    note_launch();
    if (e != cudaSuccess) return false;
    return true;
}

}  // namespace msd
