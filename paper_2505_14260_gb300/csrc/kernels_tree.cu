// Integer side of the MSD step: draft-row set-up, the draft-tree builder
// (Sec. 3.2 tree drafting), verify set-up, greedy acceptance (Eq. 6 at T = 0)
// and KV compaction (rejected drafts are discarded, Sec. 3.2).
#include "kernels_tree.h"

namespace msd {

// ---------------------------------------------------------------------------
// Pass 1 (catch-up): rows r = b*D1 + j for the pending positions of request b.
// Input f = f_down(Concat(h, e_next)) (Eq. 4); the concatenated row is built
// here and the GEMM applies f_down. K/V go to the draft cache at their
// positions; each row attends causally to the cache.
// ---------------------------------------------------------------------------
template <typename T>
__global__ void catchup_setup_kernel(const int *__restrict__ seq_len, const int *__restrict__ n_pend,
                                     const T *__restrict__ pend_h, const int *__restrict__ pend_next,
                                     const T *__restrict__ E, int H, int D1, int V,
                                     T *__restrict__ xfc, long lo, RowDesc *__restrict__ rows, int *status) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x, b = r / D1, j = r - b * D1;
    const int L = seq_len[b], P = n_pend[b];
    const bool valid = j < P;
    const int pos = L - P + j;
    if (threadIdx.x == 0) {
        RowDesc d;
        d.req = b;
        d.pos = valid ? pos : 0;
        d.plen = valid ? pos + 1 : 1;
        d.dst = valid ? pos : -1;
        rows[r] = d;
    }
    int tok = valid ? pend_next[b * D1 + j] : 0;
    if (tok < 0 || tok >= V) {
        if (threadIdx.x == 0) set_status(status, ST_BAD_TOKEN);
        tok = 0;
    }
    T *dst = xfc + (size_t)r * 2 * H;
    copy_rows2_split(dst, valid ? pend_h + (size_t)(b * D1 + j) * H : nullptr, lo, dst + H, E + (size_t)tok * H,
                     H, lo);
}

// h_hat of the root slot = draft output of the last pending row.
template <typename T>
__global__ void root_gather_kernel(const float *__restrict__ x, const int *__restrict__ n_pend, int D1,
                                   int H, float *__restrict__ hhat_root, T *__restrict__ xr, long lo) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x;
    const int r = b * D1 + max(n_pend[b] - 1, 0);
    copy_row_2dst_split(hhat_root + (size_t)b * H, xr + (size_t)b * H, lo, x + (size_t)r * H, H);
}

// Store h_hat of a tree pass's rows by slot, and a T copy for the LM head.
template <typename T>
__global__ void hhat_store_kernel(const float *__restrict__ x, const RowDesc *__restrict__ rows,
                                  int Td, int H, float *__restrict__ hhat_slot, T *__restrict__ xb, long lo) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x;
    const RowDesc d = rows[r];
    copy_row_2dst_split(hhat_slot + ((size_t)d.req * Td + d.dst) * H, xb + (size_t)r * H, lo,
                        x + (size_t)r * H, H);
}

// Assemble the draft-pass row j of request b for a frontier node with token
// `tok` at `depth`: input Concat(h_hat of its parent, e of its token), draft
// position L-1+depth, K/V slot `slot`, ancestor mask = parent's mask + own bit.
template <typename T>
__device__ void emit_frontier_row(const DraftArgs<T> &a, int b, int j, int tok, int depth,
                                  const float *parent_h, int slot, const uint64_t *parent_mask) {
    const int H = a.H, k = a.k, Wd = a.Wd;
    const int L = a.seq_len[b];
    const int r = b * k + j;
    if (threadIdx.x == 0) {
        RowDesc d;
        d.req = b;
        d.pos = L - 1 + depth;
        d.plen = L;
        d.dst = slot;
        a.rows[r] = d;
        for (int w = 0; w < Wd; ++w) {
            uint64_t m = parent_mask ? parent_mask[w] : 0ull;
            if (w == slot / 64) m |= 1ull << (slot % 64);
            a.slot_mask[((size_t)b * a.Td + slot) * Wd + w] = m;
            a.row_mask[(size_t)r * Wd + w] = m;
        }
    }
    if (tok < 0 || tok >= a.V) tok = 0;
    T *dst = a.xfc + (size_t)r * 2 * H;
    copy_rows2_split(dst, parent_h, 0, dst + H, a.E + (size_t)tok * H, H, a.lo);
}

// Depth-1 candidates from the root slot's top-k; the frontier of pass 2 is all
// of them, best first. Grid (k, B): CTA j emits row j of pass 2; CTA 0 writes
// the candidate arrays and the frontier (buffer 0).
template <typename T>
__global__ void tree_init_kernel(DraftArgs<T> a) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.y, j = blockIdx.x, k = a.k;
    __shared__ float sc[TREE_MAXK];
    __shared__ int front[TREE_MAXK];
    for (int t = threadIdx.x; t < k; t += blockDim.x) {
        const float s = a.logp[(size_t)b * k + t];
        sc[t] = s;
        if (j == 0) {
            const size_t c = (size_t)b * a.C + t;
            a.cand_tok[c] = a.ids[(size_t)b * k + t];
            a.cand_par[c] = -1;
            a.cand_depth[c] = 1;
            a.cand_score[c] = s;
        }
    }
    __syncthreads();
    for (int t = threadIdx.x; t < k; t += blockDim.x) {
        int rank = 0;
        for (int u = 0; u < k; ++u) rank += better(sc[u], u, sc[t], t);
        front[rank] = t;
    }
    __syncthreads();
    if (j == 0)
        for (int t = threadIdx.x; t < k; t += blockDim.x) a.frontier[(size_t)b * k + t] = front[t];
    if (a.D < 2) return;
    const int c = front[j];
    emit_frontier_row(a, b, j, a.ids[(size_t)b * k + c], 1, a.hhat_root + (size_t)b * a.H, j,
                      nullptr);
}

// After pass d (2..D): the k*k children of the pass rows, then (d < D) the k
// best of them form the next frontier. Grid (k, B): every CTA ranks the
// children itself (k*k values); CTA 0 writes the candidate arrays and the next
// frontier (buffer (d+1)&1; this pass read buffer d&1); CTA j emits row j of
// pass d+1.
template <typename T>
__global__ void tree_step_kernel(DraftArgs<T> a, int d) {
    wait_prior();
    allow_dependents();
    extern __shared__ float smem[];
    const int b = blockIdx.y, j = blockIdx.x, k = a.k, kk = k * k;
    const int base = k + (d - 2) * kk;
    float *sc = smem;                                  // [kk]
    int *newf = reinterpret_cast<int *>(smem + kk);    // [k]
    const int *fin = a.frontier + ((size_t)(d & 1) * a.B + b) * k;
    int *fout = a.frontier + ((size_t)((d + 1) & 1) * a.B + b) * k;
    for (int e = threadIdx.x; e < kk; e += blockDim.x) {
        const int jr = e / k, t = e - jr * k;
        const int p = fin[jr];
        const size_t src = ((size_t)b * k + jr) * k + t;
        const float s = __fadd_rn(a.cand_score[(size_t)b * a.C + p], a.logp[src]);
        sc[e] = s;
        if (j == 0) {
            const size_t c = (size_t)b * a.C + base + e;
            a.cand_tok[c] = a.ids[src];
            a.cand_par[c] = p;
            a.cand_depth[c] = d;
            a.cand_score[c] = s;
        }
    }
    __syncthreads();
    if (d >= a.D) return;
    for (int e = threadIdx.x; e < kk; e += blockDim.x) {
        int rank = 0;
        for (int u = 0; u < kk; ++u) rank += better(sc[u], u, sc[e], e);
        if (rank < k) newf[rank] = e;
    }
    __syncthreads();
    if (j == 0)
        for (int t = threadIdx.x; t < k; t += blockDim.x) fout[t] = base + newf[t];
    const int e = newf[j];
    const int jp = e / k;                              // parent's row in pass d
    const int sp = (d - 2) * k + jp;                   // parent's slot
    const int slot = (d - 1) * k + j;
    emit_frontier_row(a, b, j, a.ids[((size_t)b * k + jp) * k + (e - jp * k)], d,
                      a.hhat_slot + ((size_t)b * a.Td + sp) * a.H, slot,
                      a.slot_mask + ((size_t)b * a.Td + sp) * a.Wd);
}

// Final tree: the N-1 best candidates (score desc, creation asc), tree index
// 1 + rank; parents, depths and ancestor masks; the root is node 0. Scores,
// parents and tree indices of all candidates sit in shared memory, so the
// ancestor walks read no global memory.
constexpr int FIN_MAXW = 4;      // mask words of a node (tree_nodes <= 256)

__global__ void tree_finalize_kernel(TreeOut t, const int *__restrict__ cand_tok,
                                     const int *__restrict__ cand_par, const int *__restrict__ cand_depth,
                                     const float *__restrict__ cand_score, int *__restrict__ node_of,
                                     const int *__restrict__ root, int C, int N, int *status) {
    wait_prior();
    allow_dependents();
    extern __shared__ float ssc[];   // [C] scores, then [C] parents, [C] tree indices
    int *spar = reinterpret_cast<int *>(ssc + C), *snode = spar + C;
    const int b = blockIdx.x, W = (N + 63) / 64;
    const size_t cb = (size_t)b * C;
    for (int c = threadIdx.x; c < C; c += blockDim.x) {
        ssc[c] = cand_score[cb + c];
        spar[c] = cand_par[cb + c];
    }
    __syncthreads();
    for (int c = threadIdx.x; c < C; c += blockDim.x) {
        int rank = 0;
        const float s = ssc[c];
        for (int u = 0; u < C; ++u) rank += better(ssc[u], u, s, c);
        const int node = rank < N - 1 ? 1 + rank : -1;
        snode[c] = node;
        node_of[cb + c] = node;
    }
    __syncthreads();
    const size_t nb = (size_t)b * N;
    for (int c = threadIdx.x; c < C; c += blockDim.x) {
        const int i = snode[c];
        if (i < 0) continue;
        t.tokens[nb + i] = cand_tok[cb + c];
        t.depth[nb + i] = cand_depth[cb + c];
        const int p = spar[c];
        int pi = p < 0 ? 0 : snode[p];
        if (pi < 0 || pi >= i) { set_status(status, ST_BAD_TREE); pi = 0; }
        t.parent[nb + i] = pi;
        // ancestors-or-self: walk the candidate chain, then the root
        uint64_t mw[FIN_MAXW] = {0ull, 0ull, 0ull, 0ull};
        int cur = c, node = i;
        while (true) {
#pragma unroll
            for (int w = 0; w < FIN_MAXW; ++w)
                if (w == (node >> 6)) mw[w] |= 1ull << (node & 63);
            if (cur < 0) break;
            const int pc = spar[cur];
            node = pc < 0 ? 0 : snode[pc];
            if (node < 0) break;
            cur = pc;
        }
#pragma unroll
        for (int w = 0; w < FIN_MAXW; ++w)
            if (w < W) t.mask[(nb + i) * W + w] = mw[w];
    }
    if (threadIdx.x == 0) {
        t.tokens[nb] = root[b];
        t.parent[nb] = -1;
        t.depth[nb] = 0;
        for (int w = 0; w < W; ++w) t.mask[nb * W + w] = w == 0 ? 1ull : 0ull;
        if (t.n_nodes) t.n_nodes[b] = N;
    }
}

// ---------------------------------------------------------------------------
// Verify set-up: row r = b*N + i at position L + depth(i), sees the prefix
// [0, L) and the tree nodes of its mask (restricted to valid nodes).
// ---------------------------------------------------------------------------
__global__ void verify_setup_kernel(TreeIn t, const int *__restrict__ seq_len,
                                    const int *__restrict__ root, int B, int N, int V,
                                    RowDesc *__restrict__ rows, int *__restrict__ src,
                                    uint64_t *__restrict__ vmask, int *status) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x * blockDim.x + threadIdx.x;
    if (r >= B * N) return;
    const int b = r / N, i = r - b * N, W = (N + 63) / 64;
    const int n = t.n_nodes ? t.n_nodes[b] : N;
    const bool valid = i < n;
    const int L = seq_len[b];
    int tok = valid ? t.tokens[r] : 0;
    if (tok < 0 || tok >= V) { set_status(status, ST_BAD_TOKEN); tok = 0; }
    int depth = valid ? t.depth[r] : 0;
    if (valid) {
        const int p = t.parent[r];
        bool ok = i == 0 ? (p == -1 && depth == 0 && tok == root[b])
                         : (p >= 0 && p < i && depth == t.depth[b * N + p] + 1);
        if (!ok) { set_status(status, ST_BAD_TREE); depth = depth < 0 ? 0 : depth; }
    }
    RowDesc d;
    d.req = b;
    d.pos = L + depth;
    d.plen = L;
    d.dst = i;
    rows[r] = d;
    src[r] = tok;
    for (int w = 0; w < W; ++w) {
        uint64_t m = 0;
        if (valid) {
            m = t.mask[(size_t)r * W + w];
            const int lo = w * 64;
            if (n - lo < 64) m &= n - lo <= 0 ? 0ull : ((1ull << (n - lo)) - 1ull);
        } else if (w == i / 64) {
            m = 1ull << (i % 64);
        }
        vmask[(size_t)r * W + w] = m;
    }
}

// ---------------------------------------------------------------------------
// Root-only tree of plain greedy decoding: one thread per request.
// ---------------------------------------------------------------------------
__global__ void root_tree_kernel(const int *__restrict__ root, int B, int N, int W, int *__restrict__ tokens,
                                 int *__restrict__ parent, int *__restrict__ depth, uint64_t *__restrict__ mask,
                                 int *__restrict__ n_nodes) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    tokens[(size_t)b * N] = root[b];
    parent[(size_t)b * N] = -1;
    depth[(size_t)b * N] = 0;
    for (int w = 0; w < W; ++w) mask[(size_t)b * N * W + w] = w == 0 ? 1ull : 0ull;
    n_nodes[b] = 1;
}

// ---------------------------------------------------------------------------
// Depths and ancestor masks of a caller-planted tree (Sec. 3.2: a candidate is
// conditioned on its prefix, i.e. on its ancestors): one CTA per request, the
// parent array staged in shared memory, one thread per node walking its
// parent links to the root (at most N steps). A node whose parent does not
// precede it (or a root with a parent) sets ST_BAD_TREE and is treated as a
// child of the root, so every walk ends.
// ---------------------------------------------------------------------------
__global__ void tree_complete_kernel(const int *__restrict__ parent, int *__restrict__ depth,
                                     uint64_t *__restrict__ mask, const int *__restrict__ n_nodes, int N,
                                     int W, int b0, int *status) {
    wait_prior();
    allow_dependents();
    __shared__ int s_par[256];
    const int b = b0 + blockIdx.x;
    const int n = n_nodes ? min(max(n_nodes[b], 0), N) : N;
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        int p = i < n ? parent[(size_t)b * N + i] : -1;
        if (i < n && (i == 0 ? p != -1 : (p < 0 || p >= i))) {
            set_status(status, ST_BAD_TREE);
            p = i == 0 ? -1 : 0;
        }
        s_par[i] = p;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < N; i += blockDim.x) {
        uint64_t *m = mask + ((size_t)b * N + i) * W;
        for (int w = 0; w < W; ++w) m[w] = 0ull;
        if (i >= n) {
            depth[(size_t)b * N + i] = 0;
            continue;
        }
        int d = 0;
        for (int j = i; j >= 0; j = s_par[j]) {      // parents strictly decrease: <= N steps
            m[j >> 6] |= 1ull << (j & 63);
            if (j != i) ++d;
        }
        depth[(size_t)b * N + i] = d;
    }
}

// ---------------------------------------------------------------------------
// Greedy acceptance (Eq. 6 at T = 0): one warp per request walks from the root
// to the child whose token is the target argmax of the current node.
// ---------------------------------------------------------------------------
// Outcome of an acceptance walk of request b: path (root 0, then the a accepted
// nodes, -1 beyond) and the index map; the pending draft rows (each accepted
// position paired with the token after it: the next accepted draft token, or
// the bonus); the state update L <- L + a + 1, root <- bonus. `path` is in
// shared memory, visible to every thread of the block.
__device__ __forceinline__ void write_acceptance(const TreeIn &t, const int *path, int a, int bonus,
                                                 int b, int N, int D1, int *__restrict__ seq_len,
                                                 int *__restrict__ n_pend, int *__restrict__ root,
                                                 int *__restrict__ pend_next, int *__restrict__ acc_path,
                                                 int *__restrict__ acc_L0, int *__restrict__ acc_a,
                                                 int *__restrict__ path_out, int *__restrict__ accept_len_out,
                                                 int *__restrict__ bonus_out, int *__restrict__ index_map_out) {
    const size_t nb = (size_t)b * N;
    const int L0 = seq_len[b];
    for (int j = threadIdx.x; j < D1; j += blockDim.x) {
        const int pj = j <= a ? path[j] : -1;
        acc_path[b * D1 + j] = pj;
        if (path_out) path_out[b * D1 + j] = pj;
        if (index_map_out) index_map_out[b * D1 + j] = j <= a ? L0 + j : -1;
        if (j <= a) pend_next[b * D1 + j] = j < a ? t.tokens[nb + path[j + 1]] : bonus;
    }
    __syncthreads();   // every thread has read seq_len[b] before it changes
    if (threadIdx.x == 0) {
        acc_L0[b] = L0;
        acc_a[b] = a;
        if (accept_len_out) accept_len_out[b] = a;
        if (bonus_out) bonus_out[b] = bonus;
        n_pend[b] = a + 1;
        seq_len[b] = L0 + a + 1;
        root[b] = bonus;
    }
}

__global__ void accept_kernel(TreeIn t, const int *__restrict__ argmax, int N, int D,
                              int *__restrict__ seq_len, int *__restrict__ n_pend,
                              int *__restrict__ root, int *__restrict__ pend_next,
                              int *__restrict__ acc_path, int *__restrict__ acc_L0,
                              int *__restrict__ acc_a, int *__restrict__ path_out,
                              int *__restrict__ accept_len_out, int *__restrict__ bonus_out,
                              int *__restrict__ index_map_out) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x, lane = threadIdx.x;
    const size_t nb = (size_t)b * N;
    const int n = t.n_nodes ? t.n_nodes[b] : N;
    __shared__ int path[TREE_MAXD + 1];
    int cur = 0, a = 0;
    if (lane == 0) path[0] = 0;
    while (a < D) {
        const int want = argmax[nb + cur];
        int found = 0x7fffffff;
        for (int c = 1 + lane; c < n; c += 32)
            if (t.parent[nb + c] == cur && t.tokens[nb + c] == want) found = min(found, c);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) found = min(found, __shfl_xor_sync(0xffffffffu, found, o));
        if (found == 0x7fffffff) break;
        cur = found;
        ++a;
        if (lane == 0) path[a] = cur;
    }
    __syncwarp();
    write_acceptance(t, path, a, argmax[nb + cur], b, N, D + 1, seq_len, n_pend, root, pend_next,
                     acc_path, acc_L0, acc_a, path_out, accept_len_out, bonus_out, index_map_out);
}

// ---------------------------------------------------------------------------
// Speculative sampling over the tree at temperature T > 0 (Sec. 3.2, Eq. 6 and
// the adjusted distribution after it). The tree's candidates are the draft's
// top-k choices, so the proposal of a child -- given the siblings already
// rejected -- is a point mass at its token x: Eq. 6's min(1, p/q) accepts it
// with probability p_adj(x), and the adjusted distribution norm(max(0, p - q))
// is p_adj with x removed and renormalised. At a node, p = softmax(z / T) of
// its verify logits; the children are tried in tree order (best draft score
// first) with uniforms u[b][d][j] (d = accepted so far, j = child ordinal); an
// accepted child becomes the node. When every child is rejected, or the node
// is a leaf, the next token is drawn from p_adj by inverse CDF in token-id
// order with u[b][d][k] (the smallest token whose cumulative mass exceeds u
// times the remaining mass).
//
// Two kernels. sample_stats_kernel: per verify row, M = max z and
// S = sum exp((z - M) / T) (one CTA per row, coalesced). accept_sample_kernel
// (one CTA per request): one warp walks the tree with those statistics, then
// the block draws the token. Every exponential is exp2 of (z - M) * log2(e)/T
// in fp32 (ex2.approx, relative error below 2^-22); every sum is an fp32
// TwoSum pair (Knuth's error-free addition) per thread, pairs combined
// error-free across threads, so the decisions carry only the exponentials'
// rounding (about 1e-6 relative).
// ---------------------------------------------------------------------------
constexpr int SAMPLE_THREADS = 1024;
constexpr int STATS_THREADS = 1024;
constexpr int STATS_VEC = 8;         // float4 per thread held in registers (rows up to 32768)
constexpr int DRAW_ROUNDS = 16;      // rounds of 32 tokens a warp loads at once in the draw
constexpr int SAMPLE_MAXN = 256;     // tree nodes (the configuration's limit)
constexpr int SAMPLE_MAXU = (TREE_MAXD + 1) * (TREE_MAXK + 1);   // uniforms of one request

__device__ __forceinline__ float exp2_fast(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// hi + lo += x with the rounding error of the addition kept in lo.
__device__ __forceinline__ void two_sum_add(float &hi, float &lo, float x) {
    const float s = hi + x;
    const float bp = s - hi;
    lo += (hi - (s - bp)) + (x - bp);
    hi = s;
}

// (hi, lo) += (h2, l2); the same result on every lane of a butterfly.
__device__ __forceinline__ void pair_add(float &hi, float &lo, float h2, float l2) {
    const float s = hi + h2;
    const float bp = s - hi;
    const float e = (hi - (s - bp)) + (h2 - bp);
    lo = (lo + l2) + e;
    hi = s;
}

__device__ __forceinline__ void warp_pair_sum(float &hi, float &lo) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float h2 = __shfl_xor_sync(0xffffffffu, hi, o), l2 = __shfl_xor_sync(0xffffffffu, lo, o);
        pair_add(hi, lo, h2, l2);
    }
}

// Per verify row: M = max z, S = sum exp2((z - M) * scale) with scale =
// log2(e) / T. One CTA per row; a 16-byte-aligned row of at most 32768 logits
// is loaded once into registers (every load in flight at once), longer or
// unaligned rows are streamed twice.
__global__ void __launch_bounds__(STATS_THREADS)
sample_stats_kernel(const float *__restrict__ logits, int V, float scale, float *__restrict__ row_max,
                    double *__restrict__ row_sum) {
    wait_prior();
    allow_dependents();
    __shared__ float redf[32], rh[32], rl[32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
    const float *z = logits + (size_t)blockIdx.x * V;
    float hi = 0.f, lo = 0.f, M;
    if ((V & 3) == 0 && V <= 4 * STATS_VEC * STATS_THREADS &&
        (reinterpret_cast<uintptr_t>(z) & 15) == 0 && blockDim.x == STATS_THREADS) {
        const float4 *z4 = reinterpret_cast<const float4 *>(z);
        const int V4 = V >> 2;
        float4 v[STATS_VEC];
#pragma unroll
        for (int j = 0; j < STATS_VEC; ++j) {
            const int i = tid + j * STATS_THREADS;
            v[j] = i < V4 ? z4[i] : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
        }
        float m = -INFINITY;
#pragma unroll
        for (int j = 0; j < STATS_VEC; ++j) m = fmaxf(fmaxf(m, fmaxf(v[j].x, v[j].y)), fmaxf(v[j].z, v[j].w));
        M = block_max(m, redf);
#pragma unroll
        for (int j = 0; j < STATS_VEC; ++j) {
            if (tid + j * STATS_THREADS < V4) {
                two_sum_add(hi, lo, exp2_fast((v[j].x - M) * scale));
                two_sum_add(hi, lo, exp2_fast((v[j].y - M) * scale));
                two_sum_add(hi, lo, exp2_fast((v[j].z - M) * scale));
                two_sum_add(hi, lo, exp2_fast((v[j].w - M) * scale));
            }
        }
    } else {
        float m = -INFINITY;
#pragma unroll 8
        for (int i = tid; i < V; i += blockDim.x) m = fmaxf(m, z[i]);
        M = block_max(m, redf);
#pragma unroll 8
        for (int i = tid; i < V; i += blockDim.x) two_sum_add(hi, lo, exp2_fast((z[i] - M) * scale));
    }
    warp_pair_sum(hi, lo);
    if (lane == 0) { rh[warp] = hi; rl[warp] = lo; }
    __syncthreads();
    if (warp == 0) {
        hi = lane < nw ? rh[lane] : 0.f;
        lo = lane < nw ? rl[lane] : 0.f;
        warp_pair_sum(hi, lo);
        if (lane == 0) {
            row_max[blockIdx.x] = M;
            row_sum[blockIdx.x] = (double)hi + (double)lo;
        }
    }
}

__device__ __forceinline__ bool is_removed(const unsigned *bits, int i) {
    return (bits[i >> 5] >> (i & 31)) & 1u;
}

__global__ void __launch_bounds__(SAMPLE_THREADS)
accept_sample_kernel(TreeIn t, const float *__restrict__ logits, const float *__restrict__ row_max,
                     const double *__restrict__ row_sum, int N, int D, int k, int V, float scale,
                     const float *__restrict__ u, int *__restrict__ seq_len, int *__restrict__ n_pend,
                     int *__restrict__ root, int *__restrict__ pend_next, int *__restrict__ acc_path,
                     int *__restrict__ acc_L0, int *__restrict__ acc_a, int *__restrict__ path_out,
                     int *__restrict__ accept_len_out, int *__restrict__ bonus_out,
                     int *__restrict__ index_map_out, int *status) {
    wait_prior();
    allow_dependents();
    extern __shared__ unsigned removed_bits[];          // [(V + 31) / 32]
    const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nw = blockDim.x >> 5, D1 = D + 1, words = (V + 31) >> 5;
    const size_t nb = (size_t)b * N;
    const int n = t.n_nodes ? min(max(t.n_nodes[b], 1), N) : N;
    const float *ub = u + (size_t)b * D1 * (k + 1);
    __shared__ int path[TREE_MAXD + 1];
    __shared__ int kids[TREE_MAXK], removed[TREE_MAXK], kid_tok[TREE_MAXK];
    __shared__ double kid_p[TREE_MAXK];
    __shared__ int sh_cur, sh_a, sh_nrem, sh_warp, sh_pick;
    __shared__ double wsum[32], sh_base, sh_target;
    __shared__ int wlast[32];
    // the request's tree, row statistics and uniforms, loaded once: the walk
    // then waits on one global round trip per node (its children's logits)
    __shared__ int s_par[SAMPLE_MAXN], s_tok[SAMPLE_MAXN];
    __shared__ float s_rmax[SAMPLE_MAXN];
    __shared__ double s_rsum[SAMPLE_MAXN];
    __shared__ float s_u[SAMPLE_MAXU];
    for (int i = tid; i < words; i += blockDim.x) removed_bits[i] = 0u;
    for (int i = tid; i < n; i += blockDim.x) {
        s_par[i] = t.parent[nb + i];
        s_tok[i] = t.tokens[nb + i];
        s_rmax[i] = row_max[nb + i];
        s_rsum[i] = row_sum[nb + i];
    }
    for (int i = tid; i < D1 * (k + 1); i += blockDim.x) s_u[i] = ub[i];
    __syncthreads();

    // the walk (warp 0): Eq. 6 with point-mass proposals at every node. The
    // lanes fetch the children's tokens, probabilities and uniforms at once;
    // lane 0 then takes the decisions in tree order.
    if (warp == 0) {
        int cur = 0, a = 0, nrem = 0;
        if (lane == 0) path[0] = 0;
        for (;;) {
            const float M = s_rmax[cur];
            const double S = s_rsum[cur];
            int cnt = 0;
            for (int c0 = 1; c0 < n; c0 += 32) {
                const int c = c0 + lane;
                const bool is = c < n && s_par[c] == cur;
                const unsigned bal = __ballot_sync(0xffffffffu, is);
                const int slot = cnt + __popc(bal & ((1u << lane) - 1u));
                if (is && slot < k) kids[slot] = c;
                cnt += __popc(bal);
            }
            __syncwarp();
            const int nk = a < D ? min(cnt, k) : 0;
            if (lane < nk) {
                const int x = s_tok[kids[lane]];
                const bool ok = x >= 0 && x < V;
                kid_tok[lane] = ok ? x : -1;
                kid_p[lane] = ok ? (double)exp2_fast((logits[(nb + cur) * V + x] - M) * scale) / S : 0.0;
            }
            __syncwarp();
            int next = -1;
            nrem = 0;
            if (lane == 0) {
                if (cnt > k) set_status(status, ST_BAD_TREE);
                double gone = 0.0;        // mass of the tokens already rejected at this node
                for (int j = 0; j < nk; ++j) {
                    const int x = kid_tok[j];
                    if (x < 0) {
                        set_status(status, ST_BAD_TOKEN);
                        continue;
                    }
                    bool dup = false;
                    for (int r = 0; r < nrem; ++r) dup |= removed[r] == x;
                    const double px = dup ? 0.0 : kid_p[j];
                    if ((double)s_u[a * (k + 1) + j] * (1.0 - gone) < px) {
                        next = kids[j];
                        break;
                    }
                    if (!dup) {
                        removed[nrem++] = x;
                        gone += px;
                    }
                }
            }
            next = __shfl_sync(0xffffffffu, next, 0);
            nrem = __shfl_sync(0xffffffffu, nrem, 0);
            if (next < 0) break;
            cur = next;
            ++a;
            if (lane == 0) path[a] = cur;
            __syncwarp();
        }
        if (lane == 0) {
            sh_cur = cur;
            sh_a = a;
            sh_nrem = nrem;
            sh_warp = -1;
            sh_pick = -1;
        }
    }
    __syncthreads();
    const int cur = sh_cur, a = sh_a, nrem = sh_nrem;
    if (tid < nrem) atomicOr(&removed_bits[removed[tid] >> 5], 1u << (removed[tid] & 31));
    __syncthreads();

    // the draw: inverse CDF of p_adj at the last node in token-id order. Warp w
    // owns tokens [w*seg, (w+1)*seg) in rounds of 32 consecutive tokens (lane l
    // takes token 32j + l of round j: coalesced), DRAW_ROUNDS rounds loaded at once.
    const float *z = logits + (nb + cur) * V;
    const float M = s_rmax[cur];
    const int seg = 32 * ((V + 32 * nw - 1) / (32 * nw));
    const int t0 = warp * seg, t1 = min(t0 + seg, V);
    float hi = 0.f, lo = 0.f;
    int last = -1;
    for (int c0 = t0; c0 < t1; c0 += 32 * DRAW_ROUNDS) {
        float v[DRAW_ROUNDS];
#pragma unroll
        for (int j = 0; j < DRAW_ROUNDS; ++j) {
            const int i = c0 + 32 * j + lane;
            v[j] = i < t1 ? z[i] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < DRAW_ROUNDS; ++j) {
            const int i = c0 + 32 * j + lane;
            const float e = (i < t1 && !is_removed(removed_bits, i)) ? exp2_fast((v[j] - M) * scale) : 0.f;
            two_sum_add(hi, lo, e);
            if (e > 0.f) last = i;
        }
    }
    warp_pair_sum(hi, lo);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
    if (lane == 0) {
        wsum[warp] = (double)hi + (double)lo;
        wlast[warp] = last;
    }
    __syncthreads();
    if (warp == 0) {
        // exclusive scan of the warp segments' masses; the segment holding the target
        const double v = lane < nw ? wsum[lane] : 0.0;
        double inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const double y = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += y;
        }
        const double total = __shfl_sync(0xffffffffu, inc, 31);
        const double target = (double)s_u[a * (k + 1) + k] * total;
        double excl = __shfl_up_sync(0xffffffffu, inc, 1);   // the intervals tile [0, total)
        if (lane == 0) excl = 0.0;
        const bool here = lane < nw && v > 0.0 && excl <= target && target < inc;
        const unsigned bal = __ballot_sync(0xffffffffu, here);
        if (lane == 0) {
            sh_target = target;
            if (bal) {
                sh_warp = __ffs(bal) - 1;
            } else {
                // no segment (u >= 1 or no mass left): the last token with mass
                int lp = -1;
                for (int w = 0; w < nw; ++w) lp = max(lp, wlast[w]);
                sh_pick = lp;
            }
        }
        if (bal && lane == __ffs(bal) - 1) sh_base = excl;
    }
    __syncthreads();
    if (warp == sh_warp) {
        // walk the segment round by round: fp32 inclusive scan of each round on
        // top of the fp64 mass of the rounds before it
        const double target = sh_target;
        double cum = sh_base;
        int pick = -1;
        for (int c0 = t0; c0 < t1 && pick < 0; c0 += 32 * DRAW_ROUNDS) {
            float v[DRAW_ROUNDS];
#pragma unroll
            for (int j = 0; j < DRAW_ROUNDS; ++j) {
                const int i = c0 + 32 * j + lane;
                v[j] = i < t1 ? z[i] : 0.f;
            }
#pragma unroll
            for (int j = 0; j < DRAW_ROUNDS; ++j) {
                const int i = c0 + 32 * j + lane;
                const float e = (i < t1 && !is_removed(removed_bits, i)) ? exp2_fast((v[j] - M) * scale) : 0.f;
                float inc = e;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const float y = __shfl_up_sync(0xffffffffu, inc, o);
                    if (lane >= o) inc += y;
                }
                const unsigned hit = __ballot_sync(0xffffffffu, pick < 0 && e > 0.f && cum + (double)inc > target);
                if (hit && pick < 0) pick = c0 + 32 * j + __ffs(hit) - 1;
                cum += (double)__shfl_sync(0xffffffffu, inc, 31);
            }
        }
        if (lane == 0) sh_pick = pick >= 0 ? pick : wlast[warp];
    }
    __syncthreads();
    if (tid == 0 && sh_pick < 0) {
        // nothing drawable at all: the node's argmax
        int am = 0;
        for (int i = 0; i < V; ++i)
            if (z[i] == M) { am = i; break; }
        sh_pick = am;
    }
    __syncthreads();
    write_acceptance(t, path, a, sh_pick, b, N, D1, seq_len, n_pend, root, pend_next, acc_path, acc_L0,
                     acc_a, path_out, accept_len_out, bonus_out, index_map_out);
}

// K/V of accepted node path[j] -> cache position L0 + j, all layers and heads.
// grid (n_layers*2*nh, B); 16-byte vector copies.
__global__ void compact_kv_kernel(const uint4 *__restrict__ tree_kv, uint4 *__restrict__ cache,
                                  const int *__restrict__ acc_path, const int *__restrict__ acc_L0,
                                  const int *__restrict__ acc_a, int B, int nh, int N, int S,
                                  int D1, int vec_per_row, long tree_lo, long cache_lo, int *status) {
    wait_prior();
    allow_dependents();
    const int lkh = blockIdx.x, b = blockIdx.y;
    const int h = lkh % nh, lk = lkh / nh;           // lk = layer*2 + kv
    const int a = acc_a[b], L0 = acc_L0[b];
    if (L0 + a >= S) {
        if (threadIdx.x == 0) set_status(status, ST_RANGE);
        return;
    }
    const size_t tb = ((size_t)(lk * B + b) * nh + h) * N;
    const size_t cb = ((size_t)(lk * B + b) * nh + h) * S;
    const int total = (a + 1) * vec_per_row;
    for (int idx = threadIdx.x; idx < total; idx += blockDim.x) {
        const int j = idx / vec_per_row, v = idx - j * vec_per_row;
        const int node = acc_path[b * D1 + j];
        const size_t dst = (cb + L0 + j) * vec_per_row + v, src = (tb + node) * vec_per_row + v;
        const uint4 hi = tree_kv[src];
        if (tree_lo) {
            const uint4 lo = tree_kv[src + tree_lo];
            cache[dst + cache_lo] = lo;
        }
        cache[dst] = hi;
    }
}

// Pending draft rows: target features h of the accepted nodes.
template <typename T>
__global__ void pend_h_kernel(const T *__restrict__ hT, const int *__restrict__ acc_path,
                              const int *__restrict__ acc_a, int N, int D1, int H,
                              T *__restrict__ pend_h, long lo) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x / D1, j = blockIdx.x - b * D1;
    if (j > acc_a[b]) return;
    const int node = acc_path[b * D1 + j];
    const T *s = hT + ((size_t)b * N + node) * H;
    copy_row_split(pend_h + ((size_t)b * D1 + j) * H, lo, s, lo, H);
}

// ---------------------------------------------------------------------------
// Prefill helpers
// ---------------------------------------------------------------------------
// Decoupled draft input (Eq. 7): visual rows take the raw embedding.
template <typename T>
__global__ void select_visual_kernel(float *__restrict__ x, const T *__restrict__ emb, long slo,
                                     const int *__restrict__ src, int H) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x;
    if (src[r] >= 0) return;
    copy_row_split(x + (size_t)r * H, 0, emb + (size_t)r * H, slo, H);
}

// Concat(h_i, e_{i+1}) rows for the draft prefill (text positions; visual rows
// are overwritten after f_down by select_visual_kernel).
template <typename T>
__global__ void concat_next_kernel(const T *__restrict__ h, const T *__restrict__ emb, int H,
                                   T *__restrict__ xfc, long lo) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x;
    copy_rows2_split(xfc + (size_t)r * 2 * H, h + (size_t)r * H, lo, xfc + (size_t)r * 2 * H + H,
                     emb + (size_t)(r + 1) * H, H, lo);
}

template <typename T>
__global__ void prefill_finish_kernel(const int *__restrict__ argmax1, const T *__restrict__ h_last,
                                      int b, int L, int D1, int H, int *__restrict__ seq_len,
                                      int *__restrict__ n_pend, int *__restrict__ root,
                                      int *__restrict__ pend_next, T *__restrict__ pend_h, long lo,
                                      int *__restrict__ root_out) {
    wait_prior();
    const int x = argmax1[0];
    if (threadIdx.x == 0) {
        seq_len[b] = L;
        n_pend[b] = 1;
        root[b] = x;
        pend_next[b * D1] = x;
        if (root_out) root_out[b] = x;
    }
    copy_row_split(pend_h + (size_t)b * D1 * H, lo, h_last, lo, H);
}

// ---------------------------------------------------------------------------
// Launchers
// ---------------------------------------------------------------------------
template <typename T>
void launch_catchup_setup(const int *seq_len, const int *n_pend, const T *pend_h,
                          const int *pend_next, const T *E, int B, int H, int D1, int V, T *xfc,
                          long lo, RowDesc *rows, int *status, cudaStream_t s) {
    launch_chain(catchup_setup_kernel<T>, B * D1, 256, 0, s, seq_len, n_pend, pend_h, pend_next, E, H, D1,
                                                   V, xfc, lo, rows, status); note_launch();
}

template <typename T>
void launch_root_gather(const float *x, const int *n_pend, int B, int D1, int H, float *hhat_root,
                        T *xr, long lo, cudaStream_t s) {
    launch_chain(root_gather_kernel<T>, B, 256, 0, s, x, n_pend, D1, H, hhat_root, xr, lo); note_launch();
}

template <typename T>
void launch_hhat_store(const float *x, const RowDesc *rows, int R, int Td, int H,
                       float *hhat_slot, T *xb, long lo, cudaStream_t s) {
    launch_chain(hhat_store_kernel<T>, R, 256, 0, s, x, rows, Td, H, hhat_slot, xb, lo); note_launch();
}

template <typename T>
void launch_tree_init(const DraftArgs<T> &a, int B, cudaStream_t s) {
    launch_chain(tree_init_kernel<T>, dim3(a.k, B), 256, 0, s, a);
    note_launch();
}

template <typename T>
void launch_tree_step(const DraftArgs<T> &a, int B, int d, cudaStream_t s) {
    const size_t sm = (size_t)a.k * a.k * sizeof(float) + (size_t)a.k * sizeof(int);
    launch_chain(tree_step_kernel<T>, dim3(a.k, B), 256, sm, s, a, d);
    note_launch();
}

void launch_tree_finalize(const TreeOut &t, const int *cand_tok, const int *cand_par,
                          const int *cand_depth, const float *cand_score, int *node_of,
                          const int *root, int B, int C, int N, int *status, cudaStream_t s) {
    const size_t smem = (size_t)C * 3 * sizeof(float);
    // candidate arrays beyond 48 KB (deep, wide trees); the attribute is per device
    cudaFuncSetAttribute(tree_finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    launch_chain(tree_finalize_kernel, B, 512, smem, s, t, cand_tok, cand_par, cand_depth, cand_score, node_of,
               root, C, N, status);
    note_launch();
}

void launch_verify_setup(const TreeIn &t, const int *seq_len, const int *root, int B, int N,
                         int V, RowDesc *rows, int *src, uint64_t *vmask, int *status,
                         cudaStream_t s) {
    const int R = B * N;
    launch_chain(verify_setup_kernel, (R + 127) / 128, 128, 0, s, t, seq_len, root, B, N, V, rows, src,
                                                          vmask, status); note_launch();
}

void launch_tree_complete(const int *parent, int *depth, uint64_t *mask, const int *n_nodes, int b0, int nb,
                          int N, int *status, cudaStream_t s) {
    launch_chain(tree_complete_kernel, nb, 256, 0, s, parent, depth, mask, n_nodes, N, (N + 63) / 64, b0, status);
    note_launch();
}

void launch_root_tree(const int *root, int B, int N, int W, int *tokens, int *parent, int *depth,
                      uint64_t *mask, int *n_nodes, cudaStream_t s) {
    launch_chain(root_tree_kernel, (B + 127) / 128, 128, 0, s, root, B, N, W, tokens, parent, depth, mask, n_nodes);
    note_launch();
}

void launch_accept(const TreeIn &t, const int *argmax, int B, int N, int D, int *seq_len,
                   int *n_pend, int *root, int *pend_next, int *acc_path, int *acc_L0, int *acc_a,
                   int *path_out, int *accept_len_out, int *bonus_out, int *index_map_out,
                   cudaStream_t s) {
    launch_chain(accept_kernel, B, 32, 0, s, t, argmax, N, D, seq_len, n_pend, root, pend_next, acc_path,
                                   acc_L0, acc_a, path_out, accept_len_out, bonus_out,
                                   index_map_out); note_launch();
}

bool launch_accept_sample(const TreeIn &t, const float *logits, int B, int N, int D, int k, int V,
                          float inv_temp, const float *u, float *row_max, double *row_sum, int *seq_len,
                          int *n_pend, int *root, int *pend_next, int *acc_path, int *acc_L0, int *acc_a,
                          int *path_out, int *accept_len_out, int *bonus_out, int *index_map_out,
                          int *status, cudaStream_t s) {
    if (V > SAMPLE_MAX_VOCAB) return false;
    // the rejected-token bitmap (dynamic) sits beside about 10 KB of static
    // shared memory: raise the dynamic limit to the bitmap of the largest
    // vocabulary taken (the attribute is per device: set on every call)
    if (cudaFuncSetAttribute(accept_sample_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)(sizeof(unsigned) * (SAMPLE_MAX_VOCAB / 32))) != cudaSuccess)
        return false;
    const float scale = (float)(1.4426950408889634 * (double)inv_temp);     // log2(e) / T
    if (launch_chain(sample_stats_kernel, B * N, STATS_THREADS, 0, s, logits, V, scale, row_max, row_sum) !=
        cudaSuccess)
        return false;
    note_launch();
    const size_t smem = sizeof(unsigned) * (size_t)((V + 31) / 32);
    if (launch_chain(accept_sample_kernel, B, SAMPLE_THREADS, smem, s, t, logits, (const float *)row_max,
                   (const double *)row_sum, N, D, k, V, scale, u, seq_len, n_pend, root, pend_next, acc_path,
                   acc_L0, acc_a, path_out, accept_len_out, bonus_out, index_map_out, status) != cudaSuccess)
        return false;
    note_launch();
    return true;
}

void launch_compact_kv(const void *tree_kv, void *cache, const int *acc_path, const int *acc_L0,
                       const int *acc_a, int n_layers, int B, int nh, int N, int S, int D1,
                       int row_bytes, long lo_bytes, int *status, cudaStream_t s) {
    dim3 grid(n_layers * 2 * nh, B);
    const long lo_vec = lo_bytes / 16;      // both lo planes sit lo_bytes after their hi planes
    launch_chain(compact_kv_kernel, grid, 128, 0, s, static_cast<const uint4 *>(tree_kv),
                                           static_cast<uint4 *>(cache), acc_path, acc_L0, acc_a,
                                           B, nh, N, S, D1, row_bytes / 16, lo_vec, lo_vec, status); note_launch();
}

template <typename T>
void launch_pend_h(const T *hT, const int *acc_path, const int *acc_a, int B, int N, int D1,
                   int H, T *pend_h, long lo, cudaStream_t s) {
    launch_chain(pend_h_kernel<T>, B * D1, 256, 0, s, hT, acc_path, acc_a, N, D1, H, pend_h, lo); note_launch();
}

template <typename T>
void launch_select_visual(float *x, const T *emb, long slo, const int *src, int R, int H, cudaStream_t s) {
    if (R <= 0) return;
    launch_chain(select_visual_kernel<T>, R, 256, 0, s, x, emb, slo, src, H); note_launch();
}

template <typename T>
void launch_concat_next(const T *h, const T *emb, int R, int H, T *xfc, long lo, cudaStream_t s) {
    if (R <= 0) return;
    launch_chain(concat_next_kernel<T>, R, 256, 0, s, h, emb, H, xfc, lo); note_launch();
}

template <typename T>
void launch_prefill_finish(const int *argmax1, const T *h_last, int b, int L, int D1, int H,
                           int *seq_len, int *n_pend, int *root, int *pend_next, T *pend_h, long lo,
                           int *root_out, cudaStream_t s) {
    launch_chain(prefill_finish_kernel<T>, 1, 256, 0, s, argmax1, h_last, b, L, D1, H, seq_len, n_pend,
                                               root, pend_next, pend_h, lo, root_out); note_launch();
}

#define MSD_INST(T)                                                                             \
    template void launch_catchup_setup<T>(const int *, const int *, const T *, const int *,     \
                                          const T *, int, int, int, int, T *, long, RowDesc *,  \
                                          int *, cudaStream_t);                                 \
    template void launch_root_gather<T>(const float *, const int *, int, int, int, float *, T *, \
                                        long, cudaStream_t);                                    \
    template void launch_hhat_store<T>(const float *, const RowDesc *, int, int, int, float *,  \
                                       T *, long, cudaStream_t);                                \
    template void launch_tree_init<T>(const DraftArgs<T> &, int, cudaStream_t);                 \
    template void launch_tree_step<T>(const DraftArgs<T> &, int, int, cudaStream_t);            \
    template void launch_pend_h<T>(const T *, const int *, const int *, int, int, int, int, T *, \
                                   long, cudaStream_t);                                         \
    template void launch_select_visual<T>(float *, const T *, long, const int *, int, int,      \
                                          cudaStream_t);                                        \
    template void launch_concat_next<T>(const T *, const T *, int, int, T *, long, cudaStream_t); \
    template void launch_prefill_finish<T>(const int *, const T *, int, int, int, int, int *,   \
                                           int *, int *, int *, T *, long, int *, cudaStream_t);
MSD_INST(float)
MSD_INST(bf16)
#undef MSD_INST

}  // namespace msd
