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
                                     T *__restrict__ xfc, RowDesc *__restrict__ rows, int *status) {
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
    copy_rows2(dst, valid ? pend_h + (size_t)(b * D1 + j) * H : nullptr, dst + H, E + (size_t)tok * H, H);
}

// h_hat of the root slot = draft output of the last pending row.
template <typename T>
__global__ void root_gather_kernel(const float *__restrict__ x, const int *__restrict__ n_pend, int D1,
                                   int H, float *__restrict__ hhat_root, T *__restrict__ xr) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x;
    const int r = b * D1 + max(n_pend[b] - 1, 0);
    copy_row_2dst(hhat_root + (size_t)b * H, xr + (size_t)b * H, x + (size_t)r * H, H);
}

// Store h_hat of a tree pass's rows by slot, and a T copy for the LM head.
template <typename T>
__global__ void hhat_store_kernel(const float *__restrict__ x, const RowDesc *__restrict__ rows,
                                  int Td, int H, float *__restrict__ hhat_slot, T *__restrict__ xb) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x;
    const RowDesc d = rows[r];
    copy_row_2dst(hhat_slot + ((size_t)d.req * Td + d.dst) * H, xb + (size_t)r * H, x + (size_t)r * H, H);
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
    copy_rows2(dst, parent_h, dst + H, a.E + (size_t)tok * H, H);
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
// One CTA per request. Each thread owns a contiguous run of the vocabulary; a
// node's row is reduced twice (max, then the sum of exp((z - max) / T)), every
// exponential in fp32 and every sum as an fp32 TwoSum pair (Knuth's error-free
// addition) combined across threads in fp64, so the decisions carry only the
// exponentials' rounding (about 1e-6 relative).
// ---------------------------------------------------------------------------
constexpr int SAMPLE_THREADS = 1024;

// hi + lo += x with the rounding error of the addition kept in lo.
__device__ __forceinline__ void two_sum_add(float &hi, float &lo, float x) {
    const float s = hi + x;
    const float bp = s - hi;
    lo += (hi - (s - bp)) + (x - bp);
    hi = s;
}

__device__ __forceinline__ double block_sum_f64(double v, double *red) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    if (warp == 0) {
        double w = lane < nw ? red[lane] : 0.0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) w += __shfl_xor_sync(0xffffffffu, w, o);
        if (lane == 0) red[32] = w;
    }
    __syncthreads();
    return red[32];
}

// Exclusive prefix sum over the block in thread order; *total = the sum of all.
__device__ __forceinline__ double block_exscan_f64(double v, double *red, double *total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    double inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double y = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += y;
    }
    double excl = __shfl_up_sync(0xffffffffu, inc, 1);
    if (lane == 0) excl = 0.0;
    __syncthreads();
    if (lane == 31) red[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        double w = lane < nw ? red[lane] : 0.0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const double y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        red[lane] = w;            // inclusive prefix of the warp totals
    }
    __syncthreads();
    *total = red[nw - 1];
    return (warp > 0 ? red[warp - 1] : 0.0) + excl;
}

__global__ void __launch_bounds__(SAMPLE_THREADS)
accept_sample_kernel(TreeIn t, const float *__restrict__ logits, int N, int D, int k, int V,
                     float inv_temp, const float *__restrict__ u, int *__restrict__ seq_len,
                     int *__restrict__ n_pend, int *__restrict__ root, int *__restrict__ pend_next,
                     int *__restrict__ acc_path, int *__restrict__ acc_L0, int *__restrict__ acc_a,
                     int *__restrict__ path_out, int *__restrict__ accept_len_out,
                     int *__restrict__ bonus_out, int *__restrict__ index_map_out, int *status) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x, tid = threadIdx.x, D1 = D + 1;
    const size_t nb = (size_t)b * N;
    const int n = t.n_nodes ? min(max(t.n_nodes[b], 1), N) : N;
    const float *ub = u + (size_t)b * D1 * (k + 1);
    __shared__ int path[TREE_MAXD + 1];
    __shared__ int kids[TREE_MAXK], removed[TREE_MAXK];
    __shared__ int sh_next, sh_nrem, sh_pick, sh_last;
    __shared__ float redf[32];
    __shared__ double red[33];
    __shared__ double bound[SAMPLE_THREADS + 1];
    const int per = (V + blockDim.x - 1) / blockDim.x;
    const int lo = min(tid * per, V), hi = min(lo + per, V);
    if (tid == 0) path[0] = 0;
    int cur = 0, a = 0;
    const float *row;
    float M;
    for (;;) {
        row = logits + (nb + cur) * V;
        float m = -INFINITY;
        for (int i = lo; i < hi; ++i) m = fmaxf(m, row[i]);
        M = block_max(m, redf);
        float sh = 0.f, sl = 0.f;
        for (int i = lo; i < hi; ++i) two_sum_add(sh, sl, expf((row[i] - M) * inv_temp));
        const double S = block_sum_f64((double)sh + (double)sl, red);
        if (tid < 32) {
            // children of the node, in tree order (at most k are tried)
            int cnt = 0;
            for (int c0 = 1; c0 < n; c0 += 32) {
                const int c = c0 + tid;
                const bool is = c < n && t.parent[nb + c] == cur;
                const unsigned bal = __ballot_sync(0xffffffffu, is);
                const int slot = cnt + __popc(bal & ((1u << tid) - 1u));
                if (is && slot < k) kids[slot] = c;
                cnt += __popc(bal);
            }
            __syncwarp();
            if (tid == 0) {
                if (cnt > k) set_status(status, ST_BAD_TREE);
                const int nk = a < D ? min(cnt, k) : 0;
                int next = -1, nrem = 0;
                double gone = 0.0;        // mass of the tokens already rejected at this node
                for (int j = 0; j < nk; ++j) {
                    const int x = t.tokens[nb + kids[j]];
                    if (x < 0 || x >= V) {
                        set_status(status, ST_BAD_TOKEN);
                        continue;
                    }
                    bool dup = false;
                    for (int r = 0; r < nrem; ++r) dup |= removed[r] == x;
                    const double px = dup ? 0.0 : (double)expf((row[x] - M) * inv_temp) / S;
                    if ((double)ub[a * (k + 1) + j] * (1.0 - gone) < px) {
                        next = kids[j];
                        break;
                    }
                    if (!dup) {
                        removed[nrem++] = x;
                        gone += px;
                    }
                }
                sh_next = next;
                sh_nrem = nrem;
                sh_pick = -1;
                sh_last = -1;
            }
        }
        __syncthreads();
        const int next = sh_next;
        if (next < 0) break;
        cur = next;
        ++a;
        if (tid == 0) path[a] = cur;
    }
    // the next token: inverse CDF of p_adj at the last node, in token-id order
    const int nrem = sh_nrem;
    float ph = 0.f, pl = 0.f;
    int last = -1;
    for (int i = lo; i < hi; ++i) {
        bool rm = false;
        for (int r = 0; r < nrem; ++r) rm |= removed[r] == i;
        if (rm) continue;
        const float e = expf((row[i] - M) * inv_temp);
        two_sum_add(ph, pl, e);
        if (e > 0.f) last = i;
    }
    double total;
    const double excl = block_exscan_f64((double)ph + (double)pl, red, &total);
    bound[tid] = excl;
    if (tid == 0) bound[blockDim.x] = total;
    if (last >= 0) atomicMax(&sh_last, last);
    __syncthreads();
    const double target = (double)ub[a * (k + 1) + k] * total;
    if (bound[tid] <= target && target < bound[tid + 1]) {
        double c = excl;
        int pick = -1, lastp = -1;
        for (int i = lo; i < hi; ++i) {
            bool rm = false;
            for (int r = 0; r < nrem; ++r) rm |= removed[r] == i;
            if (rm) continue;
            const float e = expf((row[i] - M) * inv_temp);
            if (e > 0.f) lastp = i;
            c += (double)e;
            if (c > target) {
                pick = i;
                break;
            }
        }
        sh_pick = pick >= 0 ? pick : lastp;   // the bounds partition [0, total): one thread
    }
    __syncthreads();
    if (tid == 0) {
        int bo = sh_pick >= 0 ? sh_pick : sh_last;
        if (bo < 0) {
            // no mass left (only with u >= 1 or every positive token removed): the argmax
            bo = 0;
            for (int i = 0; i < V; ++i)
                if (row[i] == M) { bo = i; break; }
        }
        sh_next = bo;
    }
    __syncthreads();
    const int bonus = sh_next;
    write_acceptance(t, path, a, bonus, b, N, D1, seq_len, n_pend, root, pend_next, acc_path, acc_L0,
                     acc_a, path_out, accept_len_out, bonus_out, index_map_out);
}

// K/V of accepted node path[j] -> cache position L0 + j, all layers and heads.
// grid (n_layers*2*nh, B); 16-byte vector copies.
__global__ void compact_kv_kernel(const uint4 *__restrict__ tree_kv, uint4 *__restrict__ cache,
                                  const int *__restrict__ acc_path, const int *__restrict__ acc_L0,
                                  const int *__restrict__ acc_a, int B, int nh, int N, int S,
                                  int D1, int vec_per_row, int *status) {
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
        cache[(cb + L0 + j) * vec_per_row + v] = tree_kv[(tb + node) * vec_per_row + v];
    }
}

// Pending draft rows: target features h of the accepted nodes.
template <typename T>
__global__ void pend_h_kernel(const T *__restrict__ hT, const int *__restrict__ acc_path,
                              const int *__restrict__ acc_a, int N, int D1, int H,
                              T *__restrict__ pend_h) {
    wait_prior();
    allow_dependents();
    const int b = blockIdx.x / D1, j = blockIdx.x - b * D1;
    if (j > acc_a[b]) return;
    const int node = acc_path[b * D1 + j];
    const T *s = hT + ((size_t)b * N + node) * H;
    copy_row(pend_h + ((size_t)b * D1 + j) * H, s, H);
}

// ---------------------------------------------------------------------------
// Prefill helpers
// ---------------------------------------------------------------------------
// Decoupled draft input (Eq. 7): visual rows take the raw embedding.
template <typename T>
__global__ void select_visual_kernel(float *__restrict__ x, const T *__restrict__ emb,
                                     const int *__restrict__ src, int H) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x;
    if (src[r] >= 0) return;
    copy_row(x + (size_t)r * H, emb + (size_t)r * H, H);
}

// Concat(h_i, e_{i+1}) rows for the draft prefill (text positions; visual rows
// are overwritten after f_down by select_visual_kernel).
template <typename T>
__global__ void concat_next_kernel(const T *__restrict__ h, const T *__restrict__ emb, int H,
                                   T *__restrict__ xfc) {
    wait_prior();
    allow_dependents();
    const int r = blockIdx.x;
    copy_rows2(xfc + (size_t)r * 2 * H, h + (size_t)r * H, xfc + (size_t)r * 2 * H + H, emb + (size_t)(r + 1) * H, H);
}

template <typename T>
__global__ void prefill_finish_kernel(const int *__restrict__ argmax1, const T *__restrict__ h_last,
                                      int b, int L, int D1, int H, int *__restrict__ seq_len,
                                      int *__restrict__ n_pend, int *__restrict__ root,
                                      int *__restrict__ pend_next, T *__restrict__ pend_h,
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
    copy_row(pend_h + (size_t)b * D1 * H, h_last, H);
}

// ---------------------------------------------------------------------------
// Launchers
// ---------------------------------------------------------------------------
template <typename T>
void launch_catchup_setup(const int *seq_len, const int *n_pend, const T *pend_h,
                          const int *pend_next, const T *E, int B, int H, int D1, int V, T *xfc,
                          RowDesc *rows, int *status, cudaStream_t s) {
    launch_pdl(catchup_setup_kernel<T>, B * D1, 256, 0, s, seq_len, n_pend, pend_h, pend_next, E, H, D1,
                                                   V, xfc, rows, status); note_launch();
}

template <typename T>
void launch_root_gather(const float *x, const int *n_pend, int B, int D1, int H, float *hhat_root,
                        T *xr, cudaStream_t s) {
    launch_pdl(root_gather_kernel<T>, B, 256, 0, s, x, n_pend, D1, H, hhat_root, xr); note_launch();
}

template <typename T>
void launch_hhat_store(const float *x, const RowDesc *rows, int R, int Td, int H,
                       float *hhat_slot, T *xb, cudaStream_t s) {
    launch_pdl(hhat_store_kernel<T>, R, 256, 0, s, x, rows, Td, H, hhat_slot, xb); note_launch();
}

template <typename T>
void launch_tree_init(const DraftArgs<T> &a, int B, cudaStream_t s) {
    launch_pdl(tree_init_kernel<T>, dim3(a.k, B), 256, 0, s, a);
    note_launch();
}

template <typename T>
void launch_tree_step(const DraftArgs<T> &a, int B, int d, cudaStream_t s) {
    const size_t sm = (size_t)a.k * a.k * sizeof(float) + (size_t)a.k * sizeof(int);
    launch_pdl(tree_step_kernel<T>, dim3(a.k, B), 256, sm, s, a, d);
    note_launch();
}

void launch_tree_finalize(const TreeOut &t, const int *cand_tok, const int *cand_par,
                          const int *cand_depth, const float *cand_score, int *node_of,
                          const int *root, int B, int C, int N, int *status, cudaStream_t s) {
    const size_t smem = (size_t)C * 3 * sizeof(float);
    static bool attr = false;       // candidate arrays beyond 48 KB (deep, wide trees)
    if (!attr) {
        cudaFuncSetAttribute(tree_finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
        attr = true;
    }
    launch_pdl(tree_finalize_kernel, B, 512, smem, s, t, cand_tok, cand_par, cand_depth, cand_score, node_of,
               root, C, N, status);
    note_launch();
}

void launch_verify_setup(const TreeIn &t, const int *seq_len, const int *root, int B, int N,
                         int V, RowDesc *rows, int *src, uint64_t *vmask, int *status,
                         cudaStream_t s) {
    const int R = B * N;
    launch_pdl(verify_setup_kernel, (R + 127) / 128, 128, 0, s, t, seq_len, root, B, N, V, rows, src,
                                                          vmask, status); note_launch();
}

void launch_root_tree(const int *root, int B, int N, int W, int *tokens, int *parent, int *depth,
                      uint64_t *mask, int *n_nodes, cudaStream_t s) {
    launch_pdl(root_tree_kernel, (B + 127) / 128, 128, 0, s, root, B, N, W, tokens, parent, depth, mask, n_nodes);
    note_launch();
}

void launch_accept(const TreeIn &t, const int *argmax, int B, int N, int D, int *seq_len,
                   int *n_pend, int *root, int *pend_next, int *acc_path, int *acc_L0, int *acc_a,
                   int *path_out, int *accept_len_out, int *bonus_out, int *index_map_out,
                   cudaStream_t s) {
    launch_pdl(accept_kernel, B, 32, 0, s, t, argmax, N, D, seq_len, n_pend, root, pend_next, acc_path,
                                   acc_L0, acc_a, path_out, accept_len_out, bonus_out,
                                   index_map_out); note_launch();
}

void launch_accept_sample(const TreeIn &t, const float *logits, int B, int N, int D, int k, int V,
                          float inv_temp, const float *u, int *seq_len, int *n_pend, int *root,
                          int *pend_next, int *acc_path, int *acc_L0, int *acc_a, int *path_out,
                          int *accept_len_out, int *bonus_out, int *index_map_out, int *status,
                          cudaStream_t s) {
    launch_pdl(accept_sample_kernel, B, SAMPLE_THREADS, 0, s, t, logits, N, D, k, V, inv_temp, u, seq_len,
               n_pend, root, pend_next, acc_path, acc_L0, acc_a, path_out, accept_len_out, bonus_out,
               index_map_out, status); note_launch();
}

void launch_compact_kv(const void *tree_kv, void *cache, const int *acc_path, const int *acc_L0,
                       const int *acc_a, int n_layers, int B, int nh, int N, int S, int D1,
                       int row_bytes, int *status, cudaStream_t s) {
    dim3 grid(n_layers * 2 * nh, B);
    launch_pdl(compact_kv_kernel, grid, 128, 0, s, static_cast<const uint4 *>(tree_kv),
                                           static_cast<uint4 *>(cache), acc_path, acc_L0, acc_a,
                                           B, nh, N, S, D1, row_bytes / 16, status); note_launch();
}

template <typename T>
void launch_pend_h(const T *hT, const int *acc_path, const int *acc_a, int B, int N, int D1,
                   int H, T *pend_h, cudaStream_t s) {
    launch_pdl(pend_h_kernel<T>, B * D1, 256, 0, s, hT, acc_path, acc_a, N, D1, H, pend_h); note_launch();
}

template <typename T>
void launch_select_visual(float *x, const T *emb, const int *src, int R, int H, cudaStream_t s) {
    if (R <= 0) return;
    launch_pdl(select_visual_kernel<T>, R, 256, 0, s, x, emb, src, H); note_launch();
}

template <typename T>
void launch_concat_next(const T *h, const T *emb, int R, int H, T *xfc, cudaStream_t s) {
    if (R <= 0) return;
    launch_pdl(concat_next_kernel<T>, R, 256, 0, s, h, emb, H, xfc); note_launch();
}

template <typename T>
void launch_prefill_finish(const int *argmax1, const T *h_last, int b, int L, int D1, int H,
                           int *seq_len, int *n_pend, int *root, int *pend_next, T *pend_h,
                           int *root_out, cudaStream_t s) {
    launch_pdl(prefill_finish_kernel<T>, 1, 256, 0, s, argmax1, h_last, b, L, D1, H, seq_len, n_pend,
                                               root, pend_next, pend_h, root_out); note_launch();
}

#define MSD_INST(T)                                                                             \
    template void launch_catchup_setup<T>(const int *, const int *, const T *, const int *,     \
                                          const T *, int, int, int, int, T *, RowDesc *, int *, \
                                          cudaStream_t);                                        \
    template void launch_root_gather<T>(const float *, const int *, int, int, int, float *, T *, \
                                        cudaStream_t);                                          \
    template void launch_hhat_store<T>(const float *, const RowDesc *, int, int, int, float *,  \
                                       T *, cudaStream_t);                                      \
    template void launch_tree_init<T>(const DraftArgs<T> &, int, cudaStream_t);                 \
    template void launch_tree_step<T>(const DraftArgs<T> &, int, int, cudaStream_t);            \
    template void launch_pend_h<T>(const T *, const int *, const int *, int, int, int, int, T *, \
                                   cudaStream_t);                                               \
    template void launch_select_visual<T>(float *, const T *, const int *, int, int,            \
                                          cudaStream_t);                                        \
    template void launch_concat_next<T>(const T *, const T *, int, int, T *, cudaStream_t);     \
    template void launch_prefill_finish<T>(const int *, const T *, int, int, int, int, int *,   \
                                           int *, int *, int *, T *, int *, cudaStream_t);
MSD_INST(float)
MSD_INST(bf16)
#undef MSD_INST

}  // namespace msd
