// Launchers of the integer-side kernels (tree building, acceptance,
// compaction) and the draft/verify row set-up.
#pragma once

#include "kernels.h"

namespace msd {

constexpr int TREE_MAXK = 16;   // top-k limit (also the top-k kernel's limit)
constexpr int TREE_MAXD = 64;   // depth limit

// Draft-tree builder state and outputs of one draft pass (device pointers).
template <typename T>
struct DraftArgs {
    const int *ids;             // top-k ids of the pass rows [rows][k]
    const float *logp;          // their log-probabilities
    int k, D, C, H, V, Td, Wd, B;  // C = k + (D-1)k^2 candidates, Td = (D-1)k slots
    int *cand_tok, *cand_par, *cand_depth;   // [B][C]
    float *cand_score;                       // [B][C]
    int *frontier;                           // [2][B][k] candidate ids, best first (by pass parity)
    const float *hhat_root;                  // [B][H]
    const float *hhat_slot;                  // [B][Td][H]
    const T *E;
    const int *seq_len;
    T *xfc;                     // next pass input rows [B*k][2H] (split: lo plane at +lo)
    long lo;
    RowDesc *rows;              // next pass row descriptors [B*k]
    uint64_t *slot_mask;        // [B][Td][Wd]
    uint64_t *row_mask;         // [B*k][Wd]
};

struct TreeOut {
    int *tokens, *parent, *depth;
    uint64_t *mask;
    int *n_nodes;
};

struct TreeIn {
    const int *tokens, *parent, *depth;
    const uint64_t *mask;
    const int *n_nodes;
};

// `lo`: the lo-plane offset of the split bf16 buffers (0 for fp32 contexts).
template <typename T>
void launch_catchup_setup(const int *seq_len, const int *n_pend, const T *pend_h,
                          const int *pend_next, const T *E, int B, int H, int D1, int V, T *xfc,
                          long lo, RowDesc *rows, int *status, cudaStream_t s);
template <typename T>
void launch_root_gather(const float *x, const int *n_pend, int B, int D1, int H, float *hhat_root,
                        T *xr, long lo, cudaStream_t s);
template <typename T>
void launch_hhat_store(const float *x, const RowDesc *rows, int R, int Td, int H,
                       float *hhat_slot, T *xb, long lo, cudaStream_t s);
template <typename T>
void launch_tree_init(const DraftArgs<T> &a, int B, cudaStream_t s);
template <typename T>
void launch_tree_step(const DraftArgs<T> &a, int B, int d, cudaStream_t s);
void launch_tree_finalize(const TreeOut &t, const int *cand_tok, const int *cand_par,
                          const int *cand_depth, const float *cand_score, int *node_of,
                          const int *root, int B, int C, int N, int *status, cudaStream_t s);
void launch_verify_setup(const TreeIn &t, const int *seq_len, const int *root, int B, int N,
                         int V, RowDesc *rows, int *src, uint64_t *vmask, int *status,
                         cudaStream_t s);
// Depths and ancestor-or-self masks of caller-planted trees from their parent
// arrays, for requests b0 .. b0+nb-1 (n_nodes[b] nodes of request b; nodes
// past it get depth 0 and an empty mask). A parent that does not precede its
// node sets ST_BAD_TREE.
void launch_tree_complete(const int *parent, int *depth, uint64_t *mask, const int *n_nodes, int b0, int nb,
                          int N, int *status, cudaStream_t s);
// A tree of each request's root alone (plain greedy decoding): node 0 = root,
// parent -1, depth 0, mask = itself, n_nodes = 1; nodes 1.. are not part of it.
void launch_root_tree(const int *root, int B, int N, int W, int *tokens, int *parent, int *depth,
                      uint64_t *mask, int *n_nodes, cudaStream_t s);

void launch_accept(const TreeIn &t, const int *argmax, int B, int N, int D, int *seq_len,
                   int *n_pend, int *root, int *pend_next, int *acc_path, int *acc_L0, int *acc_a,
                   int *path_out, int *accept_len_out, int *bonus_out, int *index_map_out,
                   cudaStream_t s);
// Speculative sampling over the tree at temperature T > 0 (Eq. 6 with the
// draft's top-k candidates as point-mass proposals): logits [B][N][V] fp32 of
// the verify pass, inv_temp = 1/T, u [B][D+1][k+1] uniforms in [0, 1);
// row_max [B*N] and row_sum [B*N] are scratch for the per-row statistics.
// Same outputs and state update as launch_accept. Two launches. Returns
// false (and launches nothing more) if V > SAMPLE_MAX_VOCAB or a launch
// failed, so that the caller does not compact on stale acceptance outputs.
constexpr int SAMPLE_MAX_VOCAB = 48 * 1024 * 8;   // one bit per token in 48 KB of shared memory
bool launch_accept_sample(const TreeIn &t, const float *logits, int B, int N, int D, int k, int V,
                          float inv_temp, const float *u, float *row_max, double *row_sum, int *seq_len,
                          int *n_pend, int *root, int *pend_next, int *acc_path, int *acc_L0, int *acc_a,
                          int *path_out, int *accept_len_out, int *bonus_out, int *index_map_out,
                          int *status, cudaStream_t s);
// KV compaction; lo_bytes (0: none) = the lo planes' byte offset from their hi planes.
void launch_compact_kv(const void *tree_kv, void *cache, const int *acc_path, const int *acc_L0,
                       const int *acc_a, int n_layers, int B, int nh, int N, int S, int D1,
                       int row_bytes, long lo_bytes, int *status, cudaStream_t s);
template <typename T>
void launch_pend_h(const T *hT, const int *acc_path, const int *acc_a, int B, int N, int D1,
                   int H, T *pend_h, long lo, cudaStream_t s);
// slo: lo plane of emb (0: emb is exact, e.g. the embedding rows)
template <typename T>
void launch_select_visual(float *x, const T *emb, long slo, const int *src, int R, int H, cudaStream_t s);
template <typename T>
void launch_concat_next(const T *h, const T *emb, int R, int H, T *xfc, long lo, cudaStream_t s);
template <typename T>
void launch_prefill_finish(const int *argmax1, const T *h_last, int b, int L, int D1, int H,
                           int *seq_len, int *n_pend, int *root, int *pend_next, T *pend_h, long lo,
                           int *root_out, cudaStream_t s);

}  // namespace msd
