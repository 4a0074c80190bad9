// Step engine and C ABI of the MSD hot path (include/msd.h).
//
// Orchestrates the kernels of one decode step on one stream:
//   msd_draft_tree     catch-up pass + D-1 tree passes of the one-layer draft
//                      model (Sec. 3.2, Eq. 4-5) with the decoupled input (Eq. 7)
//   msd_verify         one tree-masked target forward (Sec. 3.2, verification)
//   msd_accept_compact greedy acceptance (Eq. 6 at T = 0) + KV compaction
//   msd_accept_sample  speculative sampling over the tree (Eq. 6, T > 0) + KV
//                      compaction
// Every size a kernel needs at run time (L, accepted length, pending rows) is
// read by the kernels from device state, so a step needs no host round trip.
#include <cmath>
#include <cstdio>
#include <algorithm>
#include <cstring>
#include <string>
#include <type_traits>
#include <vector>

#include "msd.h"
#include "kernels.h"
#include "kernels_tree.h"
#include "gemm_tc.h"
#include "attn_tc.h"

using namespace msd;

struct msd_ctx {
    msd_config cfg;
    msd_weights w;
    std::vector<msd_layer> layers;
    int dev = 0;
    size_t esz = 0;
    int B, S, N, D, D1, k, H, F, V, nh, hd, NL, W, C, Td, Wd, Rmax, chunk, Rlog;

    void *target_kv = nullptr, *draft_kv = nullptr, *tree_kv = nullptr, *dtree_kv = nullptr;
    int *seq_len = nullptr, *n_pend = nullptr, *root = nullptr, *pend_next = nullptr;
    void *pend_h = nullptr;
    float *x = nullptr, *qkv = nullptr, *gu = nullptr, *logits = nullptr;
    float *ss_part = nullptr;   // folded RMSNorm: per-tile sums of squares [Rmax][ss_ld]
    int ss_ld = 0;
    void *xn = nullptr, *q = nullptr, *attn = nullptr, *act = nullptr, *xfc = nullptr, *xr = nullptr;
    int *argmax_tmp = nullptr;
    RowDesc *rows = nullptr;
    int *src = nullptr;
    uint64_t *vmask = nullptr;
    int *cand_tok = nullptr, *cand_par = nullptr, *cand_depth = nullptr, *frontier = nullptr,
        *node_of = nullptr;
    float *cand_score = nullptr, *hhat_root = nullptr, *hhat_slot = nullptr;
    uint64_t *slot_mask = nullptr, *row_mask = nullptr;
    int *topk_ids = nullptr;
    float *topk_logp = nullptr;
    TopkScratch tks{nullptr, nullptr};
    void *hT = nullptr;
    int *acc_path = nullptr, *acc_L0 = nullptr, *acc_a = nullptr;
    float *samp_max = nullptr;      // sampling (T > 0): per verify row max logit and
    double *samp_sum = nullptr;     // sum of exp((z - max) / T)
    // plain greedy decoding (msd_ar_step): a root-only tree and its argmax
    msd_tree ar_tree{};
    int *ar_argmax = nullptr;
    bool draft_stale = false;   // msd_ar_step ran: the draft cache no longer follows the target's
    float2 *rope_tab = nullptr;
    void *h_all = nullptr, *emb_all = nullptr;
    // bf16 contexts: every bf16 buffer that feeds a tensor-core product (and the
    // KV caches) is carved from one arena whose upper half holds the lo planes
    // of the split pairs; lo = that half's size in elements (0: fp32 context)
    long lo = 0;
    int *status = nullptr;
    int *status_host = nullptr;
    cudaEvent_t status_ev = nullptr;
    bool status_pending = false;
    GemmPlan *gplan = nullptr;
    AttnTcPlan *aplan = nullptr;
    // pre-packed GEMM weights (bf16 contexts)
    struct LayerPack {
        const void *qkv = nullptr, *o = nullptr, *gu = nullptr, *down = nullptr;
    };
    std::vector<LayerPack> lpack;
    LayerPack dpack;
    const void *pk_lm = nullptr, *pk_fc = nullptr;
    void *pk_scratch = nullptr;     // msd_linear: its weight, packed per call
    size_t pk_scratch_bytes = 0;
    std::vector<void *> allocs;
    std::vector<long> L_bound;
    bool prefilled = false;
    std::string err;
    // whole-step CUDA graphs (msd_step), one per buffer set
    struct StepGraph {
        cudaGraphExec_t exec = nullptr;
        int kind = 0;               // 0: draft-verify-accept step, 1: plain greedy step,
                                    // 2: draft-verify-sample step
        msd_tree tree{};
        const void *argmax = nullptr, *path = nullptr, *alen = nullptr, *bonus = nullptr;
        const void *u = nullptr;    // kind 2: the uniforms' buffer and the temperature
        float temp = 0.f;
        long kernels = 0;
        long uses = 0;
        bool stamped = false;       // recorded with GEMM launch stamps (profile mode 2)
    };
    std::vector<StepGraph> graphs;
    cudaStream_t cap_stream = nullptr;
    bool capturing = false;
    long captured_launches = 0; // launches recorded into graphs (not executed then)
    long graph_kernels = 0;     // kernels executed by graph replays
};

namespace {

msd_status fail(msd_ctx *c, msd_status st, const std::string &msg) {
    if (c) c->err = msg;
    return st;
}

#define CU(call)                                                                          \
    do {                                                                                  \
        cudaError_t e_ = (call);                                                          \
        if (e_ != cudaSuccess)                                                            \
            return fail(c, MSD_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
    } while (0)

template <typename P>
bool dalloc(msd_ctx *c, P **p, size_t bytes) {
    void *v = nullptr;
    if (bytes == 0) bytes = 16;
    if (cudaMalloc(&v, bytes) != cudaSuccess) return false;
    cudaMemset(v, 0, bytes);
    c->allocs.push_back(v);
    *p = static_cast<P *>(v);
    return true;
}

// A runtime error left pending by code outside this call (or by an earlier
// teardown) is reported on stderr and cleared, so that a call's status reflects
// only its own launches.
bool report_stale_error(const char *where) {
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        fprintf(stderr, "msd: %s: found a pending CUDA error: %s\n", where, cudaGetErrorString(e));
    return e != cudaSuccess;
}

// The device status word of earlier calls, observed without blocking.
msd_status check_status(msd_ctx *c) {
    if (c->status_pending && cudaEventQuery(c->status_ev) == cudaSuccess) {
        c->status_pending = false;
        if (*c->status_host != 0) {
            char buf[96];
            snprintf(buf, sizeof buf, "device status word set (code %d)", *c->status_host);
            return fail(c, MSD_ERR_DEVICE, buf);
        }
    }
    return MSD_OK;
}

msd_status post_status(msd_ctx *c, cudaStream_t s) {
    CU(cudaGetLastError());
    if (c->capturing) return MSD_OK;    // the step's entry point posts after the replay
    CU(cudaMemcpyAsync(c->status_host, c->status, sizeof(int), cudaMemcpyDeviceToHost, s));
    CU(cudaEventRecord(c->status_ev, s));
    c->status_pending = true;
    return MSD_OK;
}

size_t kv_layer_elems(const msd_ctx *c, int slots) {
    return (size_t)c->B * c->nh * slots * c->hd;
}

template <typename T>
T *tkv(const msd_ctx *c, void *base, int layer, int kv, int slots) {
    return static_cast<T *>(base) + ((size_t)layer * 2 + kv) * kv_layer_elems(c, slots);
}

// Y (=|+=) X W^T on the dtype's GEMM: tcgen05 tensor cores for bf16, the
// CUDA-core kernel for fp32.
// X is a context buffer (its lo plane, if any, sits c->lo elements on) unless
// `own` is false (a caller-owned operand: hi values only).
template <typename T>
void gemm(msd_ctx *c, const T *X, int ldx, int M, int K, const GemmW &W, int O, float *Y,
          int ldy, int epi, cudaStream_t s, bool own = true);

template <>
void gemm<float>(msd_ctx *c, const float *X, int ldx, int M, int K, const GemmW &W, int O,
                 float *Y, int ldy, int epi, cudaStream_t s, bool) {
    launch_gemm_simt<float>(X, ldx, M, K, W, O, Y, ldy, epi, s);
}

template <>
void gemm<bf16>(msd_ctx *c, const bf16 *X, int ldx, int M, int K, const GemmW &W, int O,
                float *Y, int ldy, int epi, cudaStream_t s, bool own) {
    gemm_bf16(c->gplan, X, own && c->lo ? X + c->lo : nullptr, ldx, M, K, W, O, Y, ldy, epi, c->status, s);
}

// The lo plane of a context buffer (null for fp32 contexts).
const bf16 *lo_of(const msd_ctx *c, const void *hi) {
    return c->lo ? static_cast<const bf16 *>(hi) + c->lo : nullptr;
}

// One pre-norm decoder layer over R rows (target or draft).
template <typename T>
void attention(msd_ctx *c, const AttnArgs<T> &a, int rows_per_req, cudaStream_t s);

template <>
void attention<float>(msd_ctx *c, const AttnArgs<float> &a, int, cudaStream_t s) {
    launch_attention<float>(a, s);
}

template <>
void attention<bf16>(msd_ctx *c, const AttnArgs<bf16> &a, int rows_per_req, cudaStream_t s) {
    // one block per request: launch the longest requests' CTAs first (the host's
    // bound of each request's L orders them; only scheduling depends on it)
    int order[64];
    const int *ord = nullptr;
    if (a.R == c->B * rows_per_req && c->B > 1 && c->B <= 64) {
        for (int b = 0; b < c->B; ++b) order[b] = b;
        std::stable_sort(order, order + c->B, [&](int x, int y) { return c->L_bound[x] > c->L_bound[y]; });
        ord = order;
    }
    unsigned long long *st = gemm_stamp_external(c->gplan, 1, a.R, a.nh, a.hd);
    if (!launch_attention_tc(c->aplan, a, c->B, rows_per_req, ord, c->status, s, st)) {
        c->err = "tensor-core attention: unsupported shape or launch failure";
        launch_flag(c->status, ST_RANGE, s);     // reported by the next call
    }
}

// qkv = xn [wq;wk;wv]^T, then RoPE on q and k (Sec. 3.1 backbone), q to c->q
// and k, v to kdst/vdst at each row's slot. Decode shapes run it as one GEMM
// with the rotation and placement in its epilogue.
template <typename T>
void qkv_rope(msd_ctx *c, const msd_layer &lw, const msd_ctx::LayerPack &lp, int R,
              const RowDesc *rows, T *kdst, T *vdst, int dst_slots, cudaStream_t s,
              const GemmNorm *norm_in = nullptr) {
    const int H = c->H;
    GemmW wqkv = {{lw.wq, lw.wk, lw.wv}, {H, H, H}, 3, lp.qkv};
    if constexpr (std::is_same<T, bf16>::value) {
        GemmFused fx;
        memset(&fx, 0, sizeof fx);
        fx.epi = EPI_ROPE_KV;
        fx.rows = rows;
        fx.rope_tab = c->rope_tab;
        fx.max_pos = c->S;
        fx.q_out = static_cast<bf16 *>(c->q);
        fx.kdst = kdst;
        fx.vdst = vdst;
        fx.slots = dst_slots;
        fx.nh = c->nh;
        fx.hd = c->hd;
        fx.lo = c->lo;
        if (gemm_bf16_fused(c->gplan, static_cast<const bf16 *>(c->xn), lo_of(c, c->xn), H, R, H, wqkv, 3 * H,
                            fx, c->status, s, norm_in))
            return;
    }
    gemm<T>(c, static_cast<const T *>(c->xn), H, R, H, wqkv, 3 * H, c->qkv, 3 * H, EPI_STORE, s);
    launch_rope_kv<T>(c->qkv, rows, R, c->nh, c->hd, c->rope_tab, c->S, static_cast<T *>(c->q),
                      kdst, vdst, dst_slots, c->lo, c->status, s);
}

// act = silu(xn wg^T) * (xn wu^T). bf16 contexts hold gate/up glu-packed; the
// decode shapes apply the SwiGLU in the GEMM's epilogue.
template <typename T>
void gate_up_swiglu(msd_ctx *c, const msd_layer &lw, const msd_ctx::LayerPack &lp, int R,
                    cudaStream_t s, const GemmNorm *norm_in = nullptr) {
    const int H = c->H, F = c->F;
    if constexpr (std::is_same<T, bf16>::value) {
        const int O = glu_rows(F);
        GemmW wgu = {{nullptr, nullptr, nullptr}, {O, 0, 0}, 1, lp.gu};
        GemmFused fx;
        memset(&fx, 0, sizeof fx);
        fx.epi = EPI_SWIGLU;
        fx.act = static_cast<bf16 *>(c->act);
        fx.F = F;
        fx.lo = c->lo;
        if (gemm_bf16_fused(c->gplan, static_cast<const bf16 *>(c->xn), lo_of(c, c->xn), H, R, H, wgu, O, fx,
                            c->status, s, norm_in))
            return;
        gemm<T>(c, static_cast<const T *>(c->xn), H, R, H, wgu, O, c->gu, O, EPI_STORE, s);
        launch_swiglu<T>(c->gu, R, F, true, static_cast<T *>(c->act), c->lo, s);
    } else {
        GemmW wgu = {{lw.w_gate, lw.w_up, nullptr}, {F, F, 0}, 2, nullptr};
        gemm<T>(c, static_cast<const T *>(c->xn), H, R, H, wgu, 2 * F, c->gu, 2 * F, EPI_STORE, s);
        launch_swiglu<T>(c->gu, R, F, false, static_cast<T *>(c->act), c->lo, s);
    }
}

// Folded RMSNorm (bf16 decode shapes with packed weights): the GEMM that
// writes the residual stream also writes bf16(x * g) into c->xn and per-tile
// sums of squares into c->ss_part; the next projection scales its rows by
// 1/rms in its epilogue. Elsewhere the RMSNorm kernel runs.
bool folds(const msd_ctx *c, int R, const void *packed) {
    return c->esz == 2 && R <= 128 && packed != nullptr;
}

GemmNorm norm_out(msd_ctx *c, const void *g) {
    return GemmNorm{c->ss_part, c->ss_ld, static_cast<bf16 *>(c->xn), static_cast<const bf16 *>(g),
                    0, c->H, c->cfg.rms_eps, c->lo};
}

GemmNorm norm_in(msd_ctx *c) {
    return GemmNorm{c->ss_part, c->ss_ld, nullptr, nullptr, c->ss_ld, c->H, c->cfg.rms_eps, c->lo};
}

// One pre-norm decoder layer over R rows (target or draft). Rows come in
// blocks of rows_per_req per request.
// cache positions. in_folded: the layer's input norm was folded into the GEMM
// that produced x; out_norm_g (nullable): the next layer's input-norm gain,
// to fold into this layer's last GEMM. Returns whether it did.
template <typename T>
bool run_layer(msd_ctx *c, const msd_layer &lw, const msd_ctx::LayerPack &lp, int R,
               const RowDesc *rows, T *kdst, T *vdst, int dst_slots, const T *ck, const T *cv,
               int cslots, const T *tk, const T *tv, int tslots, const uint64_t *mask, int mw,
               int rows_per_req, cudaStream_t s, bool in_folded = false,
               const void *out_norm_g = nullptr) {
    const int H = c->H, F = c->F;
    const float eps = c->cfg.rms_eps;
    const bool fold = folds(c, R, lp.o) && lp.qkv && lp.gu && lp.down;
    const GemmNorm nin = norm_in(c);
    if (!(fold && in_folded))
        launch_rmsnorm<T>(c->x, static_cast<const T *>(lw.attn_norm), R, H, eps,
                          static_cast<T *>(c->xn), c->lo, s);
    qkv_rope<T>(c, lw, lp, R, rows, kdst, vdst, dst_slots, s, fold && in_folded ? &nin : nullptr);
    AttnArgs<T> a;
    a.q = static_cast<const T *>(c->q);
    a.rows = rows;
    a.R = R;
    a.cache_k = ck;
    a.cache_v = cv;
    a.cache_slots = cslots;
    a.tree_k = tk;
    a.tree_v = tv;
    a.tree_slots = tslots;
    a.mask = mask;
    a.mask_words = mw;
    a.nh = c->nh;
    a.hd = c->hd;
    a.scale = 1.0f / sqrtf((float)c->hd);
    a.out = static_cast<T *>(c->attn);
    a.cache_fresh = kdst == ck;         // this layer's own K/V go into the cache it reads
    a.lo = c->lo;
    attention<T>(c, a, rows_per_req, s);
    GemmW wo = {{lw.wo, nullptr, nullptr}, {H, 0, 0}, 1, lp.o};
    GemmW wd = {{lw.w_down, nullptr, nullptr}, {H, 0, 0}, 1, lp.down};
    if constexpr (std::is_same<T, bf16>::value) {
        if (fold) {
            const GemmNorm no = norm_out(c, lw.mlp_norm);
            gemm_bf16(c->gplan, static_cast<const bf16 *>(c->attn), lo_of(c, c->attn), H, R, H, wo, H, c->x, H,
                      EPI_ADD, c->status, s, &no);
            gate_up_swiglu<T>(c, lw, lp, R, s, &nin);
            if (out_norm_g) {
                const GemmNorm nd = norm_out(c, out_norm_g);
                gemm_bf16(c->gplan, static_cast<const bf16 *>(c->act), lo_of(c, c->act), F, R, F, wd, H, c->x, H,
                          EPI_ADD, c->status, s, &nd);
                return true;
            }
            gemm<T>(c, static_cast<const T *>(c->act), F, R, F, wd, H, c->x, H, EPI_ADD, s);
            return false;
        }
    }
    gemm<T>(c, static_cast<const T *>(c->attn), H, R, H, wo, H, c->x, H, EPI_ADD, s);
    launch_rmsnorm<T>(c->x, static_cast<const T *>(lw.mlp_norm), R, H, eps,
                      static_cast<T *>(c->xn), c->lo, s);
    gate_up_swiglu<T>(c, lw, lp, R, s);
    gemm<T>(c, static_cast<const T *>(c->act), F, R, F, wd, H, c->x, H, EPI_ADD, s);
    return false;
}

GemmW one(const void *w, int rows, const void *packed = nullptr) {
    return GemmW{{w, nullptr, nullptr}, {rows, 0, 0}, 1, packed};
}

// x = f_down(xfc) for R draft rows; with a folded norm also the draft layer's
// input norm. Returns whether it folded.
template <typename T>
bool draft_fc(msd_ctx *c, int R, cudaStream_t s) {
    const int H = c->H;
    const GemmW W = one(c->w.draft_fc, H, c->pk_fc);
    if constexpr (std::is_same<T, bf16>::value) {
        if (folds(c, R, c->pk_fc) && c->dpack.o) {
            const GemmNorm no = norm_out(c, c->w.draft.attn_norm);
            return gemm_bf16(c->gplan, static_cast<const bf16 *>(c->xfc), lo_of(c, c->xfc), 2 * H, R, 2 * H, W,
                             H, c->x, H, EPI_STORE, c->status, s, &no);
        }
    }
    gemm<T>(c, static_cast<const T *>(c->xfc), 2 * H, R, 2 * H, W, H, c->x, H, EPI_STORE, s);
    return false;
}

// ---------------------------------------------------------------------------
// Prefill
// ---------------------------------------------------------------------------
template <typename T>
msd_status prefill_impl(msd_ctx *c, int batch, const int32_t *seq_len_host, const int32_t *ids_dev,
                        int ids_stride, const void *vis_dev, const int64_t *vis_off_host,
                        int32_t *root_out, cudaStream_t s) {
    const int H = c->H, V = c->V, D1 = c->D1;
    const T *E = static_cast<const T *>(c->w.embed);
    const T *vis = static_cast<const T *>(vis_dev);
    CU(cudaMemsetAsync(c->seq_len, 0, sizeof(int) * c->B, s));
    CU(cudaMemsetAsync(c->n_pend, 0, sizeof(int) * c->B, s));
    for (int b = 0; b < c->B; ++b) c->L_bound[b] = 0;
    std::vector<int> ids, src;
    std::vector<RowDesc> rd;
    for (int b = 0; b < batch; ++b) {
        const int L = seq_len_host[b];
        ids.resize(L);
        CU(cudaMemcpy(ids.data(), ids_dev + (size_t)b * ids_stride, sizeof(int) * L,
                      cudaMemcpyDeviceToHost));
        if (ids[L - 1] < 0) return fail(c, MSD_ERR_INVALID, "a prompt must end with a text token");
        src.resize(L);
        long vrow = vis_off_host ? vis_off_host[b] : 0;
        int n_vis = 0;
        for (int i = 0; i < L; ++i) {
            if (ids[i] >= V || ids[i] < -1) return fail(c, MSD_ERR_INVALID, "token id out of range");
            if (ids[i] >= 0) src[i] = ids[i];
            else { src[i] = (int)(-1 - (vrow + n_vis)); ++n_vis; }
        }
        if (n_vis > 0 && !vis) return fail(c, MSD_ERR_INVALID, "visual slots but no visual rows");
        CU(cudaMemcpyAsync(c->src, src.data(), sizeof(int) * L, cudaMemcpyHostToDevice, s));
        // target over the prompt, causal, in chunks
        for (int r0 = 0; r0 < L; r0 += c->chunk) {
            const int n = std::min(c->chunk, L - r0);
            rd.resize(n);
            for (int i = 0; i < n; ++i) rd[i] = RowDesc{b, r0 + i, r0 + i + 1, r0 + i};
            CU(cudaMemcpyAsync(c->rows, rd.data(), sizeof(RowDesc) * n, cudaMemcpyHostToDevice, s));
            launch_embed_rows<T>(E, vis, c->src + r0, n, H, c->x,
                                 static_cast<T *>(c->emb_all) + (size_t)r0 * H, V, c->status, s);
            for (int l = 0; l < c->NL; ++l) {
                T *K = tkv<T>(c, c->target_kv, l, 0, c->S), *Vv = tkv<T>(c, c->target_kv, l, 1, c->S);
                run_layer<T>(c, c->layers[l], c->lpack[l], n, c->rows, K, Vv, c->S, K, Vv, c->S, nullptr,
                             nullptr, 0, nullptr, 0, n, s);
            }
            launch_rmsnorm<T>(c->x, static_cast<const T *>(c->w.final_norm), n, H, c->cfg.rms_eps,
                              static_cast<T *>(c->h_all) + (size_t)r0 * H, c->lo, s);
            CU(cudaStreamSynchronize(s));   // rd/src host vectors are reused
        }
        const T *h_last = static_cast<const T *>(c->h_all) + (size_t)(L - 1) * H;
        gemm<T>(c, h_last, H, 1, H, one(c->w.lm_head, V, c->pk_lm), V, c->logits, V, EPI_STORE, s);
        launch_argmax(c->logits, 1, V, c->argmax_tmp, c->tks, s);
        // draft cache over positions 0 .. L-2 with the decoupled input (Eq. 7): text
        // rows f_down(Concat(h, e_next)); visual rows e (MSD), the same
        // concatenation (Baseline) or h (Visual Feature), Sec. 5.3
        for (int r0 = 0; r0 < L - 1; r0 += c->chunk) {
            const int n = std::min(c->chunk, L - 1 - r0);
            rd.resize(n);
            for (int i = 0; i < n; ++i) rd[i] = RowDesc{b, r0 + i, r0 + i + 1, r0 + i};
            CU(cudaMemcpyAsync(c->rows, rd.data(), sizeof(RowDesc) * n, cudaMemcpyHostToDevice, s));
            launch_concat_next<T>(static_cast<const T *>(c->h_all) + (size_t)r0 * H,
                                  static_cast<const T *>(c->emb_all) + (size_t)r0 * H, n, H,
                                  static_cast<T *>(c->xfc), c->lo, s);
            gemm<T>(c, static_cast<const T *>(c->xfc), 2 * H, n, 2 * H, one(c->w.draft_fc, H, c->pk_fc), H,
                    c->x, H, EPI_STORE, s);
            if (c->cfg.draft_input != MSD_DRAFT_CONCAT) {
                const bool feat = c->cfg.draft_input == MSD_DRAFT_FEATURE;
                const void *vis_rows = feat ? c->h_all : c->emb_all;
                launch_select_visual<T>(c->x, static_cast<const T *>(vis_rows) + (size_t)r0 * H, feat ? c->lo : 0,
                                        c->src + r0, n, H, s);
            }
            T *K = tkv<T>(c, c->draft_kv, 0, 0, c->S), *Vv = tkv<T>(c, c->draft_kv, 0, 1, c->S);
            run_layer<T>(c, c->w.draft, c->dpack, n, c->rows, K, Vv, c->S, K, Vv, c->S, nullptr, nullptr, 0,
                         nullptr, 0, n, s);
            CU(cudaStreamSynchronize(s));
        }
        launch_prefill_finish<T>(c->argmax_tmp, h_last, b, L, D1, H, c->seq_len, c->n_pend, c->root,
                                 c->pend_next, static_cast<T *>(c->pend_h), c->lo, root_out, s);
        c->L_bound[b] = L;
    }
    c->prefilled = true;
    c->draft_stale = false;
    return post_status(c, s);
}

// ---------------------------------------------------------------------------
// Draft tree
// ---------------------------------------------------------------------------
template <typename T>
DraftArgs<T> draft_args(msd_ctx *c) {
    DraftArgs<T> a;
    a.ids = c->topk_ids;
    a.logp = c->topk_logp;
    a.k = c->k; a.D = c->D; a.C = c->C; a.H = c->H; a.V = c->V; a.Td = c->Td; a.Wd = c->Wd;
    a.B = c->B;
    a.cand_tok = c->cand_tok; a.cand_par = c->cand_par; a.cand_depth = c->cand_depth;
    a.cand_score = c->cand_score; a.frontier = c->frontier;
    a.hhat_root = c->hhat_root; a.hhat_slot = c->hhat_slot;
    a.E = static_cast<const T *>(c->w.embed);
    a.seq_len = c->seq_len;
    a.xfc = static_cast<T *>(c->xfc);
    a.lo = c->lo;
    a.rows = c->rows;
    a.slot_mask = c->slot_mask;
    a.row_mask = c->row_mask;
    return a;
}

msd_status record_pass(msd_ctx *c, const msd_draft_record *rec, int pass, int rows_per_req,
                       cudaStream_t s) {
    if (!rec) return MSD_OK;
    const int B = c->B, D = c->D, k = c->k, V = c->V;
    if (rec->logits)
        CU(cudaMemcpy2DAsync(rec->logits + (size_t)pass * k * V, sizeof(float) * D * k * V,
                             c->logits, sizeof(float) * rows_per_req * V,
                             sizeof(float) * rows_per_req * V, B, cudaMemcpyDeviceToDevice, s));
    if (rec->topk_ids)
        CU(cudaMemcpy2DAsync(rec->topk_ids + (size_t)pass * k * k, sizeof(int) * D * k * k,
                             c->topk_ids, sizeof(int) * rows_per_req * k,
                             sizeof(int) * rows_per_req * k, B, cudaMemcpyDeviceToDevice, s));
    if (rec->topk_logp)
        CU(cudaMemcpy2DAsync(rec->topk_logp + (size_t)pass * k * k, sizeof(float) * D * k * k,
                             c->topk_logp, sizeof(float) * rows_per_req * k,
                             sizeof(float) * rows_per_req * k, B, cudaMemcpyDeviceToDevice, s));
    return MSD_OK;
}

template <typename T>
msd_status draft_impl(msd_ctx *c, const msd_tree *out, const msd_draft_record *rec,
                      cudaStream_t s) {
    const int B = c->B, H = c->H, V = c->V, k = c->k, D1 = c->D1, S = c->S;
    const T *E = static_cast<const T *>(c->w.embed);
    T *dK = tkv<T>(c, c->draft_kv, 0, 0, S), *dV = tkv<T>(c, c->draft_kv, 0, 1, S);
    T *tK = tkv<T>(c, c->dtree_kv, 0, 0, c->Td), *tV = tkv<T>(c, c->dtree_kv, 0, 1, c->Td);
    // pass 1: catch-up rows + root slot
    const int R1 = B * D1;
    launch_catchup_setup<T>(c->seq_len, c->n_pend, static_cast<const T *>(c->pend_h), c->pend_next,
                            E, B, H, D1, V, static_cast<T *>(c->xfc), c->lo, c->rows, c->status, s);
    bool folded = draft_fc<T>(c, R1, s);
    run_layer<T>(c, c->w.draft, c->dpack, R1, c->rows, dK, dV, S, dK, dV, S, nullptr, nullptr, 0, nullptr, 0,
                 D1, s, folded);
    launch_root_gather<T>(c->x, c->n_pend, B, D1, H, c->hhat_root, static_cast<T *>(c->xr), c->lo, s);
    gemm<T>(c, static_cast<const T *>(c->xr), H, B, H, one(c->w.lm_head, V, c->pk_lm), V, c->logits, V,
            EPI_STORE, s);
    launch_topk_logp(c->logits, B, V, k, c->topk_ids, c->topk_logp, c->tks, s);
    msd_status st = record_pass(c, rec, 0, 1, s);
    if (st != MSD_OK) return st;
    DraftArgs<T> a = draft_args<T>(c);
    launch_tree_init<T>(a, B, s);
    // passes 2..D: expand the frontier
    const int Rk = B * k;
    for (int d = 2; d <= c->D; ++d) {
        folded = draft_fc<T>(c, Rk, s);
        run_layer<T>(c, c->w.draft, c->dpack, Rk, c->rows, tK, tV, c->Td, dK, dV, S, tK, tV, c->Td,
                     c->row_mask, c->Wd, k, s, folded);
        launch_hhat_store<T>(c->x, c->rows, Rk, c->Td, H, c->hhat_slot, static_cast<T *>(c->xr), c->lo, s);
        gemm<T>(c, static_cast<const T *>(c->xr), H, Rk, H, one(c->w.lm_head, V, c->pk_lm), V, c->logits, V,
                EPI_STORE, s);
        launch_topk_logp(c->logits, Rk, V, k, c->topk_ids, c->topk_logp, c->tks, s);
        st = record_pass(c, rec, d - 1, k, s);
        if (st != MSD_OK) return st;
        launch_tree_step<T>(a, B, d, s);
    }
    TreeOut t{out->tokens, out->parent, out->depth, out->mask, out->n_nodes};
    launch_tree_finalize(t, c->cand_tok, c->cand_par, c->cand_depth, c->cand_score, c->node_of,
                         c->root, B, c->C, c->N, c->status, s);
    return post_status(c, s);
}

// ---------------------------------------------------------------------------
// Verify
// ---------------------------------------------------------------------------
template <typename T>
msd_status verify_impl(msd_ctx *c, const msd_tree *tree, int32_t *argmax_dev, float *logits_dev,
                       cudaStream_t s) {
    const int B = c->B, N = c->N, H = c->H, V = c->V, R = B * N;
    TreeIn t{tree->tokens, tree->parent, tree->depth, tree->mask, tree->n_nodes};
    launch_verify_setup(t, c->seq_len, c->root, B, N, V, c->rows, c->src, c->vmask, c->status, s);
    launch_embed_rows<T>(static_cast<const T *>(c->w.embed), nullptr, c->src, R, H, c->x, nullptr,
                         V, c->status, s);
    bool folded = false;
    for (int l = 0; l < c->NL; ++l) {
        T *K = tkv<T>(c, c->target_kv, l, 0, c->S), *Vv = tkv<T>(c, c->target_kv, l, 1, c->S);
        T *tK = tkv<T>(c, c->tree_kv, l, 0, N), *tV = tkv<T>(c, c->tree_kv, l, 1, N);
        const void *next_g = l + 1 < c->NL ? c->layers[l + 1].attn_norm : nullptr;
        folded = run_layer<T>(c, c->layers[l], c->lpack[l], R, c->rows, tK, tV, N, K, Vv, c->S, tK, tV, N,
                              c->vmask, c->W, N, s, folded, next_g);
    }
    launch_rmsnorm<T>(c->x, static_cast<const T *>(c->w.final_norm), R, H, c->cfg.rms_eps,
                      static_cast<T *>(c->hT), c->lo, s);
    float *lg = logits_dev ? logits_dev : c->logits;
    gemm<T>(c, static_cast<const T *>(c->hT), H, R, H, one(c->w.lm_head, V, c->pk_lm), V, lg, V, EPI_STORE,
            s);
    launch_argmax(lg, R, V, argmax_dev, c->tks, s);
    return post_status(c, s);
}

// Compaction after an acceptance kernel has written acc_path / acc_L0 / acc_a:
// the accepted nodes' K/V move into the cache, their features become the
// draft's pending rows.
template <typename T>
msd_status compact_impl(msd_ctx *c, cudaStream_t s, int grow) {
    launch_compact_kv(c->tree_kv, c->target_kv, c->acc_path, c->acc_L0, c->acc_a, c->NL, c->B, c->nh,
                      c->N, c->S, c->D1, (int)(c->hd * c->esz), c->lo * (long)c->esz, c->status, s);
    launch_pend_h<T>(static_cast<const T *>(c->hT), c->acc_path, c->acc_a, c->B, c->N, c->D1, c->H,
                     static_cast<T *>(c->pend_h), c->lo, s);
    if (!c->capturing)
        for (int b = 0; b < c->B; ++b) c->L_bound[b] += grow < 0 ? c->D1 : grow;
    return post_status(c, s);
}

template <typename T>
msd_status accept_impl(msd_ctx *c, const msd_tree *tree, const int32_t *argmax, int32_t *path,
                       int32_t *alen, int32_t *bonus, int32_t *imap, cudaStream_t s, int grow = -1) {
    TreeIn t{tree->tokens, tree->parent, tree->depth, tree->mask, tree->n_nodes};
    launch_accept(t, argmax, c->B, c->N, c->D, c->seq_len, c->n_pend, c->root, c->pend_next,
                  c->acc_path, c->acc_L0, c->acc_a, path, alen, bonus, imap, s);
    return compact_impl<T>(c, s, grow);
}

// Speculative sampling at temperature T > 0 (Eq. 6 over the tree), then the
// same compaction. `logits` are the verify pass's [B][N][V].
template <typename T>
msd_status accept_sample_impl(msd_ctx *c, const msd_tree *tree, const float *logits, float temp,
                              const float *u, int32_t *path, int32_t *alen, int32_t *bonus,
                              int32_t *imap, cudaStream_t s) {
    TreeIn t{tree->tokens, tree->parent, tree->depth, tree->mask, tree->n_nodes};
    if (!launch_accept_sample(t, logits, c->B, c->N, c->D, c->k, c->V, (float)(1.0 / (double)temp), u,
                              c->samp_max, c->samp_sum, c->seq_len, c->n_pend, c->root, c->pend_next,
                              c->acc_path, c->acc_L0, c->acc_a, path, alen, bonus, imap, c->status, s)) {
        const cudaError_t e = cudaGetLastError();
        return fail(c, MSD_ERR_CUDA, std::string("sampling kernels did not launch: ") + cudaGetErrorString(e));
    }
    return compact_impl<T>(c, s, -1);
}

// Plain greedy autoregressive decoding, the baseline of the speedup ratio
// (Sec. 4.1, Eq. 9's T_p): a tree of the root alone, verified and accepted —
// one target forward over each request's root token at position L, its K/V
// appended at L, the argmax the next root.
template <typename T>
msd_status ar_impl(msd_ctx *c, int32_t *token_out, cudaStream_t s) {
    launch_root_tree(c->root, c->B, c->N, c->W, c->ar_tree.tokens, c->ar_tree.parent, c->ar_tree.depth,
                     c->ar_tree.mask, c->ar_tree.n_nodes, s);
    msd_status st = verify_impl<T>(c, &c->ar_tree, c->ar_argmax, nullptr, s);
    if (st == MSD_OK)
        st = accept_impl<T>(c, &c->ar_tree, c->ar_argmax, nullptr, nullptr, token_out, nullptr, s, 1);
    return st;
}

// A step writes at most positions L .. L+D (tree K/V land at L+depth only in
// scratch), so L + D + 1 <= max_seq keeps every write in bounds. The host
// keeps an upper bound of L and reads the true value only when the bound
// says it may be too large.
msd_status check_capacity(msd_ctx *c) {
    bool tight = false;
    for (int b = 0; b < c->B; ++b)
        if (c->L_bound[b] + c->D + 1 > c->S) tight = true;
    if (!tight) return MSD_OK;
    std::vector<int> L(c->B);
    CU(cudaDeviceSynchronize());
    CU(cudaMemcpy(L.data(), c->seq_len, sizeof(int) * c->B, cudaMemcpyDeviceToHost));
    for (int b = 0; b < c->B; ++b) {
        c->L_bound[b] = L[b];
        if (L[b] + c->D + 1 > c->S) return fail(c, MSD_ERR_CAPACITY, "request would exceed max_seq");
    }
    return MSD_OK;
}

// Packs every GEMM weight once (tile-contiguous, pre-swizzled) so that a
// pipeline stage is one contiguous 16 KB read.
bool pack_one(msd_ctx *c, const GemmW &W, int K, const void **out) {
    void *dst = nullptr;
    if (!dalloc(c, &dst, gemm_pack_bytes(W, K))) return false;
    gemm_pack(W, K, dst, 0);
    *out = dst;
    return true;
}

bool pack_glu(msd_ctx *c, const void *gate, const void *up, int F, int K, const void **out) {
    void *dst = nullptr;
    if (!dalloc(c, &dst, gemm_pack_glu_bytes(F, K))) return false;
    gemm_pack_glu(gate, up, F, K, dst, 0);
    *out = dst;
    return true;
}

bool pack_layer(msd_ctx *c, const msd_layer &lw, msd_ctx::LayerPack &lp) {
    const int H = c->H, F = c->F;
    return pack_one(c, GemmW{{lw.wq, lw.wk, lw.wv}, {H, H, H}, 3, nullptr}, H, &lp.qkv) &&
           pack_one(c, GemmW{{lw.wo, nullptr, nullptr}, {H, 0, 0}, 1, nullptr}, H, &lp.o) &&
           pack_glu(c, lw.w_gate, lw.w_up, F, H, &lp.gu) &&
           pack_one(c, GemmW{{lw.w_down, nullptr, nullptr}, {H, 0, 0}, 1, nullptr}, F, &lp.down);
}

bool pack_weights(msd_ctx *c) {
    for (int l = 0; l < c->NL; ++l)
        if (!pack_layer(c, c->layers[l], c->lpack[l])) return false;
    if (!pack_layer(c, c->w.draft, c->dpack)) return false;
    if (!pack_one(c, one(c->w.lm_head, c->V), c->H, &c->pk_lm)) return false;
    if (!pack_one(c, one(c->w.draft_fc, c->H), 2 * c->H, &c->pk_fc)) return false;
    return cudaDeviceSynchronize() == cudaSuccess;
}

msd_status validate_config(const msd_config *g) {
    if (!g) return MSD_ERR_INVALID;
    if (g->n_layers < 1 || g->hidden < 1 || g->n_heads < 1 || g->ffn < 1 || g->vocab < 2)
        return MSD_ERR_INVALID;
    if (g->head_dim != 64 && g->head_dim != 128) return MSD_ERR_INVALID;
    if (g->n_heads * g->head_dim != g->hidden) return MSD_ERR_INVALID;
    if (g->hidden % 64 || g->ffn % 16 || g->hidden > 8192) return MSD_ERR_INVALID;
    if (g->dtype != MSD_F32 && g->dtype != MSD_BF16) return MSD_ERR_INVALID;
    if (g->max_batch < 1 || g->max_seq < 2) return MSD_ERR_INVALID;
    if (g->tree_nodes < 1 || g->tree_nodes > 256) return MSD_ERR_INVALID;
    if (g->tree_depth < 1 || g->tree_depth > TREE_MAXD) return MSD_ERR_INVALID;
    if (g->topk < 1 || g->topk > TREE_MAXK || g->topk > g->vocab) return MSD_ERR_INVALID;
    if (!topk_supported(g->vocab, g->topk)) return MSD_ERR_INVALID;
    if (g->draft_input != MSD_DRAFT_EMBEDDING && g->draft_input != MSD_DRAFT_CONCAT &&
        g->draft_input != MSD_DRAFT_FEATURE)
        return MSD_ERR_INVALID;
    const long cand = g->topk + (long)(g->tree_depth - 1) * g->topk * g->topk;
    if (cand < g->tree_nodes - 1) return MSD_ERR_INVALID;
    return MSD_OK;
}

template <typename T>
msd_status step_eager(msd_ctx *c, const msd_tree *tree, int32_t *argmax, int32_t *path,
                      int32_t *alen, int32_t *bonus, cudaStream_t s) {
    msd_status st = draft_impl<T>(c, tree, nullptr, s);
    if (st == MSD_OK) st = verify_impl<T>(c, tree, argmax, nullptr, s);
    if (st == MSD_OK) st = accept_impl<T>(c, tree, argmax, path, alen, bonus, nullptr, s);
    return st;
}

// The sampling step: the verify logits stay in the context's buffer.
template <typename T>
msd_status step_sample_eager(msd_ctx *c, const msd_tree *tree, int32_t *argmax, float temp,
                             const float *u, int32_t *path, int32_t *alen, int32_t *bonus,
                             cudaStream_t s) {
    msd_status st = draft_impl<T>(c, tree, nullptr, s);
    if (st == MSD_OK) st = verify_impl<T>(c, tree, argmax, nullptr, s);
    if (st == MSD_OK) st = accept_sample_impl<T>(c, tree, c->logits, temp, u, path, alen, bonus, nullptr, s);
    return st;
}

// Sampling parameters of a kind-2 step.
struct SampleArgs {
    const float *u;
    float temp;
};

bool same_buffers(const msd_ctx::StepGraph &g, int kind, const msd_tree *t, const void *a,
                         const void *p, const void *l, const void *b, const SampleArgs *sa) {
    return g.kind == kind && g.tree.tokens == t->tokens && g.tree.parent == t->parent && g.tree.depth == t->depth &&
           g.tree.mask == t->mask && g.tree.n_nodes == t->n_nodes && g.argmax == a &&
           g.path == p && g.alen == l && g.bonus == b &&
           (!sa || (g.u == sa->u && g.temp == sa->temp));
}

}  // namespace

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------
extern "C" {

msd_status msd_create(const msd_config *cfg, const msd_weights *w, msd_ctx **out) {
    if (!out) return MSD_ERR_INVALID;
    *out = nullptr;
    if (validate_config(cfg) != MSD_OK || !w || !w->layers) return MSD_ERR_INVALID;
    const void *need[] = {w->embed, w->final_norm, w->lm_head, w->draft_fc, w->draft.attn_norm,
                          w->draft.wq, w->draft.wk, w->draft.wv, w->draft.wo, w->draft.mlp_norm,
                          w->draft.w_gate, w->draft.w_up, w->draft.w_down};
    for (const void *p : need)
        if (!p) return MSD_ERR_INVALID;
    for (int l = 0; l < cfg->n_layers; ++l) {
        const msd_layer &L = w->layers[l];
        const void *lp[] = {L.attn_norm, L.wq, L.wk, L.wv, L.wo, L.mlp_norm, L.w_gate, L.w_up, L.w_down};
        for (const void *p : lp)
            if (!p) return MSD_ERR_INVALID;
    }
    // (arguments are checked first: that needs no GPU)
    if (report_stale_error("msd_create")) return MSD_ERR_CUDA;
    msd_ctx *c = new msd_ctx();
    c->cfg = *cfg;
    c->w = *w;
    c->layers.assign(w->layers, w->layers + cfg->n_layers);
    c->w.layers = c->layers.data();
    cudaGetDevice(&c->dev);
    c->esz = cfg->dtype == MSD_BF16 ? 2 : 4;
    c->B = cfg->max_batch; c->S = cfg->max_seq; c->N = cfg->tree_nodes; c->D = cfg->tree_depth;
    c->D1 = c->D + 1; c->k = cfg->topk; c->H = cfg->hidden; c->F = cfg->ffn; c->V = cfg->vocab;
    c->nh = cfg->n_heads; c->hd = cfg->head_dim; c->NL = cfg->n_layers;
    c->W = (c->N + 63) / 64;
    c->C = c->k + (c->D - 1) * c->k * c->k;
    c->Td = std::max(1, (c->D - 1) * c->k);
    c->Wd = (c->Td + 63) / 64;
    c->chunk = std::min(c->S, 1024);
    c->Rmax = std::max(std::max(c->B * c->N, c->B * c->D1), std::max(c->B * c->k, c->chunk));
    c->Rlog = std::max(std::max(c->B * c->N, c->B * c->k), 1);
    c->L_bound.assign(c->B, 0);
    const size_t e = c->esz, H = c->H, F = c->F, R = c->Rmax;
    bool ok = true;
    // Buffers in the model dtype. In bf16 contexts they are split pairs: one
    // arena holds them all, and its upper half (lo elements on) their lo planes.
    struct Carve { void **p; size_t elems; };
    const Carve split_bufs[] = {
        {&c->target_kv, (size_t)c->NL * 2 * kv_layer_elems(c, c->S)},
        {&c->draft_kv, 2 * kv_layer_elems(c, c->S)},
        {&c->tree_kv, (size_t)c->NL * 2 * kv_layer_elems(c, c->N)},
        {&c->dtree_kv, 2 * kv_layer_elems(c, c->Td)},
        {&c->pend_h, (size_t)c->B * c->D1 * H},
        {&c->xn, R * H},
        {&c->q, R * H},
        {&c->attn, R * H},
        {&c->act, R * F},
        {&c->xfc, R * 2 * H},
        {&c->xr, R * H},
        {&c->hT, (size_t)c->B * c->N * H},
        {&c->h_all, (size_t)c->S * H},
    };
    if (cfg->dtype == MSD_BF16) {
        size_t total = 0;
        for (const Carve &b : split_bufs) total += (b.elems + 127) / 128 * 128;     // 256-byte pieces
        const size_t quantum = H * 64;      // the lo offset is a whole number of rows of any buffer
        total = (total + quantum - 1) / quantum * quantum;
        void *arena = nullptr;
        ok &= dalloc(c, &arena, 2 * total * e);
        if (ok) {
            size_t off = 0;
            for (const Carve &b : split_bufs) {
                *b.p = static_cast<bf16 *>(arena) + off;
                off += (b.elems + 127) / 128 * 128;
            }
            c->lo = (long)total;
        }
    } else {
        for (const Carve &b : split_bufs) ok &= dalloc(c, b.p, b.elems * e);
    }
    ok &= dalloc(c, &c->seq_len, sizeof(int) * c->B);
    ok &= dalloc(c, &c->n_pend, sizeof(int) * c->B);
    ok &= dalloc(c, &c->root, sizeof(int) * c->B);
    ok &= dalloc(c, &c->pend_next, sizeof(int) * c->B * c->D1);
    ok &= dalloc(c, &c->x, R * H * 4);
    ok &= dalloc(c, &c->qkv, R * 3 * H * 4);
    c->ss_ld = (H + 127) / 128;
    ok &= dalloc(c, &c->ss_part, R * (size_t)c->ss_ld * 4);
    ok &= dalloc(c, &c->gu, R * std::max<size_t>(2 * F, glu_rows(c->F)) * 4);
    ok &= dalloc(c, &c->logits, (size_t)c->Rlog * c->V * 4);
    ok &= dalloc(c, &c->argmax_tmp, sizeof(int) * 4);
    ok &= dalloc(c, &c->rows, sizeof(RowDesc) * R);
    ok &= dalloc(c, &c->src, sizeof(int) * std::max<size_t>(R, c->S));
    ok &= dalloc(c, &c->vmask, sizeof(uint64_t) * c->B * c->N * c->W);
    ok &= dalloc(c, &c->cand_tok, sizeof(int) * c->B * c->C);
    ok &= dalloc(c, &c->cand_par, sizeof(int) * c->B * c->C);
    ok &= dalloc(c, &c->cand_depth, sizeof(int) * c->B * c->C);
    ok &= dalloc(c, &c->cand_score, sizeof(float) * c->B * c->C);
    ok &= dalloc(c, &c->node_of, sizeof(int) * c->B * c->C);
    ok &= dalloc(c, &c->frontier, sizeof(int) * 2 * c->B * c->k);
    ok &= dalloc(c, &c->hhat_root, sizeof(float) * c->B * H);
    ok &= dalloc(c, &c->hhat_slot, sizeof(float) * c->B * c->Td * H);
    ok &= dalloc(c, &c->slot_mask, sizeof(uint64_t) * c->B * c->Td * c->Wd);
    ok &= dalloc(c, &c->row_mask, sizeof(uint64_t) * c->B * c->k * c->Wd);
    ok &= dalloc(c, &c->topk_ids, sizeof(int) * c->Rlog * c->k);
    ok &= dalloc(c, &c->topk_logp, sizeof(float) * c->Rlog * c->k);
    ok &= dalloc(c, &c->tks.ws, sizeof(float) * topk_scratch_floats(c->Rlog, c->V));
    ok &= dalloc(c, &c->tks.counters, sizeof(int) * c->Rlog);
    ok &= dalloc(c, &c->acc_path, sizeof(int) * c->B * c->D1);
    ok &= dalloc(c, &c->acc_L0, sizeof(int) * c->B);
    ok &= dalloc(c, &c->acc_a, sizeof(int) * c->B);
    ok &= dalloc(c, &c->samp_max, sizeof(float) * c->B * c->N);
    ok &= dalloc(c, &c->samp_sum, sizeof(double) * c->B * c->N);
    ok &= dalloc(c, &c->ar_tree.tokens, sizeof(int) * c->B * c->N);
    ok &= dalloc(c, &c->ar_tree.parent, sizeof(int) * c->B * c->N);
    ok &= dalloc(c, &c->ar_tree.depth, sizeof(int) * c->B * c->N);
    ok &= dalloc(c, &c->ar_tree.mask, sizeof(uint64_t) * c->B * c->N * c->W);
    ok &= dalloc(c, &c->ar_tree.n_nodes, sizeof(int) * c->B);
    ok &= dalloc(c, &c->ar_argmax, sizeof(int) * c->B * c->N);
    ok &= dalloc(c, &c->rope_tab, sizeof(float2) * (size_t)c->S * (c->hd / 2));
    ok &= dalloc(c, &c->emb_all, (size_t)c->S * H * e);
    ok &= dalloc(c, &c->status, sizeof(int));
    if (ok) ok = cudaMallocHost(&c->status_host, sizeof(int)) == cudaSuccess;
    if (ok) ok = cudaEventCreateWithFlags(&c->status_ev, cudaEventDisableTiming) == cudaSuccess;
    if (ok && cfg->dtype == MSD_BF16) ok = gemm_plan_create(&c->gplan, c->Rmax, c->H, c->F, c->V);
    if (ok && cfg->dtype == MSD_BF16) ok = attn_tc_plan_create(&c->aplan);
    c->lpack.assign(c->NL, msd_ctx::LayerPack());
    if (ok && cfg->dtype == MSD_BF16) ok = pack_weights(c);
    if (!ok) {
        msd_destroy(c);
        cudaGetLastError();
        return MSD_ERR_OOM;
    }
    *c->status_host = 0;
    // RoPE table: (cos, sin) of pos * base^(-2i/hd), computed in double.
    std::vector<float2> tab((size_t)c->S * (c->hd / 2));
    for (int p = 0; p < c->S; ++p)
        for (int i = 0; i < c->hd / 2; ++i) {
            const double th = std::pow((double)cfg->rope_base, -2.0 * i / c->hd);
            const double ang = (double)p * th;
            tab[(size_t)p * (c->hd / 2) + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
        }
    if (cudaMemcpy(c->rope_tab, tab.data(), sizeof(float2) * tab.size(), cudaMemcpyHostToDevice) !=
            cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess) {
        msd_destroy(c);
        return MSD_ERR_CUDA;
    }
    *out = c;
    return MSD_OK;
}

#define MSD_TEARDOWN(call)                                                               \
    do {                                                                                 \
        cudaError_t e_ = (call);                                                         \
        if (e_ != cudaSuccess)                                                           \
            fprintf(stderr, "msd_destroy: %s: %s\n", #call, cudaGetErrorString(e_));     \
    } while (0)

msd_status msd_destroy(msd_ctx *c) {
    if (!c) return MSD_OK;
    report_stale_error("msd_destroy");
    MSD_TEARDOWN(cudaDeviceSynchronize());
    for (void *p : c->allocs) MSD_TEARDOWN(cudaFree(p));
    if (c->status_host) MSD_TEARDOWN(cudaFreeHost(c->status_host));
    if (c->status_ev) MSD_TEARDOWN(cudaEventDestroy(c->status_ev));
    if (c->gplan) gemm_plan_destroy(c->gplan);
    if (c->aplan) attn_tc_plan_destroy(c->aplan);
    if (c->pk_scratch) MSD_TEARDOWN(cudaFree(c->pk_scratch));
    for (auto &g : c->graphs)
        if (g.exec) MSD_TEARDOWN(cudaGraphExecDestroy(g.exec));
    if (c->cap_stream) {
        const cudaError_t e = cudaStreamDestroy(c->cap_stream);
        if (e != cudaSuccess)
            fprintf(stderr, "msd_destroy: ctx %p: cudaStreamDestroy(%p): %s\n", (void *)c,
                    (void *)c->cap_stream, cudaGetErrorString(e));
    }
    report_stale_error("msd_destroy (end)");
    delete c;
    return MSD_OK;
}

msd_status msd_prefill(msd_ctx *c, int32_t batch, const int32_t *seq_len_host,
                       const int32_t *ids_dev, int32_t ids_stride, const void *vis_dev,
                       const int64_t *vis_off_host, int32_t *root_out_dev, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_prefill"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (batch < 1 || batch > c->B || !seq_len_host || !ids_dev)
        return fail(c, MSD_ERR_INVALID, "bad batch or null argument");
    if (batch != c->B) return fail(c, MSD_ERR_INVALID, "batch must equal max_batch");
    for (int b = 0; b < batch; ++b) {
        if (seq_len_host[b] < 1) return fail(c, MSD_ERR_INVALID, "empty prompt");
        if (seq_len_host[b] > ids_stride) return fail(c, MSD_ERR_INVALID, "prompt longer than ids_stride");
        if ((long)seq_len_host[b] + c->D + 1 > c->S) return fail(c, MSD_ERR_CAPACITY, "prompt exceeds max_seq");
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (c->cfg.dtype == MSD_BF16)
        return prefill_impl<bf16>(c, batch, seq_len_host, ids_dev, ids_stride, vis_dev, vis_off_host,
                                  root_out_dev, s);
    return prefill_impl<float>(c, batch, seq_len_host, ids_dev, ids_stride, vis_dev, vis_off_host,
                               root_out_dev, s);
}

static bool tree_ok(const msd_tree *t) {
    return t && t->tokens && t->parent && t->depth && t->mask;
}

msd_status msd_draft_tree(msd_ctx *c, const msd_tree *out, const msd_draft_record *rec,
                          void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_draft_tree"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(out)) return fail(c, MSD_ERR_INVALID, "null tree array");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    if (c->draft_stale)
        return fail(c, MSD_ERR_INVALID, "msd_ar_step ran since the last msd_prefill: the draft cache is stale");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (c->cfg.dtype == MSD_BF16) return draft_impl<bf16>(c, out, rec, s);
    return draft_impl<float>(c, out, rec, s);
}

msd_status msd_verify(msd_ctx *c, const msd_tree *tree, int32_t *argmax_dev, float *logits_dev,
                      void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_verify"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(tree) || !argmax_dev) return fail(c, MSD_ERR_INVALID, "null tree or argmax");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (c->cfg.dtype == MSD_BF16) return verify_impl<bf16>(c, tree, argmax_dev, logits_dev, s);
    return verify_impl<float>(c, tree, argmax_dev, logits_dev, s);
}

msd_status msd_accept_compact(msd_ctx *c, const msd_tree *tree, const int32_t *argmax_dev,
                              int32_t *path_dev, int32_t *accept_len_dev, int32_t *bonus_dev,
                              int32_t *index_map_dev, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_accept_compact"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(tree) || !argmax_dev) return fail(c, MSD_ERR_INVALID, "null tree or argmax");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (c->cfg.dtype == MSD_BF16)
        return accept_impl<bf16>(c, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev,
                                 index_map_dev, s);
    return accept_impl<float>(c, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev,
                              index_map_dev, s);
}

namespace {

// One step (kind 0: draft, verify, accept; kind 1: plain greedy; kind 2:
// draft, verify, sample) recorded once into a CUDA graph per set of buffers,
// then replayed: every kernel reads the lengths it needs from device state.
msd_status step_kind_eager(msd_ctx *c, int kind, const msd_tree *tree, int32_t *argmax_dev,
                           int32_t *path_dev, int32_t *accept_len_dev, int32_t *bonus_dev,
                           const SampleArgs *sa, cudaStream_t s) {
    const bool bf = c->cfg.dtype == MSD_BF16;
    if (kind == 1) return bf ? ar_impl<bf16>(c, bonus_dev, s) : ar_impl<float>(c, bonus_dev, s);
    if (kind == 2)
        return bf ? step_sample_eager<bf16>(c, tree, argmax_dev, sa->temp, sa->u, path_dev, accept_len_dev,
                                            bonus_dev, s)
                  : step_sample_eager<float>(c, tree, argmax_dev, sa->temp, sa->u, path_dev, accept_len_dev,
                                             bonus_dev, s);
    return bf ? step_eager<bf16>(c, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, s)
              : step_eager<float>(c, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, s);
}

msd_status run_step_graph(msd_ctx *c, int kind, const msd_tree *tree, int32_t *argmax_dev, int32_t *path_dev,
                          int32_t *accept_len_dev, int32_t *bonus_dev, const SampleArgs *sa,
                          cudaStream_t s) {
    msd_status st;
    const int grow = kind == 1 ? 1 : c->D1;      // upper bound of L's growth per step
    // While GEMM profiling is on, steps run eagerly (events bracket each GEMM).
    if (c->cfg.dtype == MSD_BF16 && c->gplan && gemm_profile_on(c->gplan)) {
        st = step_kind_eager(c, kind, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, sa, s);
        return st == MSD_OK ? post_status(c, s) : st;
    }
    const bool stamped = c->gplan && gemm_stamp_on(c->gplan);
    msd_ctx::StepGraph *g = nullptr;
    for (auto &x : c->graphs)
        if (x.stamped == stamped && same_buffers(x, kind, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, sa))
            g = &x;
    if (!g) {
        msd_ctx::StepGraph ng;
        ng.kind = kind;
        ng.stamped = stamped;
        ng.tree = *tree;
        ng.argmax = argmax_dev; ng.path = path_dev; ng.alen = accept_len_dev; ng.bonus = bonus_dev;
        if (sa) { ng.u = sa->u; ng.temp = sa->temp; }
        if (!c->cap_stream)   // graphs are recorded on a stream of the context's own
            CU(cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking));
        const long l0 = launch_count();
        c->capturing = true;
        cudaGraph_t graph = nullptr;
        cudaError_t ce = cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal);
        if (ce == cudaSuccess) {
            if (stamped) gemm_stamp_begin(c->gplan);    // the graph closes its own window
            st = step_kind_eager(c, kind, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, sa,
                                 c->cap_stream);
            if (stamped) gemm_stamp_end(c->gplan, c->cap_stream);
            ce = cudaStreamEndCapture(c->cap_stream, &graph);
        } else {
            st = MSD_OK;
        }
        c->capturing = false;
        ng.kernels = launch_count() - l0;
        c->captured_launches += ng.kernels;
        if (ce != cudaSuccess || st != MSD_OK || !graph) {
            if (graph) cudaGraphDestroy(graph);
            cudaGetLastError();
            return st != MSD_OK ? st : fail(c, MSD_ERR_CUDA, std::string("step capture: ") +
                                                                 cudaGetErrorString(ce));
        }
        ce = cudaGraphInstantiate(&ng.exec, graph, 0);
        cudaGraphDestroy(graph);
        if (ce != cudaSuccess)
            return fail(c, MSD_ERR_CUDA, std::string("step graph: ") + cudaGetErrorString(ce));
        if (c->graphs.size() >= 8) {     // keep the most used graphs
            auto victim = std::min_element(c->graphs.begin(), c->graphs.end(),
                                           [](const msd_ctx::StepGraph &a,
                                              const msd_ctx::StepGraph &b) { return a.uses < b.uses; });
            cudaGraphExecDestroy(victim->exec);
            c->graphs.erase(victim);
        }
        c->graphs.push_back(ng);
        g = &c->graphs.back();
    }
    CU(cudaGraphLaunch(g->exec, s));
    g->uses += 1;
    c->graph_kernels += g->kernels;
    for (int b = 0; b < c->B; ++b) c->L_bound[b] += grow;
    return post_status(c, s);
}

}  // namespace

msd_status msd_step(msd_ctx *c, const msd_tree *tree, int32_t *argmax_dev, int32_t *path_dev,
                    int32_t *accept_len_dev, int32_t *bonus_dev, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_step"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(tree) || !argmax_dev) return fail(c, MSD_ERR_INVALID, "null tree or argmax");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    if (c->draft_stale)
        return fail(c, MSD_ERR_INVALID, "msd_ar_step ran since the last msd_prefill: the draft cache is stale");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    return run_step_graph(c, 0, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, nullptr,
                          static_cast<cudaStream_t>(stream));
}

msd_status msd_ar_step(msd_ctx *c, int32_t *token_dev, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_ar_step"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!token_dev) return fail(c, MSD_ERR_INVALID, "null token output");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    c->draft_stale = true;
    return run_step_graph(c, 1, &c->ar_tree, c->ar_argmax, nullptr, nullptr, token_dev, nullptr,
                          static_cast<cudaStream_t>(stream));
}

// The kernel scales logits by the fp32 1/T: T must be finite, > 0, and have a
// finite fp32 reciprocal.
// The sampling kernel keeps a bitmap of the rejected tokens in shared memory
// (one bit per token, within the default 48 KB of dynamic shared memory).
constexpr int MSD_SAMPLE_MAX_VOCAB = SAMPLE_MAX_VOCAB;

static bool temperature_ok(float t) {
    return std::isfinite(t) && t > 0.f && std::isfinite((float)(1.0 / (double)t));
}

msd_status msd_accept_sample(msd_ctx *c, const msd_tree *tree, const float *logits_dev, float temperature,
                             const float *u_dev, int32_t *path_dev, int32_t *accept_len_dev,
                             int32_t *bonus_dev, int32_t *index_map_dev, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_accept_sample"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(tree) || !u_dev) return fail(c, MSD_ERR_INVALID, "null tree or uniforms");
    if (!temperature_ok(temperature)) return fail(c, MSD_ERR_INVALID, "temperature must be finite and > 0");
    if (c->V > MSD_SAMPLE_MAX_VOCAB) return fail(c, MSD_ERR_INVALID, "vocabulary too large for sampling");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const float *lg = logits_dev ? logits_dev : c->logits;
    if (c->cfg.dtype == MSD_BF16)
        return accept_sample_impl<bf16>(c, tree, lg, temperature, u_dev, path_dev, accept_len_dev, bonus_dev,
                                        index_map_dev, s);
    return accept_sample_impl<float>(c, tree, lg, temperature, u_dev, path_dev, accept_len_dev, bonus_dev,
                                     index_map_dev, s);
}

msd_status msd_step_sample(msd_ctx *c, const msd_tree *tree, float temperature, const float *u_dev,
                           int32_t *argmax_dev, int32_t *path_dev, int32_t *accept_len_dev,
                           int32_t *bonus_dev, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_step_sample"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(tree) || !argmax_dev || !u_dev)
        return fail(c, MSD_ERR_INVALID, "null tree, argmax or uniforms");
    if (!temperature_ok(temperature)) return fail(c, MSD_ERR_INVALID, "temperature must be finite and > 0");
    if (c->V > MSD_SAMPLE_MAX_VOCAB) return fail(c, MSD_ERR_INVALID, "vocabulary too large for sampling");
    if (!c->prefilled) return fail(c, MSD_ERR_INVALID, "msd_prefill has not run");
    if (c->draft_stale)
        return fail(c, MSD_ERR_INVALID, "msd_ar_step ran since the last msd_prefill: the draft cache is stale");
    st = check_capacity(c);
    if (st != MSD_OK) return st;
    const SampleArgs sa{u_dev, temperature};
    return run_step_graph(c, 2, tree, argmax_dev, path_dev, accept_len_dev, bonus_dev, &sa,
                          static_cast<cudaStream_t>(stream));
}

msd_status msd_linear(msd_ctx *c, const void *x, int32_t ldx, int32_t m, int32_t k, const void *w,
                      int32_t o, float *y, int32_t ldy, int32_t accumulate, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_linear"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    if (!x || !w || !y || m <= 0 || k <= 0 || o <= 0 || ldx < k || ldy < o)
        return fail(c, MSD_ERR_INVALID, "bad msd_linear arguments");
    if (c->cfg.dtype == MSD_BF16 && (ldx % 8 || k % 8))
        return fail(c, MSD_ERR_INVALID, "bf16 rows must be 16-byte aligned");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    GemmW W = one(w, o);
    const int epi = accumulate ? EPI_ADD : EPI_STORE;
    if (c->cfg.dtype == MSD_BF16) {
        // pack w into the context's scratch (grown on demand), then the GEMM
        const size_t need = gemm_pack_bytes(W, k);
        if (need > c->pk_scratch_bytes) {
            CU(cudaStreamSynchronize(s));
            if (c->pk_scratch) CU(cudaFree(c->pk_scratch));
            c->pk_scratch = nullptr;
            c->pk_scratch_bytes = 0;
            if (cudaMalloc(&c->pk_scratch, need) != cudaSuccess)
                return fail(c, MSD_ERR_OOM, "msd_linear: packing scratch");
            c->pk_scratch_bytes = need;
        }
        gemm_pack(W, k, c->pk_scratch, s);
        W.packed = c->pk_scratch;
        gemm<bf16>(c, static_cast<const bf16 *>(x), ldx, m, k, W, o, y, ldy, epi, s, false);
    } else
        gemm<float>(c, static_cast<const float *>(x), ldx, m, k, W, o, y, ldy, epi, s);
    return post_status(c, s);
}

msd_status msd_profile_enable(msd_ctx *c, int32_t mode) {
    if (!c || mode < 0 || mode > 2) return MSD_ERR_INVALID;
    c->err.clear();
    if (c->gplan && !gemm_profile_enable(c->gplan, mode))
        return fail(c, MSD_ERR_CUDA, "GEMM launch stamps: reset failed");
    return MSD_OK;
}

msd_status msd_profile_read(msd_ctx *c, msd_profile *out) {
    if (!c || !out) return MSD_ERR_INVALID;
    memset(out, 0, sizeof *out);
    out->kernel_launches = launch_count() - c->captured_launches + c->graph_kernels;
    if (c->gplan) {
        const GemmProfile g = gemm_profile_read(c->gplan);
        out->gemm_launches = g.launches;
        out->gemm_ms = g.ms;
        out->gemm_bytes = g.bytes;
        out->gemm_weight_bytes = g.weight_bytes;
        out->gemm_critical_ms = g.critical_ms;
        out->windows = g.windows;
        out->gemm_flops = g.flops;
        out->gemm_mma_flops = g.mma_flops;
        out->gemm_prefetch_bytes = g.prefetch_bytes;
    }
    return MSD_OK;
}

msd_status msd_profile_slots(msd_ctx *c, msd_kernel_slot *out, int32_t max, int32_t *n) {
    if (!c || !n || max < 0 || (max > 0 && !out)) return MSD_ERR_INVALID;
    *n = 0;
    if (!c->gplan || max == 0) return MSD_OK;
    // (a window holds at most 2560 stamped launches)
    const int cap = std::min<int32_t>(max, 4096);
    std::vector<GemmSlot> g((size_t)cap);
    const int k = gemm_profile_slots(c->gplan, g.data(), cap);
    if (k < 0) return fail(c, MSD_ERR_CUDA, "reading the stamp slots failed");
    for (int i = 0; i < k; ++i) {
        out[i].kind = g[i].kind;
        out[i].rows = g[i].rows;
        out[i].outputs = g[i].outputs;
        out[i].inner = g[i].inner;
        out[i].launches = g[i].launches;
        out[i].bytes = g[i].bytes;
        out[i].critical_ms = g[i].critical_ms;
        out[i].span_ms = g[i].ms;
    }
    *n = k;
    return MSD_OK;
}

msd_status msd_tree_complete(msd_ctx *c, const msd_tree *tree, int32_t request, void *stream) {
    if (!c) return MSD_ERR_INVALID;
    c->err.clear();
    if (report_stale_error("msd_tree_complete"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    msd_status st = check_status(c);
    if (st != MSD_OK) return st;
    if (!tree_ok(tree)) return fail(c, MSD_ERR_INVALID, "null tree array");
    if (request < -1 || request >= c->B) return fail(c, MSD_ERR_INVALID, "request out of range");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int b0 = request < 0 ? 0 : request, nb = request < 0 ? c->B : 1;
    launch_tree_complete(tree->parent, tree->depth, tree->mask, tree->n_nodes, b0, nb, c->N, c->status, s);
    return post_status(c, s);
}

msd_status msd_test_wait_timeout(msd_ctx *c, int64_t limit_ns, void *stream) {
    if (limit_ns < 1000 || limit_ns > 2000000000LL) return fail(c, MSD_ERR_INVALID, "limit out of range");
    if (report_stale_error("msd_test_wait_timeout"))
        return fail(c, MSD_ERR_CUDA, "a CUDA error was pending before the call");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int *status = c ? c->status : noalloc_status_word();
    if (!status) return MSD_ERR_CUDA;
    if (!launch_wait_probe(status, (long long)limit_ns, s)) return fail(c, MSD_ERR_CUDA, "probe launch failed");
    return c ? post_status(c, s) : MSD_OK;
}

msd_status msd_state(msd_ctx *c, msd_state_view *out) {
    if (!c || !out) return MSD_ERR_INVALID;
    out->target_kv = c->target_kv;
    out->draft_kv = c->draft_kv;
    out->seq_len = c->seq_len;
    out->n_pending = c->n_pend;
    out->root = c->root;
    out->elem_bytes = (int64_t)c->esz;
    out->lo_offset = (int64_t)c->lo;
    return MSD_OK;
}

const char *msd_last_error(const msd_ctx *c) {
    if (!c) return "null context";
    return c->err.c_str();
}

}  // extern "C"
