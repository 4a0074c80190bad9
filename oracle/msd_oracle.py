"""CPU oracle of one greedy MSD draft-then-verify decode step.

TEST INFRASTRUCTURE ONLY. Nothing in the product path imports, calls or links
this module: only the tests, ``__graft_entry__.smoke()`` and the bench's
``cpu_baseline`` / ``--impl reference`` legs may use it. It shares no code with
the CUDA path.

Plain, slow and written to be checked against the paper by eye. All floating
point is float64 (numpy), except the two places where the kernels take an
integer decision from a float32 value (tree scores, see ``TreeBuilder``), which
are done in float32 exactly as described there.

What it computes (arXiv 2505.14260, "Speculative Decoding Reimagined for
Multimodal Large Language Models"):

* Sec. 3.1, Eq. 1-3: the target input is the interleaved sequence of text
  embeddings E_t(t_i) and projected visual embeddings e_{v_i}.
* Sec. 3.1: the target (a LLaMA-style decoder, LLaVA-1.5) maps it to features
  h_{x_i}; the LM head maps h to p(x_{i+1} | x_{<i+1}).
* Sec. 3.2, Eq. 4-5: the feature-level draft model is one decoder layer fed
  f_{x_i} = f_down(Concat(h_{x_i}, e_{x_{i+1}})); its output goes through the
  target's LM head to give q.
* Sec. 4.1, Eq. 7 (eq:decouple): MSD feeds the raw embedding e_{x_i} at visual
  positions and keeps the concatenation at text positions.
* Sec. 3.2: drafting grows a tree of depth m, one forward pass per depth,
  expanding leaves with several candidates each.
* Sec. 3.2, Eq. 6 and the residual rule after it, at temperature 0: a draft token
  is accepted iff it equals the target argmax; on rejection the next token is the
  target argmax; if all are accepted a bonus token is taken from the target.

Readings where the paper is silent (each also listed in the design notes):
  R1 decoder: pre-norm LLaMA layer, RMSNorm y = x / sqrt(mean(x^2) + eps) * g,
     RoPE with rotate-half pairing (i, i + hd/2), theta_i = base^(-2i/hd),
     attention scale 1/sqrt(hd), SwiGLU MLP, no biases, untied LM head.
  R2 h is the output of the target's final RMSNorm; logits = lm_head @ h.
     The draft layer's output goes to the LM head with no extra norm.
  R3 tree: depth-1 = top-k of the root-slot distribution; at depth d >= 2 the k
     highest-scoring depth-(d-1) candidates are expanded with top-k children
     each; score = sum of log-probabilities along the path; the final tree keeps
     the N-1 best candidates. Ties: higher value first, then lower depth, then
     earlier creation; top-k / argmax ties go to the lower token id.
  R4 N counts the root; D = number of draft passes = maximum accepted length.
  R5 draft positions: the draft row that carries h_i sits at position i; a
     depth-d tree node sits at draft position L-1+d and target position L+d.
  R6 a prefix must end with a text token.
  R7 temperature T > 0 (speculative sampling): the target distribution at a
     node is p = softmax(logits / T). The tree's candidates are the draft's
     top-k choices, not samples of q, so the distribution that proposed a
     candidate -- given the siblings already rejected -- is a point mass at it:
     Eq. 6's min(1, p/q) accepts it with probability p(x), and the adjusted
     distribution norm(max(0, p - q)) is p with x removed and renormalised.
     Children are tried in tree order (best draft score first); the token that
     ends the walk is drawn from the adjusted p (all children rejected) or from
     p itself (a leaf). Draws are inverse-CDF in token-id order. The uniforms
     are inputs: u[d][j] for the j-th child tried at depth d, u[d][k] for the
     token drawn at depth d.
  R8 draft input of a visual prefix position (Sec. 5.3, ablation of the input
     strategy; the paper compares three): "embedding" -- MSD, Eq. 7, the raw
     visual embedding e_{x_i}; "concat" -- the Baseline of Sec. 3.3, the same
     f_down(Concat(h_{x_i}, e_{x_{i+1}})) as a text position; "feature" -- the
     target's feature h_{x_i} of that position (R2), with no concatenation.
     Text positions always take the concatenation. Only prefix positions can
     be visual: the decode step's positions are generated text.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

F64 = np.float64


# ----------------------------------------------------------------------------
# Model configuration and weights
# ----------------------------------------------------------------------------

@dataclass
class OracleConfig:
    n_layers: int
    hidden: int
    n_heads: int
    head_dim: int
    ffn: int
    vocab: int
    tree_nodes: int
    tree_depth: int
    topk: int
    rms_eps: float = 1e-6
    rope_base: float = 10000.0
    draft_input: str = "embedding"      # R8: "embedding" (MSD), "concat", "feature"


DRAFT_INPUTS = ("embedding", "concat", "feature")


class OracleModel:
    """Holds the weights (any float numpy dtype; upcast to float64 on use)."""

    def __init__(self, cfg: OracleConfig, weights: dict):
        self.cfg = cfg
        self.w = weights

    def mat(self, m) -> np.ndarray:
        return np.asarray(m, dtype=F64)


# ----------------------------------------------------------------------------
# Elementary operations (R1)
# ----------------------------------------------------------------------------

def rms_norm(x: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm of each row: x / sqrt(mean(x^2) + eps) * gain."""
    x = np.asarray(x, F64)
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(gain, F64)


def rope(x: np.ndarray, pos: np.ndarray, n_heads: int, head_dim: int,
         base: float) -> np.ndarray:
    """Rotary position embedding, rotate-half pairing (i, i + hd/2) per head.

    Element pair (a, b) = (x[i], x[i + hd/2]) at position p is rotated by the
    angle p * base^(-2i/hd).
    """
    x = np.asarray(x, F64)
    R = x.shape[0]
    half = head_dim // 2
    theta = float(base) ** (-2.0 * np.arange(half, dtype=F64) / head_dim)
    ang = np.asarray(pos, F64)[:, None] * theta[None, :]          # [R, half]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    xh = x.reshape(R, n_heads, head_dim)
    a, b = xh[..., :half], xh[..., half:]
    out = np.concatenate([a * c - b * s, b * c + a * s], axis=-1)
    return out.reshape(R, n_heads * head_dim)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def softmax(s: np.ndarray) -> np.ndarray:
    s = s - np.max(s, axis=-1, keepdims=True)
    e = np.exp(s)
    return e / np.sum(e, axis=-1, keepdims=True)


def log_softmax(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, F64)
    m = np.max(z, axis=-1, keepdims=True)
    return z - m - np.log(np.sum(np.exp(z - m), axis=-1, keepdims=True))


def topk_ids(values: np.ndarray, k: int) -> np.ndarray:
    """Indices of the k largest values; ties go to the lower index (R3)."""
    v = np.asarray(values)
    order = sorted(range(v.shape[0]), key=lambda i: (-v[i], i))
    return np.asarray(order[:k], dtype=np.int64)


def argmax_lowest(values: np.ndarray) -> int:
    """Argmax; among equal maxima the lowest index (R3)."""
    v = np.asarray(values)
    return int(np.flatnonzero(v == v.max())[0])


# ----------------------------------------------------------------------------
# Attention with an explicit visibility structure
# ----------------------------------------------------------------------------

def attend(q, cache_k, cache_v, prefix_len, tree_k, tree_v, tree_vis,
           n_heads, head_dim):
    """Softmax attention of each query row over the keys it may see.

    Row r sees cache rows [0, prefix_len[r]) and the tree rows j with
    tree_vis[r, j] true. Keys and values are [rows, H]. Written as masked
    attention: the scores of a block of rows against every key, the keys a row
    may not see set to -inf (weight exactly 0 after the softmax), then the
    weighted sum of the values.
    """
    R = q.shape[0]
    H = n_heads * head_dim
    keys = [np.asarray(cache_k, F64).reshape(-1, H)]
    vals = [np.asarray(cache_v, F64).reshape(-1, H)]
    C = keys[0].shape[0]
    has_tree = tree_k is not None and tree_k.shape[0] > 0
    if has_tree:
        keys.append(np.asarray(tree_k, F64).reshape(-1, H))
        vals.append(np.asarray(tree_v, F64).reshape(-1, H))
    K = np.concatenate(keys, axis=0).reshape(-1, n_heads, head_dim).transpose(1, 0, 2)   # [h, T, d]
    V = np.concatenate(vals, axis=0).reshape(-1, n_heads, head_dim).transpose(1, 0, 2)
    scale = 1.0 / np.sqrt(head_dim)
    out = np.zeros((R, H), F64)
    for r0 in range(0, R, 128):
        r1 = min(R, r0 + 128)
        qh = np.asarray(q[r0:r1], F64).reshape(-1, n_heads, head_dim).transpose(1, 0, 2)  # [h, n, d]
        s = np.matmul(qh, K.transpose(0, 2, 1)) * scale                                  # [h, n, T]
        vis = np.arange(C)[None, :] < np.asarray(prefix_len[r0:r1])[:, None]              # [n, C]
        if has_tree:
            vis = np.concatenate([vis, np.asarray(tree_vis[r0:r1], bool)], axis=1)
        s = np.where(vis[None], s, -np.inf)
        p = softmax(s)
        out[r0:r1] = np.matmul(p, V).transpose(1, 0, 2).reshape(r1 - r0, H)
    return out


def decoder_layer(model: OracleModel, lw: dict, x, pos, cache_k, cache_v,
                  prefix_len, tree_k_prev, tree_v_prev, tree_vis):
    """One pre-norm LLaMA decoder layer over the rows x (R1).

    The rows' own keys/values are appended after tree_k_prev/tree_v_prev to
    form the tree key set that tree_vis indexes. Returns (x_out, k, v) where k
    (after RoPE) and v are the rows' own keys and values.
    """
    cfg = model.cfg
    m = model.mat
    xn = rms_norm(x, lw["attn_norm"], cfg.rms_eps)
    q = xn @ m(lw["wq"]).T
    k = xn @ m(lw["wk"]).T
    v = xn @ m(lw["wv"]).T
    q = rope(q, pos, cfg.n_heads, cfg.head_dim, cfg.rope_base)
    k = rope(k, pos, cfg.n_heads, cfg.head_dim, cfg.rope_base)
    H = cfg.hidden
    tk_prev = np.zeros((0, H)) if tree_k_prev is None else tree_k_prev
    tv_prev = np.zeros((0, H)) if tree_v_prev is None else tree_v_prev
    tk = np.concatenate([tk_prev, k], axis=0)
    tv = np.concatenate([tv_prev, v], axis=0)
    a = attend(q, cache_k, cache_v, prefix_len, tk, tv, tree_vis,
               cfg.n_heads, cfg.head_dim)
    x = np.asarray(x, F64) + a @ m(lw["wo"]).T
    xn2 = rms_norm(x, lw["mlp_norm"], cfg.rms_eps)
    g = xn2 @ m(lw["w_gate"]).T
    u = xn2 @ m(lw["w_up"]).T
    x = x + (silu(g) * u) @ m(lw["w_down"]).T
    return x, k, v


def target_forward(model: OracleModel, emb, pos, caches, prefix_len,
                   tree_prev, tree_vis):
    """Target decoder stack over the rows emb (Sec. 3.1).

    caches[l] = (K, V) cache rows of layer l; tree_prev[l] = (K, V) of tree
    rows computed earlier in the same pass structure (or None). Returns
    (h, new_kv) with h the final-normed features (R2) and new_kv[l] = (k, v).
    """
    cfg = model.cfg
    x = np.asarray(emb, F64)
    new_kv = []
    for l, lw in enumerate(model.w["layers"]):
        ck, cv = caches[l]
        tkp, tvp = (None, None) if tree_prev is None else tree_prev[l]
        x, k, v = decoder_layer(model, lw, x, pos, ck, cv, prefix_len,
                                tkp, tvp, tree_vis)
        new_kv.append((k, v))
    h = rms_norm(x, model.w["final_norm"], cfg.rms_eps)
    return h, new_kv


def lm_logits(model: OracleModel, h) -> np.ndarray:
    """LM head: logits = lm_head @ h for each row (Sec. 3.1, Eq. 5)."""
    return np.asarray(h, F64) @ model.mat(model.w["lm_head"]).T


def embed_prompt(model: OracleModel, ids, vis) -> np.ndarray:
    """Interleaved multimodal input sequence (Eq. 1-3).

    ids[i] >= 0 is a text token (row of E_t); ids[i] == -1 takes the next row of
    the projected visual embeddings in order.
    """
    E = model.w["embed"]
    rows = []
    j = 0
    for t in ids:
        if t >= 0:
            rows.append(np.asarray(E[t], F64))
        else:
            rows.append(np.asarray(vis[j], F64))
            j += 1
    return np.stack(rows)


def draft_fc(model: OracleModel, h, e) -> np.ndarray:
    """f_down(Concat(h, e)) of Eq. 4: a [H, 2H] projection of [h ; e]."""
    cat = np.concatenate([np.asarray(h, F64), np.asarray(e, F64)], axis=-1)
    return cat @ model.mat(model.w["draft_fc"]).T


def decoupled_draft_inputs(model: OracleModel, ids, emb, h) -> np.ndarray:
    """Draft inputs f_{x_i} for the prefix positions i = 0 .. L-2 (Eq. 7).

    Text position i: f_down(Concat(h_{x_i}, e_{x_{i+1}})), where e_{x_{i+1}} is
    whatever embedding the next position carries (text or visual).
    Visual position i, by the model's draft-input strategy (R8): the raw
    embedding e_{x_i} (MSD, Eq. 7), the same concatenation as a text position
    (Baseline, Sec. 3.3), or the target feature h_{x_i} (Visual Feature).
    """
    mode = model.cfg.draft_input
    if mode not in DRAFT_INPUTS:
        raise ValueError(f"unknown draft input strategy {mode!r}")
    L = len(ids)
    rows = []
    for i in range(L - 1):
        if ids[i] >= 0 or mode == "concat":
            rows.append(draft_fc(model, h[i:i + 1], emb[i + 1:i + 2])[0])
        elif mode == "embedding":
            rows.append(np.asarray(emb[i], F64))
        else:
            rows.append(np.asarray(h[i], F64))
    return np.stack(rows) if rows else np.zeros((0, model.cfg.hidden))


def draft_forward(model: OracleModel, f, pos, cache_k, cache_v, prefix_len,
                  tree_k_prev, tree_v_prev, tree_vis):
    """The one-layer draft model M_q over rows f (Eq. 4). Returns (h_hat, k, v)."""
    return decoder_layer(model, model.w["draft"], f, pos, cache_k, cache_v,
                         prefix_len, tree_k_prev, tree_v_prev, tree_vis)


def causal_vis(R: int) -> np.ndarray:
    return np.tril(np.ones((R, R), dtype=bool))


# ----------------------------------------------------------------------------
# Request state
# ----------------------------------------------------------------------------

@dataclass
class RequestState:
    L: int                       # committed target length (root sits at L)
    K: list                      # per layer [L, H] (post-RoPE)
    V: list
    dK: np.ndarray               # draft cache [L - P, H]
    dV: np.ndarray
    pend_h: np.ndarray           # [P, H] target features of pending positions
    pend_next: np.ndarray        # [P] the token that follows each pending position
    root: int
    emitted: list = field(default_factory=list)


def prefill(model: OracleModel, ids, vis) -> RequestState:
    """Target forward over the prompt, root token, and draft cache (Sec. 3, Eq. 7).

    The draft cache covers positions 0 .. L-2; position L-1 is pending because
    its input needs the embedding of the root token x_L.
    """
    cfg = model.cfg
    ids = np.asarray(ids, np.int64)
    L = ids.shape[0]
    if L < 1 or ids[-1] < 0:
        raise ValueError("a prefix must be non-empty and end with a text token")
    emb = embed_prompt(model, ids, vis)
    pos = np.arange(L)
    empty = np.zeros((0, cfg.hidden))
    caches = [(empty, empty)] * cfg.n_layers
    h, kv = target_forward(model, emb, pos, caches, np.zeros(L, np.int64),
                           None, causal_vis(L))
    root = argmax_lowest(lm_logits(model, h[L - 1:L])[0])
    f = decoupled_draft_inputs(model, ids, emb, h)
    _, dk, dv = draft_forward(model, f, np.arange(L - 1), empty, empty,
                              np.zeros(L - 1, np.int64), None, None,
                              causal_vis(L - 1))
    return RequestState(L=L, K=[k for k, _ in kv], V=[v for _, v in kv],
                        dK=dk, dV=dv, pend_h=h[L - 1:L].copy(),
                        pend_next=np.array([root]), root=root, emitted=[root])


# ----------------------------------------------------------------------------
# Draft tree (Sec. 3.2, tree drafting; reading R3)
# ----------------------------------------------------------------------------

class TreeBuilder:
    """Incremental draft-tree construction.

    Candidates are created in order (depth, rank of the expanded parent,
    child rank); that order is the creation index. Scores are float32 sums of
    log-probabilities along the path: the score of a child is
    float32(score(parent) + logp(child)), the same single float32 addition the
    kernel performs, so that ranking decisions are taken in one precision.
    """

    def __init__(self, k: int):
        self.k = k
        self.token, self.parent, self.depth, self.score = [], [], [], []

    def add_children(self, parent: int, ids, logp):
        """parent = -1 for the root; ids/logp = the parent's top-k."""
        base = np.float32(0.0) if parent < 0 else self.score[parent]
        d = 1 if parent < 0 else self.depth[parent] + 1
        for t, lp in zip(ids, logp):
            self.token.append(int(t))
            self.parent.append(int(parent))
            self.depth.append(d)
            s = np.float32(lp) if parent < 0 else np.float32(base + np.float32(lp))
            self.score.append(s)

    def rank_key(self, c):
        return (-float(self.score[c]), self.depth[c], c)

    def frontier(self, depth: int) -> list:
        """The k best candidates at the given depth, best first."""
        cands = [c for c in range(len(self.token)) if self.depth[c] == depth]
        cands.sort(key=self.rank_key)
        return cands[:self.k]

    def finalize(self, n_nodes: int) -> "Tree":
        """Keep the N-1 best candidates; tree index = 1 + rank, root = 0."""
        order = sorted(range(len(self.token)), key=self.rank_key)[:n_nodes - 1]
        index = {c: i + 1 for i, c in enumerate(order)}
        tokens = np.zeros(n_nodes, np.int64)
        parent = np.full(n_nodes, -1, np.int64)
        depth = np.zeros(n_nodes, np.int64)
        for c, i in index.items():
            tokens[i] = self.token[c]
            depth[i] = self.depth[c]
            p = self.parent[c]
            if p >= 0 and p not in index:
                raise AssertionError("selected set is not ancestor-closed")
            parent[i] = 0 if p < 0 else index[p]
        return Tree(tokens=tokens, parent=parent, depth=depth)


@dataclass
class Tree:
    tokens: np.ndarray      # [N]; tokens[0] is the root token (set by caller)
    parent: np.ndarray      # [N]; parent[0] = -1
    depth: np.ndarray       # [N]

    @property
    def n(self) -> int:
        return int(self.tokens.shape[0])

    def ancestors_or_self(self) -> np.ndarray:
        """vis[i, j] = j is an ancestor of i or j == i (walk of parent links)."""
        N = self.n
        vis = np.zeros((N, N), dtype=bool)
        for i in range(N):
            j = i
            while j >= 0:
                vis[i, j] = True
                j = int(self.parent[j])
        return vis

    def mask_words(self) -> np.ndarray:
        """The same relation as uint64 words: bit j%64 of word j//64 of row i."""
        vis = self.ancestors_or_self()
        N = self.n
        W = (N + 63) // 64
        words = np.zeros((N, W), np.uint64)
        for i in range(N):
            for j in np.flatnonzero(vis[i]):
                words[i, j // 64] |= np.uint64(1) << np.uint64(j % 64)
        return words


@dataclass
class DraftRecord:
    """What each draft pass produced (for comparison with the kernels)."""
    logits: list = field(default_factory=list)     # per pass [rows, V] float64
    rows: list = field(default_factory=list)       # per pass: candidate ids expanded
    topk: list = field(default_factory=list)       # per pass [rows, k] ids
    logp: list = field(default_factory=list)       # per pass [rows, k] float32


def draft_catch_up(model: OracleModel, st: RequestState):
    """Pass 1: draft rows for the pending positions, root slot last (Eq. 4, 7).

    Pending positions hold generated (text) tokens, so each takes
    f_down(Concat(h, e_next)). The rows attend causally to the draft cache and
    to each other, and are then committed to the draft cache.
    Returns h_hat of the root slot (draft position L-1).
    """
    cfg = model.cfg
    P = st.pend_h.shape[0]
    e_next = np.asarray(model.w["embed"][st.pend_next], F64)
    f = draft_fc(model, st.pend_h, e_next)
    c0 = st.L - P
    pos = np.arange(c0, st.L)
    hh, k, v = draft_forward(model, f, pos, st.dK, st.dV,
                             np.full(P, c0, np.int64), None, None, causal_vis(P))
    st.dK = np.concatenate([st.dK, k], axis=0)
    st.dV = np.concatenate([st.dV, v], axis=0)
    return hh[P - 1]


def draft_pass_logits(model: OracleModel, h_hat_rows) -> np.ndarray:
    """q = LM head applied to the draft features (Eq. 5), as logits."""
    return lm_logits(model, h_hat_rows)


def draft_tree(model: OracleModel, st: RequestState, record: DraftRecord = None,
               forced_logp=None) -> Tree:
    """Draft a tree of depth D with top-k expansion (Sec. 3.2, reading R3).

    forced_logp, if given, is a function (pass, rows) -> (topk ids, float32
    logp) that replaces the oracle's own top-k decision; the comparison tests
    use it to follow the kernels' decisions while the oracle still computes
    every feature and logit itself.
    """
    cfg = model.cfg
    k, D, L = cfg.topk, cfg.tree_depth, st.L
    h_root = draft_catch_up(model, st)

    def decide(pass_idx, rows_logits):
        if forced_logp is not None:
            return forced_logp(pass_idx, rows_logits)
        ids, lps = [], []
        for z in rows_logits:
            lp = log_softmax(z)
            t = topk_ids(z, k)
            ids.append(t)
            lps.append(lp[t].astype(np.float32))
        return np.array(ids), np.array(lps)

    tb = TreeBuilder(k)
    z1 = draft_pass_logits(model, h_root[None, :])
    ids, lps = decide(0, z1)
    tb.add_children(-1, ids[0], lps[0])
    if record is not None:
        record.logits.append(z1); record.rows.append([-1])
        record.topk.append(ids); record.logp.append(lps)

    # Draft rows of expanded candidates: their K/V and h_hat.
    tree_k = np.zeros((0, cfg.hidden)); tree_v = np.zeros((0, cfg.hidden))
    row_of = {}             # candidate -> draft tree row
    h_hat = {}              # candidate -> draft output feature
    for d in range(2, D + 1):
        fr = tb.frontier(d - 1)
        parent_h = np.stack([h_root if tb.parent[c] < 0 else h_hat[tb.parent[c]]
                             for c in fr])
        e_tok = np.asarray(model.w["embed"][[tb.token[c] for c in fr]], F64)
        f = draft_fc(model, parent_h, e_tok)
        pos = np.array([L - 1 + tb.depth[c] for c in fr])
        T0 = tree_k.shape[0]
        R = len(fr)
        vis = np.zeros((R, T0 + R), dtype=bool)
        for r, c in enumerate(fr):
            a = tb.parent[c]
            while a >= 0:
                vis[r, row_of[a]] = True
                a = tb.parent[a]
            vis[r, T0 + r] = True
        hh, kk, vv = draft_forward(model, f, pos, st.dK, st.dV,
                                   np.full(R, L, np.int64), tree_k, tree_v, vis)
        tree_k = np.concatenate([tree_k, kk]); tree_v = np.concatenate([tree_v, vv])
        for r, c in enumerate(fr):
            row_of[c] = T0 + r
            h_hat[c] = hh[r]
        z = draft_pass_logits(model, hh)
        ids, lps = decide(d - 1, z)
        for r, c in enumerate(fr):
            tb.add_children(c, ids[r], lps[r])
        if record is not None:
            record.logits.append(z); record.rows.append(fr)
            record.topk.append(ids); record.logp.append(lps)

    tree = tb.finalize(cfg.tree_nodes)
    tree.tokens[0] = st.root
    return tree


# ----------------------------------------------------------------------------
# Verify, accept, compact (Sec. 3.2, Eq. 6 at T = 0)
# ----------------------------------------------------------------------------

@dataclass
class VerifyResult:
    h: np.ndarray           # [N, H]
    logits: np.ndarray      # [N, V]
    argmax: np.ndarray      # [N]
    kv: list                # per layer (k [N, H], v [N, H])


def verify(model: OracleModel, st: RequestState, tree: Tree) -> VerifyResult:
    """Target forward over all tree tokens in one pass (Sec. 3.2).

    Node i sits at position L + depth(i) and sees the whole prefix [0, L) and
    its ancestors and itself.
    """
    cfg = model.cfg
    N = tree.n
    emb = np.asarray(model.w["embed"][tree.tokens], F64)
    pos = st.L + tree.depth
    caches = list(zip(st.K, st.V))
    h, kv = target_forward(model, emb, pos, caches, np.full(N, st.L, np.int64),
                           None, tree.ancestors_or_self())
    z = lm_logits(model, h)
    g = np.array([argmax_lowest(r) for r in z], np.int64)
    return VerifyResult(h=h, logits=z, argmax=g, kv=kv)


def accept(tree: Tree, argmax) -> tuple:
    """Greedy acceptance (Eq. 6 at T = 0).

    From the root, move to the child whose token equals the target argmax at
    the current node; stop when there is none. The next token after the last
    accepted node is the target argmax there (the residual rule at T = 0 and the
    bonus token). Returns (path, a, bonus) with path[0] = 0 (the root).
    """
    path = [0]
    cur = 0
    while True:
        nxt = [c for c in range(tree.n)
               if tree.parent[c] == cur and tree.tokens[c] == argmax[cur]]
        if not nxt:
            break
        cur = nxt[0]
        path.append(cur)
    return np.array(path, np.int64), len(path) - 1, int(argmax[cur])


def sample_index(p: np.ndarray, u: float, removed=()) -> int:
    """Inverse-CDF draw from p restricted to the tokens not in `removed`:
    the smallest token id t whose cumulative mass (token-id order, removed
    tokens skipped) exceeds u times the remaining mass (R7)."""
    q = np.asarray(p, F64).copy()
    for x in removed:
        q[x] = 0.0
    target = float(u) * q.sum()
    c = np.cumsum(q)
    hit = np.flatnonzero(c > target)
    if hit.size:
        return int(hit[0])
    return int(np.flatnonzero(q > 0)[-1])           # rounding at the very top


def accept_sample(tree: Tree, logits, temperature: float, u, k: int) -> tuple:
    """Speculative sampling over the tree at temperature T > 0 (Sec. 3.2,
    Eq. 6 and the adjusted distribution after it; reading R7).

    From the root: p = softmax(logits[node] / T); each child x in tree order is
    accepted with probability p_adj(x) (a draw u < p_adj(x)); a rejection
    removes x from p_adj. An accepted child becomes the node and the walk goes
    on; when a node's children are all rejected, or it has none, the next
    token is drawn from p_adj and the walk ends. Returns (path, a, bonus).
    """
    path = [0]
    cur = 0
    d = 0
    while True:
        z = np.asarray(logits[cur], F64) / float(temperature)
        p = softmax(z)
        children = [c for c in range(tree.n) if tree.parent[c] == cur]
        removed = []
        nxt = None
        for j, c in enumerate(children):
            x = int(tree.tokens[c])
            rest = 1.0 - sum(p[r] for r in removed)
            px = 0.0 if x in removed else p[x]
            if u[d][j] * rest < px:
                nxt = c
                break
            if x not in removed:
                removed.append(x)
        if nxt is None:
            return np.array(path, np.int64), len(path) - 1, sample_index(p, u[d][k], removed)
        path.append(nxt)
        cur = nxt
        d += 1


def compact(st: RequestState, tree: Tree, vr: VerifyResult, path, bonus):
    """Keep the accepted nodes' K/V at positions L .. L+a, drop the rest.

    The accepted nodes' target features become the draft's pending rows, each
    paired with the token that follows it.
    """
    a = len(path) - 1
    for l in range(len(st.K)):
        k, v = vr.kv[l]
        st.K[l] = np.concatenate([st.K[l], k[path]], axis=0)
        st.V[l] = np.concatenate([st.V[l], v[path]], axis=0)
    nxt = [int(tree.tokens[path[j + 1]]) for j in range(a)] + [bonus]
    st.pend_h = vr.h[path].copy()
    st.pend_next = np.array(nxt, np.int64)
    st.L += a + 1
    st.root = bonus
    st.emitted.extend([int(tree.tokens[p]) for p in path[1:]] + [bonus])


def spec_step(model: OracleModel, st: RequestState, tree: Tree = None):
    """One draft -> verify -> accept -> compact step. A caller-planted tree
    skips drafting (the draft cache is still caught up)."""
    if tree is None:
        tree = draft_tree(model, st)
    else:
        draft_catch_up(model, st)
        tree.tokens[0] = st.root
    vr = verify(model, st, tree)
    path, a, bonus = accept(tree, vr.argmax)
    compact(st, tree, vr, path, bonus)
    return tree, vr, path, a, bonus


# ----------------------------------------------------------------------------
# Plain greedy autoregressive decoding of the target (the lossless reference)
# ----------------------------------------------------------------------------

def greedy_ar(model: OracleModel, ids, vis, n_tokens: int) -> list:
    """Vanilla greedy decoding: one target forward per token, with a KV cache."""
    cfg = model.cfg
    ids = np.asarray(ids, np.int64)
    L = ids.shape[0]
    emb = embed_prompt(model, ids, vis)
    empty = np.zeros((0, cfg.hidden))
    h, kv = target_forward(model, emb, np.arange(L),
                           [(empty, empty)] * cfg.n_layers,
                           np.zeros(L, np.int64), None, causal_vis(L))
    K = [k for k, _ in kv]; V = [v for _, v in kv]
    tok = argmax_lowest(lm_logits(model, h[L - 1:L])[0])
    out = [tok]
    pos = L
    while len(out) < n_tokens:
        e = np.asarray(model.w["embed"][[tok]], F64)
        h, kv = target_forward(model, e, np.array([pos]), list(zip(K, V)),
                               np.array([pos]), None, np.ones((1, 1), bool))
        for l in range(cfg.n_layers):
            K[l] = np.concatenate([K[l], kv[l][0]]); V[l] = np.concatenate([V[l], kv[l][1]])
        tok = argmax_lowest(lm_logits(model, h)[0])
        out.append(tok)
        pos += 1
    return out
