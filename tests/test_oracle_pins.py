"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a library
routine, a closed form, an invariant, or brute force on a tiny case. The set is
chosen so that a plausible slip in the oracle (a dropped term, a wrong sign or
index, a transposed operand, a wrong position) fails at least one of them.
"""
import cmath

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import synth
from tests.oracle_support import oracle_model, prompt_numpy, tiny

pytestmark = pytest.mark.filterwarnings("ignore::UserWarning")


# ----------------------------------------------------------------------------
# Elementary operations
# ----------------------------------------------------------------------------

def test_rms_norm_matches_torch_library():
    rng = np.random.default_rng(0)
    x = rng.normal(size=(5, 48)) * 3
    g = rng.normal(size=48)
    ref = F.rms_norm(torch.from_numpy(x), (48,), torch.from_numpy(g), eps=1e-6).numpy()
    np.testing.assert_allclose(O.rms_norm(x, g, 1e-6), ref, rtol=1e-12, atol=1e-12)


def test_rms_norm_unit_rms_and_scale_invariance():
    rng = np.random.default_rng(1)
    x = rng.normal(size=(3, 64))
    y = O.rms_norm(x, np.ones(64), 0.0)
    np.testing.assert_allclose(np.mean(y * y, axis=1), 1.0, rtol=1e-12)
    np.testing.assert_allclose(O.rms_norm(7.5 * x, np.ones(64), 0.0), y, rtol=1e-12)


def test_rope_equals_complex_rotation():
    """Rotate-half RoPE == multiplying (x_i + i*x_{i+hd/2}) by exp(i*p*theta_i)."""
    rng = np.random.default_rng(2)
    nh, hd, base = 2, 8, 10000.0
    x = rng.normal(size=(3, nh * hd))
    pos = np.array([0, 5, 1234])
    y = O.rope(x, pos, nh, hd, base)
    for r in range(3):
        for h in range(nh):
            for i in range(hd // 2):
                a, b = x[r, h * hd + i], x[r, h * hd + i + hd // 2]
                theta = base ** (-2.0 * i / hd)
                z = complex(a, b) * cmath.exp(1j * pos[r] * theta)
                assert abs(y[r, h * hd + i] - z.real) < 1e-9
                assert abs(y[r, h * hd + i + hd // 2] - z.imag) < 1e-9


def test_rope_depends_on_relative_position_only():
    rng = np.random.default_rng(3)
    nh, hd = 1, 16
    q, k = rng.normal(size=(1, hd)), rng.normal(size=(1, hd))
    d1 = O.rope(q, np.array([10]), nh, hd, 1e4) @ O.rope(k, np.array([3]), nh, hd, 1e4).T
    d2 = O.rope(q, np.array([107]), nh, hd, 1e4) @ O.rope(k, np.array([100]), nh, hd, 1e4).T
    np.testing.assert_allclose(d1, d2, rtol=1e-10)
    np.testing.assert_allclose(O.rope(q, np.array([0]), nh, hd, 1e4), q, rtol=0, atol=0)


def test_attend_matches_sdpa_causal():
    rng = np.random.default_rng(4)
    R, nh, hd = 7, 3, 16
    q, k, v = (rng.normal(size=(R, nh * hd)) for _ in range(3))
    out = O.attend(q, np.zeros((0, nh * hd)), np.zeros((0, nh * hd)), np.zeros(R, int),
                   k, v, O.causal_vis(R), nh, hd)
    t = lambda a: torch.from_numpy(a.reshape(R, nh, hd).transpose(1, 0, 2).copy())
    ref = F.scaled_dot_product_attention(t(q), t(k), t(v), is_causal=True)
    np.testing.assert_allclose(out, ref.numpy().transpose(1, 0, 2).reshape(R, -1),
                               rtol=1e-10, atol=1e-12)


def test_attend_prefix_and_tree_split_is_order_free():
    """Seeing prefix rows via the cache or via the tree part gives the same result."""
    rng = np.random.default_rng(5)
    nh, hd, P = 2, 8, 6
    q = rng.normal(size=(1, nh * hd))
    k, v = rng.normal(size=(P, nh * hd)), rng.normal(size=(P, nh * hd))
    a = O.attend(q, k, v, np.array([P]), np.zeros((0, nh * hd)), None, None, nh, hd)
    b = O.attend(q, k[:2], v[:2], np.array([2]), k[2:], v[2:], np.ones((1, P - 2), bool), nh, hd)
    np.testing.assert_allclose(a, b, rtol=1e-12)


def test_topk_and_argmax_tie_rules_match_stable_sort():
    rng = np.random.default_rng(6)
    for _ in range(20):
        v = rng.integers(0, 5, size=30).astype(np.float32)
        np.testing.assert_array_equal(O.topk_ids(v, 7), np.argsort(-v, kind="stable")[:7])
        assert O.argmax_lowest(v) == int(np.argmax(v))   # numpy returns the first maximum


def test_log_softmax_matches_torch():
    rng = np.random.default_rng(7)
    z = rng.normal(size=(3, 100)) * 4
    np.testing.assert_allclose(O.log_softmax(z), torch.log_softmax(torch.from_numpy(z), -1).numpy(),
                               rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------
# Whole target forward vs an independently written library implementation
# ----------------------------------------------------------------------------

def _torch_llama_forward(wl, w, emb):
    """LLaMA-style causal forward written with torch library ops (float64):
    F.rms_norm, complex-number RoPE, F.scaled_dot_product_attention, F.silu."""
    d = lambda t: t.to(torch.float64)
    nh, hd = wl.n_heads, wl.head_dim
    L = emb.shape[0]
    x = torch.from_numpy(emb).to(torch.float64)
    half = hd // 2
    theta = wl.rope_base ** (-torch.arange(half, dtype=torch.float64) * 2 / hd)
    rot = torch.polar(torch.ones(L, half, dtype=torch.float64),
                      torch.arange(L, dtype=torch.float64)[:, None] * theta[None, :])

    def rope_c(t):
        t = t.view(L, nh, hd)
        c = torch.complex(t[..., :half], t[..., half:]) * rot[:, None, :]
        return torch.cat([c.real, c.imag], dim=-1)

    for lw in w["layers"]:
        xn = F.rms_norm(x, (wl.hidden,), d(lw["attn_norm"]), eps=wl.rms_eps)
        q, k, v = xn @ d(lw["wq"]).T, xn @ d(lw["wk"]).T, xn @ d(lw["wv"]).T
        q, k = rope_c(q).transpose(0, 1), rope_c(k).transpose(0, 1)
        v = v.view(L, nh, hd).transpose(0, 1)
        a = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        x = x + a.transpose(0, 1).reshape(L, -1) @ d(lw["wo"]).T
        xn = F.rms_norm(x, (wl.hidden,), d(lw["mlp_norm"]), eps=wl.rms_eps)
        x = x + (F.silu(xn @ d(lw["w_gate"]).T) * (xn @ d(lw["w_up"]).T)) @ d(lw["w_down"]).T
    h = F.rms_norm(x, (wl.hidden,), d(w["final_norm"]), eps=wl.rms_eps)
    return h.numpy(), (h @ d(w["lm_head"]).T).numpy()


@pytest.fixture(scope="module")
def tiny_setup():
    wl = tiny(n_layers=2)
    w = synth.make_weights(wl)
    m = oracle_model(wl, w)
    ids, vis = prompt_numpy(synth.make_prompts(wl)[0])
    return wl, w, m, ids, vis


def test_target_forward_matches_library_llama(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    emb = O.embed_prompt(m, ids, vis)
    L = len(ids)
    e0 = np.zeros((0, wl.hidden))
    h, _ = O.target_forward(m, emb, np.arange(L), [(e0, e0)] * wl.n_layers,
                            np.zeros(L, int), None, O.causal_vis(L))
    h_ref, z_ref = _torch_llama_forward(wl, w, emb)
    np.testing.assert_allclose(h, h_ref, rtol=1e-9, atol=1e-9)
    np.testing.assert_allclose(O.lm_logits(m, h), z_ref, rtol=1e-9, atol=1e-9)


def test_embed_prompt_interleaves_eq3(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    ids2 = np.array([5, 6, -1, -1, 7, -1, 9])
    vis2 = np.arange(3 * wl.hidden, dtype=np.float32).reshape(3, wl.hidden)
    e = O.embed_prompt(m, ids2, vis2)
    E = m.w["embed"]
    for i, j in [(0, 5), (1, 6), (4, 7), (6, 9)]:
        np.testing.assert_array_equal(e[i], E[j])
    for i, r in [(2, 0), (3, 1), (5, 2)]:
        np.testing.assert_array_equal(e[i], vis2[r])


# ----------------------------------------------------------------------------
# Tree attention: brute force against causal sequences
# ----------------------------------------------------------------------------

def _causal_last_logits(m, ids_prompt, vis, extra_tokens):
    """Plain causal forward of prompt + extra text tokens; logits of every
    position after the prompt (brute force)."""
    ids = np.concatenate([ids_prompt, np.asarray(extra_tokens, np.int64)])
    emb = O.embed_prompt(m, ids, vis)
    L = len(ids)
    e0 = np.zeros((0, m.cfg.hidden))
    h, kv = O.target_forward(m, emb, np.arange(L), [(e0, e0)] * m.cfg.n_layers,
                             np.zeros(L, int), None, O.causal_vis(L))
    return O.lm_logits(m, h), kv


def test_tree_verify_equals_causal_path_bruteforce(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    tree = O.draft_tree(m, st)
    vr = O.verify(m, st, tree)
    L = st.L
    for i in range(tree.n):
        chain = []
        j = i
        while j >= 0:
            chain.append(int(tree.tokens[j])); j = int(tree.parent[j])
        chain = chain[::-1]        # root .. i
        z, _ = _causal_last_logits(m, ids, vis, chain)
        np.testing.assert_allclose(vr.logits[i], z[L + len(chain) - 1], rtol=1e-9, atol=1e-9)


def test_single_node_tree_is_one_ar_step(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    t = O.Tree(tokens=np.array([st.root]), parent=np.array([-1]), depth=np.array([0]))
    vr = O.verify(m, st, t)
    ar = O.greedy_ar(m, ids, vis, 2)
    assert ar[0] == st.root and vr.argmax[0] == ar[1]


def test_chain_tree_equals_causal_prefill(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    toks = np.array([st.root, 3, 17, 99, 5])
    t = O.Tree(tokens=toks, parent=np.arange(-1, 4), depth=np.arange(5))
    vr = O.verify(m, st, t)
    z, _ = _causal_last_logits(m, ids, vis, toks)
    np.testing.assert_allclose(vr.logits, z[st.L:], rtol=1e-9, atol=1e-9)


def test_causality_non_ancestor_rows_bit_identical(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    tree = O.draft_tree(m, st)
    vr = O.verify(m, st, tree)
    vis_m = tree.ancestors_or_self()
    j = tree.n - 1                      # a leaf-or-deep node
    t2 = O.Tree(tokens=tree.tokens.copy(), parent=tree.parent, depth=tree.depth)
    t2.tokens[j] = (t2.tokens[j] + 1) % wl.vocab
    vr2 = O.verify(m, st, t2)
    for i in range(tree.n):
        if vis_m[i, j]:
            assert np.max(np.abs(vr2.logits[i] - vr.logits[i])) > 0
        else:
            np.testing.assert_array_equal(vr2.logits[i], vr.logits[i])


def test_prefix_perturbation_changes_every_row(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    tree = O.draft_tree(m, st)
    vr = O.verify(m, st, tree)
    ids2 = ids.copy(); ids2[-2] = (ids2[-2] + 1) % wl.vocab
    st2 = O.prefill(m, ids2, vis)
    vr2 = O.verify(m, st2, tree)
    assert all(np.max(np.abs(vr2.logits[i] - vr.logits[i])) > 0 for i in range(tree.n))


# ----------------------------------------------------------------------------
# Decoupled draft inputs (Eq. 7)
# ----------------------------------------------------------------------------

def test_decoupled_inputs_follow_eq7(tiny_setup):
    wl, w, m, _, _ = tiny_setup
    H = wl.hidden
    rng = np.random.default_rng(8)
    ids = np.array([4, 8, -1, -1, -1, 12, 13, -1, 20])
    vis = rng.normal(size=(4, H)) * 0.5
    emb = O.embed_prompt(m, ids, vis)
    h = rng.normal(size=(len(ids), H))
    f = O.decoupled_draft_inputs(m, ids, emb, h)
    Wfc = np.asarray(m.w["draft_fc"], np.float64)
    assert f.shape == (len(ids) - 1, H)
    for i in range(len(ids) - 1):
        if ids[i] < 0:
            np.testing.assert_array_equal(f[i], emb[i])       # raw visual embedding
        else:                                                 # W[:, :H] h_i + W[:, H:] e_{i+1}
            np.testing.assert_allclose(f[i], Wfc[:, :H] @ h[i] + Wfc[:, H:] @ emb[i + 1],
                                       rtol=1e-10, atol=1e-12)
    # changing visual row 1 (position 3) moves f only at 3 (itself, visual) and 2
    # (visual: unaffected) -> only position 3; changing visual row 3 (position 7)
    # moves 7 and the text position 6 before it.
    vis2 = vis.copy(); vis2[3] += 1.0
    f2 = O.decoupled_draft_inputs(m, ids, O.embed_prompt(m, ids, vis2), h)
    changed = [i for i in range(len(f)) if np.any(f2[i] != f[i])]
    assert changed == [6, 7]
    vis3 = vis.copy(); vis3[1] += 1.0
    f3 = O.decoupled_draft_inputs(m, ids, O.embed_prompt(m, ids, vis3), h)
    assert [i for i in range(len(f)) if np.any(f3[i] != f[i])] == [3]


def _variant(m, mode):
    import dataclasses
    return O.OracleModel(dataclasses.replace(m.cfg, draft_input=mode), m.w)


@pytest.mark.parametrize("mode,moved_by_pos3,moved_by_pos7", [
    ("embedding", [3], [6, 7]),      # MSD: a visual row is its own embedding
    ("concat", [2], [6]),            # Baseline: a row carries the NEXT position's embedding
    ("feature", [], [6]),            # Visual Feature: a visual row is h, no embedding at all
])
def test_draft_input_strategies_dependency_structure(tiny_setup, mode, moved_by_pos3, moved_by_pos7):
    """The three visual-input strategies of the paper's ablation (Sec. 5.3),
    told apart by which draft rows a visual embedding reaches (h held fixed):
    ids 4 8 V V V 12 13 V 20 with visual rows at positions 2, 3, 4 and 7."""
    wl, w, m, _, _ = tiny_setup
    mv = _variant(m, mode)
    H = wl.hidden
    rng = np.random.default_rng(8)
    ids = np.array([4, 8, -1, -1, -1, 12, 13, -1, 20])
    vis = rng.normal(size=(4, H)) * 0.5
    h = rng.normal(size=(len(ids), H))
    f = O.decoupled_draft_inputs(mv, ids, O.embed_prompt(mv, ids, vis), h)
    for row, expect in ((1, moved_by_pos3), (3, moved_by_pos7)):
        v2 = vis.copy(); v2[row] += 1.0
        f2 = O.decoupled_draft_inputs(mv, ids, O.embed_prompt(mv, ids, v2), h)
        assert [i for i in range(len(f)) if np.any(f2[i] != f[i])] == expect, (mode, row)


def test_draft_input_strategies_rows(tiny_setup):
    """Visual Feature rows are the features bit-exactly; Baseline rows are the
    split-matrix form W[:, :H] h_i + W[:, H:] e_{i+1} at every position; text
    rows are the same under all three strategies."""
    wl, w, m, _, _ = tiny_setup
    H = wl.hidden
    rng = np.random.default_rng(9)
    ids = np.array([3, -1, -1, 7, -1, 9])
    vis = rng.normal(size=(3, H)) * 0.5
    emb = O.embed_prompt(m, ids, vis)
    h = rng.normal(size=(len(ids), H))
    Wfc = np.asarray(m.w["draft_fc"], np.float64)
    fe = O.decoupled_draft_inputs(_variant(m, "embedding"), ids, emb, h)
    fc = O.decoupled_draft_inputs(_variant(m, "concat"), ids, emb, h)
    ff = O.decoupled_draft_inputs(_variant(m, "feature"), ids, emb, h)
    for i in range(len(ids) - 1):
        np.testing.assert_allclose(fc[i], Wfc[:, :H] @ h[i] + Wfc[:, H:] @ emb[i + 1], rtol=1e-10, atol=1e-12)
        if ids[i] < 0:
            np.testing.assert_array_equal(ff[i], h[i])
            np.testing.assert_array_equal(fe[i], emb[i])
        else:
            np.testing.assert_array_equal(fe[i], fc[i])
            np.testing.assert_array_equal(ff[i], fc[i])
    with pytest.raises(ValueError):
        O.decoupled_draft_inputs(_variant(m, "bogus"), ids, emb, h)


def test_draft_input_strategies_agree_without_visual_tokens(tiny_setup):
    """On a text-only prompt the three strategies build the same draft cache."""
    wl, w, m, _, _ = tiny_setup
    ids = np.arange(5, 25)
    sts = [O.prefill(_variant(m, mode), ids, np.zeros((0, wl.hidden))) for mode in O.DRAFT_INPUTS]
    for st in sts[1:]:
        np.testing.assert_array_equal(st.dK, sts[0].dK)
        np.testing.assert_array_equal(st.dV, sts[0].dV)


def test_draft_node_equals_causal_draft_chain(tiny_setup):
    """A depth-d draft row equals the draft layer run causally over the committed
    draft cache and the chain of its ancestors' inputs at consecutive positions."""
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    rec = O.DraftRecord()
    st_copy = O.RequestState(**{k: (v.copy() if isinstance(v, np.ndarray) else
                                    (list(v) if isinstance(v, list) else v))
                                for k, v in st.__dict__.items()})
    O.draft_tree(m, st, record=rec)
    # Reconstruct the chain for the first row of the last pass.
    L = st.L
    hroot = O.draft_catch_up(m, st_copy)
    # Walk: pass d row r is candidate rec.rows[d][r]; rebuild from a fresh builder.
    tb = O.TreeBuilder(wl.topk)
    tb.add_children(-1, rec.topk[0][0], rec.logp[0][0])
    for d in range(1, len(rec.rows)):
        for r, c in enumerate(rec.rows[d]):
            tb.add_children(c, rec.topk[d][r], rec.logp[d][r])
    c = rec.rows[-1][0]
    chain = []
    a = c
    while a >= 0:
        chain.append(a); a = tb.parent[a]
    chain = chain[::-1]                      # depth 1 .. D-1
    feats, f_rows = [hroot], []
    for depth, cand in enumerate(chain, start=1):
        e = np.asarray(m.w["embed"][[tb.token[cand]]], np.float64)
        f_rows.append(O.draft_fc(m, feats[-1][None, :], e)[0])
        pos = np.arange(L, L + depth)
        hh, _, _ = O.draft_forward(m, np.stack(f_rows), pos, st_copy.dK, st_copy.dV,
                                   np.full(depth, L, int), None, None, O.causal_vis(depth))
        feats.append(hh[-1])
    z = O.lm_logits(m, feats[-1][None, :])[0]
    np.testing.assert_allclose(rec.logits[-1][0], z, rtol=1e-9, atol=1e-9)


# ----------------------------------------------------------------------------
# Tree construction (reading R3)
# ----------------------------------------------------------------------------

def _check_tree_invariants(tree, k):
    N = tree.n
    assert tree.parent[0] == -1 and tree.depth[0] == 0
    for i in range(1, N):
        p = tree.parent[i]
        assert 0 <= p < i
        assert tree.depth[i] == tree.depth[p] + 1
    for p in range(N):
        kids = [tree.tokens[c] for c in range(N) if tree.parent[c] == p]
        assert len(kids) == len(set(kids)) and len(kids) <= k
    words = tree.mask_words()
    vis = tree.ancestors_or_self()
    for i in range(N):
        for j in range(N):
            bit = (int(words[i, j // 64]) >> (j % 64)) & 1
            assert bit == int(vis[i, j])


def test_tree_builder_invariants_and_frontier_bruteforce():
    rng = np.random.default_rng(9)
    k, D, N = 4, 4, 16
    tb = O.TreeBuilder(k)
    lp = -np.sort(rng.exponential(size=k)).astype(np.float32)
    tb.add_children(-1, rng.choice(100, k, replace=False), lp)
    for d in range(2, D + 1):
        fr = tb.frontier(d - 1)
        same_depth = [c for c in range(len(tb.token)) if tb.depth[c] == d - 1]
        brute = sorted(same_depth, key=lambda c: (-tb.score[c], c))[:k]
        assert fr == brute
        for c in fr:
            tb.add_children(c, rng.choice(100, k, replace=False),
                            -np.sort(rng.exponential(size=k)).astype(np.float32))
    assert len(tb.token) == k + (D - 1) * k * k
    tree = tb.finalize(N)
    _check_tree_invariants(tree, k)
    # the kept set is the N-1 best by score (ties: depth, creation)
    best = sorted(range(len(tb.token)), key=lambda c: (-tb.score[c], tb.depth[c], c))[:N - 1]
    assert sorted(tree.tokens[1:].tolist()) == sorted(tb.token[c] for c in best)


def test_tree_keeping_every_candidate_and_chain():
    rng = np.random.default_rng(10)
    k, D = 2, 3
    tb = O.TreeBuilder(k)
    tb.add_children(-1, [1, 2], np.float32([-0.1, -0.2]))
    for d in range(2, D + 1):
        for c in tb.frontier(d - 1):
            tb.add_children(c, [3, 4], np.float32([-0.3, -0.5]))
    n_all = k + (D - 1) * k * k
    tree = tb.finalize(n_all + 1)
    _check_tree_invariants(tree, k)
    assert (tree.depth[1:] > 0).all() and tree.n == n_all + 1
    # k = 1 gives the greedy chain
    tb1 = O.TreeBuilder(1)
    tb1.add_children(-1, [7], np.float32([-1.0]))
    for d in range(2, 5):
        tb1.add_children(tb1.frontier(d - 1)[0], [7 + d], np.float32([-1.0]))
    t1 = tb1.finalize(5)
    np.testing.assert_array_equal(t1.parent, [-1, 0, 1, 2, 3])
    np.testing.assert_array_equal(t1.tokens[1:], [7, 9, 10, 11])


def test_drafted_tree_invariants(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    tree = O.draft_tree(m, st)
    assert tree.n == wl.tree_nodes and tree.depth.max() <= wl.tree_depth
    _check_tree_invariants(tree, wl.topk)


# ----------------------------------------------------------------------------
# Acceptance (Eq. 6 at T = 0)
# ----------------------------------------------------------------------------

def _tree(parent, tokens):
    parent = np.asarray(parent)
    depth = np.zeros(len(parent), int)
    for i in range(1, len(parent)):
        depth[i] = depth[parent[i]] + 1
    return O.Tree(tokens=np.asarray(tokens), parent=parent, depth=depth)


def test_accept_handbuilt_cases():
    t = _tree([-1, 0, 0, 1, 1, 3], [9, 10, 11, 12, 13, 14])
    path, a, bonus = O.accept(t, np.array([10, 12, 0, 14, 0, 77]))
    assert path.tolist() == [0, 1, 3, 5] and a == 3 and bonus == 77
    path, a, bonus = O.accept(t, np.array([55, 12, 0, 14, 0, 77]))
    assert path.tolist() == [0] and a == 0 and bonus == 55
    path, a, bonus = O.accept(t, np.array([11, 0, 5, 0, 0, 0]))
    assert path.tolist() == [0, 2] and a == 1 and bonus == 5


def test_accept_matches_bruteforce_longest_matching_path():
    rng = np.random.default_rng(11)
    for _ in range(200):
        N = int(rng.integers(1, 12))
        parent = [-1] + [int(rng.integers(0, i)) for i in range(1, N)]
        toks = [0] * N
        for p in range(N):           # siblings distinct
            kids = [c for c in range(N) if parent[c] == p]
            vals = rng.choice(6, len(kids), replace=False)
            for c, v in zip(kids, vals):
                toks[c] = int(v)
        t = _tree(parent, toks)
        g = rng.integers(0, 6, size=N)
        best = [0]
        for leaf in range(N):        # every root-to-node path, keep the longest valid one
            chain = []
            j = leaf
            while j >= 0:
                chain.append(j); j = parent[j]
            chain = chain[::-1]
            if all(toks[chain[i + 1]] == g[chain[i]] for i in range(len(chain) - 1)):
                if len(chain) > len(best):
                    best = chain
        path, a, bonus = O.accept(t, g)
        assert path.tolist() == best and bonus == g[best[-1]]


# ----------------------------------------------------------------------------
# Lossless: speculative decoding emits the greedy autoregressive sequence
# ----------------------------------------------------------------------------

def _spec_tokens(m, ids, vis, steps, plant=None):
    st = O.prefill(m, ids, vis)
    accepted = []
    for s in range(steps):
        tree = None if plant is None else plant(st, s)
        _, _, _, a, _ = O.spec_step(m, st, tree)
        accepted.append(a)
    return st.emitted, accepted


def test_lossless_random_draft(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    emitted, _ = _spec_tokens(m, ids, vis, wl.steps)
    assert emitted == O.greedy_ar(m, ids, vis, len(emitted))


def test_lossless_planted_full_accept(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    D = wl.tree_depth
    ar = O.greedy_ar(m, ids, vis, 1 + 6 * (D + 1) + D + 2)
    rng = np.random.default_rng(12)

    def plant(st, s):
        # position in the AR stream of the current root
        j = len(st.emitted) - 1
        cont = ar[j + 1:j + 1 + D]
        N = wl.tree_nodes
        parent = list(range(-1, D))                 # chain root..D
        toks = [st.root] + cont
        while len(parent) < N:                      # distractor leaves off the chain
            p = int(rng.integers(0, D + 1))
            parent.append(p)
            used = {toks[c] for c in range(len(toks)) if parent[c] == p}
            t = int(rng.integers(0, wl.vocab))
            while t in used:
                t = (t + 1) % wl.vocab
            toks.append(t)
        return _tree(parent, toks)

    emitted, acc = _spec_tokens(m, ids, vis, 6, plant)
    assert acc == [D] * 6
    assert emitted == ar[:len(emitted)]


def test_lossless_planted_random_depth(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    D = wl.tree_depth
    ar = O.greedy_ar(m, ids, vis, 1 + 6 * (D + 1) + D + 2)
    rng = np.random.default_rng(13)
    depths = []

    def plant(st, s):
        j = len(st.emitted) - 1
        d = int(rng.integers(0, D + 1))
        depths.append(d)
        cont = ar[j + 1:j + 1 + d]
        wrong = (ar[j + 1 + d] + 1) % wl.vocab      # a wrong token at depth d+1
        parent = list(range(-1, d)) + [d]
        toks = [st.root] + cont + [wrong]
        return _tree(parent, toks)

    emitted, acc = _spec_tokens(m, ids, vis, 6, plant)
    assert acc == depths
    assert emitted == ar[:len(emitted)]


def test_compaction_equals_causal_forward(tiny_setup):
    """After accepting, the cache equals a plain causal forward over the prefix
    and the emitted tokens."""
    wl, w, m, ids, vis = tiny_setup
    st = O.prefill(m, ids, vis)
    for _ in range(3):
        O.spec_step(m, st)
    committed = st.emitted[:st.L - len(ids)]
    _, kv = _causal_last_logits(m, ids, vis, committed)
    for l in range(wl.n_layers):
        np.testing.assert_allclose(st.K[l], kv[l][0], rtol=1e-9, atol=1e-10)
        np.testing.assert_allclose(st.V[l], kv[l][1], rtol=1e-9, atol=1e-10)
    # the draft cache + pending rows cover exactly the committed positions
    assert st.dK.shape[0] + st.pend_h.shape[0] == st.L


def test_prefix_must_end_in_text(tiny_setup):
    wl, w, m, ids, vis = tiny_setup
    with pytest.raises(ValueError):
        O.prefill(m, np.array([1, 2, -1]), vis)


def test_draft_cache_after_steps_equals_draft_prefill_of_committed(tiny_setup):
    """With a forced full accept each step, the draft cache and the pending rows
    equal what a fresh prefill over prompt + emitted tokens would produce."""
    wl, w, m, ids, vis = tiny_setup
    D = wl.tree_depth
    ar = O.greedy_ar(m, ids, vis, 1 + 3 * (D + 1) + D + 2)
    st = O.prefill(m, ids, vis)
    for _ in range(3):
        j = len(st.emitted) - 1
        tree = _tree(list(range(-1, D)), [st.root] + ar[j + 1:j + 1 + D])
        _, _, _, a, _ = O.spec_step(m, st, tree)
        assert a == D
    committed_ids = np.concatenate([ids, np.asarray(st.emitted[:st.L - len(ids)], np.int64)])
    assert committed_ids.shape[0] == st.L
    ref = O.prefill(m, committed_ids, vis)           # draft cache covers 0 .. L-2
    P = st.pend_h.shape[0]
    np.testing.assert_allclose(st.dK, ref.dK[:st.L - P], rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(st.dV, ref.dV[:st.L - P], rtol=1e-9, atol=1e-10)
    # pending rows are the target features of the last P committed positions
    emb = O.embed_prompt(m, committed_ids, vis)
    e0 = np.zeros((0, wl.hidden))
    h, _ = O.target_forward(m, emb, np.arange(st.L), [(e0, e0)] * wl.n_layers,
                            np.zeros(st.L, int), None, O.causal_vis(st.L))
    np.testing.assert_allclose(st.pend_h, h[st.L - P:], rtol=1e-9, atol=1e-10)
    assert st.pend_next.tolist() == committed_ids[st.L - P + 1:].tolist() + [st.root]
