"""Speculative sampling at temperature T > 0 on the GPU path (msd_accept_sample,
msd_step_sample) against the oracle's accept_sample (Sec. 3.2, Eq. 6 and the
adjusted distribution after it, with the draft's top-k candidates as point-mass
proposals), given identical logits and identical uniforms.

The integer outcome of each walk (accepted path, accepted length, drawn token,
index map) is compared exactly. The kernel evaluates p = softmax(z / T) with
fp32 exponentials (about 1e-6 relative error) and error-free sums, the oracle
in float64, so the two can differ only where a uniform lies within about 1e-6
(relative) of a decision boundary. Such a near tie is recognised by re-running
the oracle with every uniform scaled by 1 +- 1e-5 (ten times the kernel's
error): the kernel's outcome must then equal one of those; near ties are
counted and must stay rare. After each step the state (L, root, pending rows)
and the KV caches are checked against the oracle following the same decisions.
"""
import numpy as np
import pytest
import torch

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import KV_REL_L2, TOL, assert_close, open_engine, plant, tree_numpy
from tests.oracle_support import oracle_model, prompt_numpy
from tests.parity_support import kv_compare

pytestmark = pytest.mark.gpu

DELTA = 1e-5          # relative perturbation of the uniforms that exposes a near tie


def _outcome(tree, logits, T, u, k):
    path, a, bonus = O.accept_sample(tree, logits, T, u, k)
    return [int(x) for x in path], int(a), int(bonus)


def check_walk(gpu, tree, logits, T, u, k, what):
    """Returns 0 if the kernel's walk equals the oracle's, 1 if it equals the
    oracle's under a 1 +- DELTA rescaling of the uniforms (a near tie)."""
    ref = _outcome(tree, logits, T, u, k)
    if gpu == ref:
        return 0
    top = np.nextafter(1.0, 0.0)
    for s in (1.0 + DELTA, 1.0 - DELTA):
        if gpu == _outcome(tree, logits, T, np.minimum(u * s, top), k):
            return 1
    raise AssertionError(f"{what}: kernel walk {gpu} != oracle walk {ref}")


def spine_tree(eng, logits, wl, b, width):
    """A caller-planted tree for request b whose every level holds the target's
    `width` likeliest tokens under the first node of the level above (each
    level read from a verify of the tree grown so far): at a low temperature
    its walk accepts deep. The other requests keep a root-only tree."""
    N, D = wl.tree_nodes, wl.tree_depth
    assert 1 + D * width <= N
    roots = eng.state()["root"].cpu().numpy()
    t = msd.Tree(wl.batch, N)
    for r in range(wl.batch):
        plant(eng, t, r, [int(roots[r])], [-1])
    toks, par, head = [int(roots[b])], [-1], 0
    for _ in range(D):
        plant(eng, t, b, toks, par)
        eng.verify(tree=t, logits=logits)
        row = logits[b * N + head].cpu().numpy()
        top = O.topk_ids(row, width)
        first = len(toks)
        toks += [int(x) for x in top]
        par += [head] * width
        head = first
    plant(eng, t, b, toks, par)
    return t


def run_sampling(wl, T, steps, spine_every=0, seed=0):
    """Prefill + `steps` sampling steps through the C ABI, every request
    checked against the oracle. With spine_every = s > 0, every s-th step
    verifies a planted spine tree for request 0 instead of the drafted tree.
    Returns (near ties, accepted drafts summed over steps and requests)."""
    B, N, D, k, V = wl.batch, wl.tree_nodes, wl.tree_depth, wl.topk, wl.vocab
    tol, kv_tol = TOL[wl.dtype], KV_REL_L2[wl.dtype]
    eng, w = open_engine(wl, steps=steps)
    m = oracle_model(wl, w)
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng.prefill(ids, lens, vis, offs)
    torch.cuda.synchronize()
    roots = eng.root_out.cpu().numpy()
    states = []
    for b in range(B):
        st = O.prefill(m, *prompt_numpy(prompts[b]))
        assert int(roots[b]) == st.root, f"request {b}: root"
        states.append(st)
    gen = torch.Generator().manual_seed(seed)
    logits = torch.zeros(B * N, V, device="cuda")
    near, accepted = 0, 0
    for step in range(steps):
        eng.draft_tree()
        tree = eng.tree
        if spine_every and step % spine_every == 0:
            tree = spine_tree(eng, logits, wl, 0, min(k, (N - 1) // D))
        eng.verify(tree=tree, logits=logits)
        u = torch.rand(B, D + 1, k + 1, generator=gen)
        eng.accept_sample(T, u.cuda(), logits=logits, tree=tree)
        torch.cuda.synchronize()
        g_all = logits.cpu().numpy().astype(np.float64)
        path_all, alen = eng.path.cpu().numpy(), eng.accept_len.cpu().numpy()
        bonus, imap_all = eng.bonus.cpu().numpy(), eng.index_map.cpu().numpy()
        s = eng.state()
        seq, root, npend = (s[n].cpu().numpy() for n in ("seq_len", "root", "n_pending"))
        for b in range(B):
            st = states[b]
            what = f"T={T} request {b} step {step}"
            toks, par, dep, _ = tree_numpy(tree, b)
            n = int(tree.n_nodes[b].cpu())
            otree = O.Tree(tokens=toks[:n].copy(), parent=par[:n].copy(), depth=dep[:n].copy())
            a = int(alen[b])
            path = path_all[b * (D + 1):(b + 1) * (D + 1)]
            gpu = ([int(x) for x in path[:a + 1]], a, int(bonus[b]))
            assert (path[a + 1:] == -1).all(), what
            g = g_all[b * N:b * N + n]
            near += check_walk(gpu, otree, g, T, u[b].numpy().astype(np.float64), k, what)
            accepted += a
            np.testing.assert_array_equal(imap_all[b * (D + 1):b * (D + 1) + a + 1], st.L + np.arange(a + 1))
            # the oracle follows the kernel's decisions: same draft catch-up,
            # verify of the same tree, compaction of the same path
            O.draft_catch_up(m, st)
            otree.tokens[0] = st.root
            vr = O.verify(m, st, otree)
            assert_close(g, vr.logits, tol, f"{what} verify logits")
            O.compact(st, otree, vr, np.array(gpu[0], np.int64), gpu[2])
            assert int(seq[b]) == st.L and int(root[b]) == st.root and int(npend[b]) == a + 1, what
            kv_compare(eng, st, wl, b, st.L, kv_tol, what)
    eng.close()
    return near, accepted


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sampling_drafted_trees_match_oracle(dtype):
    """T = 1 on the drafted trees of a ragged batch of three requests: the walk
    mostly rejects and draws from the adjusted distribution."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype, batch=3, n_text=(24, 40), steps=4)
    near, _ = run_sampling(wl, 1.0, wl.steps, seed=1)
    assert near <= 1


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sampling_deep_acceptance_matches_oracle(dtype):
    """T = 0.05 with planted spine trees on alternate steps (drafted trees on
    the others): walks that accept several drafts, reject some and draw at
    interior nodes and at leaves. (At this temperature the tiny model's three
    likeliest tokens hold about 97% of a node's mass.)"""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype, steps=8)
    near, accepted = run_sampling(wl, 0.05, wl.steps, spine_every=2, seed=2)
    assert near <= 1
    assert accepted >= 2, accepted


def test_low_temperature_is_greedy_acceptance():
    """At T = 1e-6 the sampled walk equals greedy acceptance on the kernels'
    argmax wherever the top-2 logit margin dwarfs T (the zero-temperature
    limit of Eq. 6), here on a spine tree that accepts fully."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="f32")
    N, D, k = wl.tree_nodes, wl.tree_depth, wl.topk
    eng, w = open_engine(wl)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    logits = torch.zeros(N, wl.vocab, device="cuda")
    eng.draft_tree()
    t = spine_tree(eng, logits, wl, 0, 3)
    eng.verify(tree=t, logits=logits)
    torch.cuda.synchronize()
    toks, par, dep, _ = tree_numpy(t, 0)
    n = int(t.n_nodes[0].cpu())
    otree = O.Tree(tokens=toks[:n], parent=par[:n], depth=dep[:n])
    gpath, ga, gbonus = O.accept(otree, eng.argmax.cpu().numpy().astype(np.int64))
    assert ga == D
    srt = np.sort(logits.cpu().numpy()[gpath], axis=1)
    assert (srt[:, -1] - srt[:, -2]).min() > 5e-5       # exp(-margin / T) < e^-50
    u = torch.rand(1, D + 1, k + 1, generator=torch.Generator().manual_seed(4))
    eng.accept_sample(1e-6, u.cuda(), logits=logits, tree=t)
    torch.cuda.synchronize()
    assert int(eng.accept_len.cpu()[0]) == ga and int(eng.bonus.cpu()[0]) == gbonus
    assert eng.path.cpu().numpy().tolist() == [int(x) for x in gpath]
    eng.close()


def test_step_sample_graph_matches_separate_calls():
    """msd_step_sample (a replayed CUDA graph reading the uniforms' buffer when
    it runs) gives bit-identical steps to msd_draft_tree + msd_verify (logits
    kept in the context) + msd_accept_sample."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", steps=8)
    D, k = wl.tree_depth, wl.topk
    w = synth.make_weights(wl)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    ea, _ = open_engine(wl, w)
    eb, _ = open_engine(wl, w)
    ea.prefill(ids, lens, vis, offs)
    eb.prefill(ids, lens, vis, offs)
    gen = torch.Generator().manual_seed(9)
    u_buf = torch.zeros(1, D + 1, k + 1, device="cuda")
    for step in range(wl.steps):
        u = torch.rand(1, D + 1, k + 1, generator=gen).cuda()
        u_buf.copy_(u)
        pa = [t.clone() for t in ea.step_sample(0.7, u_buf)]
        eb.draft_tree()
        eb.verify()
        pb = [t.clone() for t in eb.accept_sample(0.7, u)]
        torch.cuda.synchronize()
        for x, y in zip(pa, pb):
            assert torch.equal(x, y), step
        assert torch.equal(ea.tree.tokens, eb.tree.tokens)
    sa, sb = ea.state(), eb.state()
    L = int(sa["seq_len"][0])
    assert torch.equal(sa["seq_len"], sb["seq_len"]) and torch.equal(sa["root"], sb["root"])
    for name in [n for n in ("target_kv", "target_kv_lo") if n in sa]:   # hi and lo planes
        assert torch.equal(sa[name][..., :L, :], sb[name][..., :L, :]), name
    ea.close(); eb.close()


def test_sample_argument_errors():
    """Bad temperatures and null uniforms are refused on the host before any
    launch; a planted node with more than k children is reported through the
    device status word."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="f32")
    N, D, k = wl.tree_nodes, wl.tree_depth, wl.topk
    eng, _ = open_engine(wl)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    u = torch.full((1, D + 1, k + 1), 0.5, device="cuda")
    for T in (0.0, -1.0, float("inf"), float("nan"), 1e-45):
        with pytest.raises(msd.MsdError) as e:
            eng.accept_sample(T, u)
        assert e.value.status == msd.MSD_ERR_INVALID, T
        with pytest.raises(msd.MsdError) as e:
            eng.step_sample(T, u)
        assert e.value.status == msd.MSD_ERR_INVALID, T
    with pytest.raises(msd.MsdError) as e:
        eng.accept_sample(1.0, None)
    assert e.value.status == msd.MSD_ERR_INVALID
    eng.draft_tree()
    root = int(eng.state()["root"].cpu()[0])
    t = msd.Tree(1, N)
    plant(eng, t, 0, [root] + list(range(k + 1)), [-1] + [0] * (k + 1))     # k + 1 children
    eng.verify(tree=t)
    eng.accept_sample(1.0, u, tree=t)
    torch.cuda.synchronize()
    with pytest.raises(msd.MsdError) as e:
        eng.verify(tree=t)
    assert e.value.status == msd.MSD_ERR_DEVICE
    eng.close()


def test_many_walks_match_oracle():
    """96 walks (32 ragged requests x 3 steps at T = 0.2, 1 and 3) against the
    oracle's accept_sample on the kernels' logits with the same uniforms: the
    walk and the drawn token only (the caches are checked by the tests above)."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", batch=32, n_text=(8, 60), steps=3)
    B, N, D, k, V = wl.batch, wl.tree_nodes, wl.tree_depth, wl.topk, wl.vocab
    eng, _ = open_engine(wl, steps=wl.steps)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    logits = torch.zeros(B * N, V, device="cuda")
    gen = torch.Generator().manual_seed(21)
    near = walks = 0
    for step, T in enumerate((0.2, 1.0, 3.0)):
        eng.draft_tree()
        eng.verify(logits=logits)
        u = torch.rand(B, D + 1, k + 1, generator=gen)
        eng.accept_sample(T, u.cuda(), logits=logits)
        torch.cuda.synchronize()
        g_all = logits.cpu().numpy().astype(np.float64)
        path_all, alen, bonus = eng.path.cpu().numpy(), eng.accept_len.cpu().numpy(), eng.bonus.cpu().numpy()
        for b in range(B):
            toks, par, dep, _ = tree_numpy(eng.tree, b)
            otree = O.Tree(tokens=toks, parent=par, depth=dep)
            a = int(alen[b])
            gpu = ([int(x) for x in path_all[b * (D + 1):b * (D + 1) + a + 1]], a, int(bonus[b]))
            near += check_walk(gpu, otree, g_all[b * N:(b + 1) * N], T, u[b].numpy().astype(np.float64), k,
                               f"T={T} request {b} step {step}")
            walks += 1
    eng.close()
    assert walks == 96 and near <= 2


def test_sampling_at_the_vocabulary_limit_matches_oracle():
    """msd_accept_sample at the largest vocabulary it accepts (393216 tokens:
    one removed-candidate bit per token fills its 48 KB of shared memory),
    on caller-supplied logits, against the oracle's accept_sample. In the
    middle step request 0 verifies a planted tree whose candidates are the
    vocabulary's last three tokens and draws uniforms that reject both root
    children, so the residual draw runs with the top bits of the mask set."""
    V = 48 * 1024 * 8
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", vocab=V, topk=2, tree_nodes=5, tree_depth=2,
                                       batch=2, steps=3)
    B, N, D, k = wl.batch, wl.tree_nodes, wl.tree_depth, wl.topk
    eng, _ = open_engine(wl, steps=wl.steps)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    logits = torch.zeros(B * N, V, device="cuda")
    gen = torch.Generator().manual_seed(31)
    near = 0
    for step in range(wl.steps):
        eng.draft_tree()
        tree = eng.tree
        u = torch.rand(B, D + 1, k + 1, generator=gen)
        if step == 1:
            tree = msd.Tree(B, N)
            roots = eng.state()["root"].cpu().numpy()
            plant(eng, tree, 0, [int(roots[0]), V - 1, V - 2, V - 3], [-1, 0, 0, 1])
            plant(eng, tree, 1, [int(roots[1])], [-1])
        eng.verify(tree=tree, logits=logits)
        if step == 1:
            z = torch.randn(N, V, generator=gen) * 0.5
            z[:, V - 4:] += torch.tensor([13.0, 13.0, 13.5, 14.0])  # about 86% of the mass
            logits[:N] = z.cuda()
            u[0, 0, :k] = 0.999                                     # reject both root children
        eng.accept_sample(1.0, u.cuda(), logits=logits, tree=tree)
        torch.cuda.synchronize()
        g_all = logits.cpu().numpy().astype(np.float64)
        path_all, alen, bonus = eng.path.cpu().numpy(), eng.accept_len.cpu().numpy(), eng.bonus.cpu().numpy()
        n_nodes = tree.n_nodes.cpu().numpy()
        for b in range(B):
            toks, par, dep, _ = tree_numpy(tree, b)
            n = int(n_nodes[b])
            otree = O.Tree(tokens=toks[:n], parent=par[:n], depth=dep[:n])
            a = int(alen[b])
            gpu = ([int(x) for x in path_all[b * (D + 1):b * (D + 1) + a + 1]], a, int(bonus[b]))
            near += check_walk(gpu, otree, g_all[b * N:(b + 1) * N], 1.0, u[b].numpy().astype(np.float64), k,
                               f"request {b} step {step}")
            if step == 1 and b == 0:
                assert a == 0 and gpu[2] not in (V - 1, V - 2), gpu
    eng.close()
    assert near <= 1
