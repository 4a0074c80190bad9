"""GPU-vs-oracle parity of whole decode steps, shared by the tiny and the
full-width parity tests (GPU tests only).

For each checked request: the prefill's KV caches and root; then, every step,
the draft tree bit-exactly given the kernels' top-k decisions, the draft and
verify logits within tolerance, top-k ids and argmax bit-exactly on the
kernels' own logits, the argmax against the oracle's wherever its top-2 margin
exceeds the tolerance, and the accepted path, length, bonus, index map and
caches after compaction. The oracle follows the kernels' integer decisions, so
both sides stay on the same tokens for every step.
"""
import numpy as np
import torch

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import (KV_REL_L2, TOL, abs_bound, assert_close, open_engine, rel_l2,
                               record_buffers, top2_margin, tree_numpy)
from tests.oracle_support import oracle_model, prompt_numpy


def cache_values(s, name, idx):
    """The cached values at idx: fp32 entries, or hi + lo of bf16 split pairs."""
    v = s[name][idx].double()
    if s.get("lo_offset"):
        v = v + s[name + "_lo"][idx].double()
    return v.cpu().numpy()


def kv_compare(eng, st, wl, b, L, kv_tol, what):
    s = eng.state()
    nh, hd = wl.n_heads, wl.head_dim
    for l in range(wl.n_layers):
        for kv, ref in ((0, st.K[l]), (1, st.V[l])):
            g = cache_values(s, "target_kv", (l, kv, b, slice(None), slice(0, L), slice(None)))   # [nh, L, hd]
            r = np.asarray(ref[:L]).reshape(L, nh, hd).transpose(1, 0, 2)
            assert rel_l2(g, r) <= kv_tol, f"{what} layer {l} kv {kv}: {rel_l2(g, r)}"
    Ld = st.dK.shape[0]
    for kv, ref in ((0, st.dK), (1, st.dV)):
        g = cache_values(s, "draft_kv", (kv, b, slice(None), slice(0, Ld), slice(None)))
        r = np.asarray(ref).reshape(Ld, nh, hd).transpose(1, 0, 2)
        assert rel_l2(g, r) <= kv_tol, f"{what} draft kv {kv}: {rel_l2(g, r)}"


def run_parity(wl: synth.Workload, steps: int, requests=None, tol=None, kv_tol=None):
    """Prefill + `steps` decode steps of workload `wl` through the C ABI,
    checked against the oracle for the requests in `requests` (all if None),
    with the logit tolerance `tol` and the KV-cache relative-L2 bound `kv_tol`
    (the dtype's stated ones by default)."""
    dtype = wl.dtype
    tol = TOL[dtype] if tol is None else tol
    kv_tol = KV_REL_L2[dtype] if kv_tol is None else kv_tol
    B = wl.batch
    requests = list(range(B)) if requests is None else list(requests)
    eng, w = open_engine(wl, steps=steps)
    m = oracle_model(wl, w)
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng.prefill(ids, lens, vis, offs)
    torch.cuda.synchronize()
    roots = eng.root_out.cpu().numpy()
    states = {}
    for b in requests:
        ids_np, vis_np = prompt_numpy(prompts[b])
        st = O.prefill(m, ids_np, vis_np)
        if int(roots[b]) != st.root:
            # the root is the argmax of the last prompt position: equal unless a near tie
            z = O.lm_logits(m, O.target_forward(
                m, O.embed_prompt(m, ids_np, vis_np), np.arange(len(ids_np)),
                [(np.zeros((0, wl.hidden)),) * 2] * wl.n_layers, np.zeros(len(ids_np), int), None,
                O.causal_vis(len(ids_np)))[0][-1:])[0]
            assert top2_margin(z) <= abs_bound(z, tol), f"request {b}: root differs"
            st.root = int(roots[b]); st.pend_next = np.array([st.root]); st.emitted = [st.root]
        kv_compare(eng, st, wl, b, st.L, kv_tol, f"request {b} prefill")
        states[b] = st

    D, k, N, V = wl.tree_depth, wl.topk, wl.tree_nodes, wl.vocab
    logits = torch.zeros(B * N, V, device="cuda")
    for step in range(steps):
        rec = record_buffers(wl)
        eng.draft_tree(record=rec)
        torch.cuda.synchronize()
        R = {n: t.cpu().numpy() for n, t in rec.items()}
        eng.verify(logits=logits)
        torch.cuda.synchronize()
        g_all = logits.cpu().numpy()
        a_all = eng.argmax.cpu().numpy().astype(np.int64)
        eng.accept_compact()
        torch.cuda.synchronize()
        path_all = eng.path.cpu().numpy()
        alen = eng.accept_len.cpu().numpy()
        bonus = eng.bonus.cpu().numpy()
        imap_all = eng.index_map.cpu().numpy()
        s = eng.state()
        seq = s["seq_len"].cpu().numpy()
        root = s["root"].cpu().numpy()
        npend = s["n_pending"].cpu().numpy()
        for b in requests:
            st = states[b]
            what = f"request {b} step {step}"

            def forced(p, rows_logits, b=b):
                n = rows_logits.shape[0]
                return (R["topk_ids"][b, p, :n].astype(np.int64),
                        R["topk_logp"][b, p, :n].astype(np.float32))

            orec = O.DraftRecord()
            otree = O.draft_tree(m, st, record=orec, forced_logp=forced)
            toks, par, dep, mask = tree_numpy(eng.tree, b)
            np.testing.assert_array_equal(toks, otree.tokens, err_msg=f"{what} tokens")
            np.testing.assert_array_equal(par, otree.parent, err_msg=f"{what} parent")
            np.testing.assert_array_equal(dep, otree.depth, err_msg=f"{what} depth")
            np.testing.assert_array_equal(mask, otree.mask_words(), err_msg=f"{what} mask")
            for p in range(D):
                rows = orec.logits[p].shape[0]
                g = R["logits"][b, p, :rows]
                assert_close(g, orec.logits[p], tol, f"{what} draft pass {p} logits")
                for r in range(rows):
                    np.testing.assert_array_equal(R["topk_ids"][b, p, r], O.topk_ids(g[r], k))
                    lp = O.log_softmax(g[r].astype(np.float64))[R["topk_ids"][b, p, r]]
                    np.testing.assert_allclose(R["topk_logp"][b, p, r], lp, atol=2e-5, rtol=1e-5)

            g_logits = g_all[b * N:(b + 1) * N]
            g_arg = a_all[b * N:(b + 1) * N]
            vr = O.verify(m, st, otree)
            assert_close(g_logits, vr.logits, tol, f"{what} verify logits")
            margin = abs_bound(vr.logits, tol)
            for i in range(N):
                assert g_arg[i] == O.argmax_lowest(g_logits[i])      # bit-exact given logits
                if top2_margin(vr.logits[i]) > margin:
                    assert g_arg[i] == vr.argmax[i], f"{what} node {i} argmax"

            opath, oa, obonus = O.accept(otree, g_arg)
            path = path_all[b * (D + 1):(b + 1) * (D + 1)]
            assert int(alen[b]) == oa and int(bonus[b]) == obonus, what
            np.testing.assert_array_equal(path[:oa + 1], opath)
            assert (path[oa + 1:] == -1).all()
            imap = imap_all[b * (D + 1):(b + 1) * (D + 1)]
            np.testing.assert_array_equal(imap[:oa + 1], st.L + np.arange(oa + 1))
            O.compact(st, otree, vr, opath, obonus)
            assert int(seq[b]) == st.L and int(root[b]) == st.root, what
            assert int(npend[b]) == oa + 1, what
            kv_compare(eng, st, wl, b, st.L, kv_tol, what)
    eng.close()
