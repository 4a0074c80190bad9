"""GPU path vs the CPU oracle at the full width of the 7B, 13B, long-prefix
and batch-16 workloads.

Tolerance: the relative full-width bound of tests/gpu_support.py (the stated
absolute bound holds on the tiny workload, not at this width; see there).

The oracle (float64 numpy) cannot run 32 or 40 layers over 600-3400-token
prefixes in a test, so each workload is cut to 2 layers: every other size
(hidden, heads, FFN, vocabulary, prefix lengths, tree N/D/k, batch) is the
workload's own, so every kernel runs with the grid, tile, split and cluster
shapes that the benchmark times. For batch 16 three requests are checked
against the oracle (each request is independent: the others go through the
same launches). The full-depth 7B model is checked by the lossless property
instead: verifying a planted chain of the greedy continuation reproduces the
single-token greedy decode (logits within the bf16 tolerance, tokens equal
wherever the top-2 margin exceeds it, the whole chain accepted).
"""
import numpy as np
import pytest
import torch

from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import KV_REL_L2_FULL, TOL_FULL, abs_bound, assert_close, plant, top2_margin
from tests.parity_support import run_parity

pytestmark = pytest.mark.gpu

CASES = [("llava7b", None), ("llava13b", None), ("long7b", None), ("batch16", (0, 7, 15))]


@pytest.mark.parametrize("name,requests", CASES, ids=[c[0] for c in CASES])
def test_full_width_two_layers_match_oracle(name, requests):
    wl = synth.WORKLOADS[name].with_(n_layers=2)
    run_parity(wl, 2, requests, TOL_FULL, KV_REL_L2_FULL)


def test_llava7b_chain_drafts_two_layers_match_oracle():
    """Chain drafts at the 7B width (top-1 at every depth, N = D + 1 = 7), the
    drafting mode of the paper's n-alpha measurement and of the bench's chain
    timing, cut to 2 layers."""
    wl = synth.WORKLOADS["llava7b"].with_(n_layers=2, topk=1, tree_nodes=7)
    run_parity(wl, 2, None, TOL_FULL, KV_REL_L2_FULL)


def test_llava7b_full_depth_lossless_chain():
    wl = synth.WORKLOADS["llava7b"]
    D, N, V = wl.tree_depth, wl.tree_nodes, wl.vocab
    tol = TOL_FULL
    steps = 3
    n_ar = 1 + steps * (D + 1) + 1
    w = synth.make_weights(wl, "cuda")
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    cfg = msd.make_config(wl, wl.max_seq(n_ar))
    logits = torch.zeros(N, V, device="cuda")

    # greedy autoregressive decode: single-node trees, one token per step
    eng = msd.Engine(cfg, w)
    eng.prefill(ids, lens, vis, offs)
    t = msd.Tree(1, N)
    ar = [int(eng.root_out.cpu()[0])]
    ar_logits = []
    for _ in range(n_ar - 1):
        eng.draft_tree()
        plant(eng, t, 0, [ar[-1]], [-1])
        eng.verify(tree=t, logits=logits)
        eng.accept_compact(tree=t)
        ar_logits.append(logits[0].cpu().numpy().copy())
        ar.append(int(eng.bonus.cpu()[0]))
    eng.close()

    # speculative steps verifying planted chains of that continuation
    eng = msd.Engine(cfg, w)
    eng.prefill(ids, lens, vis, offs)
    emitted = [int(eng.root_out.cpu()[0])]
    assert emitted[0] == ar[0]
    for s in range(steps):
        j = len(emitted) - 1
        chain = [emitted[-1]] + ar[j + 1:j + 1 + D]
        eng.draft_tree()
        plant(eng, t, 0, chain, list(range(-1, D)))
        eng.verify(tree=t, logits=logits)
        eng.accept_compact(tree=t)
        g = logits[:D + 1].cpu().numpy()
        for i in range(D + 1):
            assert_close(g[i], ar_logits[j + i], tol, f"step {s} chain row {i}")
            if top2_margin(ar_logits[j + i]) > abs_bound(ar_logits[j + i], tol):
                assert int(np.argmax(g[i])) == ar[j + i + 1], (s, i)
        a = int(eng.accept_len.cpu()[0])
        path = eng.path.cpu().numpy()[:a + 1]
        emitted += [chain[p] for p in path[1:]] + [int(eng.bonus.cpu()[0])]
        if emitted != ar[:len(emitted)]:
            # only a near tie may flip a token; the rest of the run then diverges
            k = next(i for i in range(len(emitted)) if emitted[i] != ar[i])
            assert top2_margin(ar_logits[k - 1]) <= abs_bound(ar_logits[k - 1], tol), (s, k)
            break
        assert a == D, (s, a)
    eng.close()
