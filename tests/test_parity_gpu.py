"""GPU path vs the CPU oracle on the tiny workload (fp32 and bf16), every step.

Integer work (draft trees, top-k ids, argmax, accepted path, accepted length,
bonus, index map) is compared bit-exactly given the kernels' own float
outputs; floating-point outputs (draft logits, verify logits, KV caches) are
compared with the oracle's float64 values within the stated tolerances. The
oracle follows the kernels' integer decisions so that both sides stay on the
same tokens for all steps.
"""
import numpy as np
import pytest
import torch

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import TOL, open_engine, plant, tree_numpy
from tests.oracle_support import oracle_model, prompt_numpy
from tests.parity_support import run_parity

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype,long_prompt", [("f32", False), ("bf16", False), ("bf16", True)],
                         ids=["f32", "bf16", "bf16-long-prompt"])
def test_tiny_all_steps_match_oracle(dtype, long_prompt):
    """Every step of the tiny workload against the oracle. The long prompt
    (364 positions) takes the prefill through the GEMM's many-row path
    (separate RoPE, SwiGLU and RMSNorm kernels); the short one and every decode
    step through the fused-epilogue path."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype)
    if long_prompt:
        wl = wl.with_(n_text=(300, 300), steps=3)
    run_parity(wl, wl.steps)


@pytest.mark.parametrize("dtype,mode", [("f32", "concat"), ("f32", "feature"), ("bf16", "concat"),
                                        ("bf16", "feature")])
def test_draft_input_strategies_match_oracle(dtype, mode):
    """The paper's other visual draft-input strategies (Baseline concatenation,
    Visual Feature; Sec. 5.3) through msd_prefill's draft cache and two steps,
    against the oracle with the same strategy."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype, draft_input=mode, steps=2)
    run_parity(wl, wl.steps)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_chain_drafts_match_oracle(dtype):
    """Chain drafts (top-1 at every depth, N = D + 1), the drafting mode of the
    paper's n-alpha measurement (Sec. 5.1), against the oracle."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype, topk=1, tree_nodes=5, steps=3)
    run_parity(wl, wl.steps)


def _gpu_greedy_ar(eng, n_tokens):
    """Plain greedy decoding on the GPU path: single-node trees, one per token."""
    out = [int(eng.state()["root"].cpu()[0])]
    t = msd.Tree(1, eng.cfg.tree_nodes)
    for _ in range(n_tokens - 1):
        eng.draft_tree()            # keeps the draft cache caught up
        plant(eng, t, 0, [out[-1]], [-1])
        eng.verify(tree=t)
        eng.accept_compact(tree=t)
        out.append(int(eng.bonus.cpu()[0]))
    return out


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_lossless_planted_trees_match_greedy(dtype):
    """Speculative decoding emits the greedy autoregressive tokens (the lossless
    property), with planted trees forcing full and partial acceptance."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype)
    D = wl.tree_depth
    steps = 6
    n_ar = 1 + steps * (D + 1) + D + 2
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng, w = open_engine(wl, steps=n_ar)
    eng.prefill(ids, lens, vis, offs)
    ar = _gpu_greedy_ar(eng, n_ar)
    eng.close()
    if dtype == "f32":      # the fp32 GPU path reproduces the oracle's greedy decode
        m = oracle_model(wl, w)
        ids_np, vis_np = prompt_numpy(prompts[0])
        assert ar == O.greedy_ar(m, ids_np, vis_np, n_ar)

    eng, _ = open_engine(wl, w, steps=n_ar)
    eng.prefill(ids, lens, vis, offs)
    rng = np.random.default_rng(0)
    t = msd.Tree(1, wl.tree_nodes)
    emitted = [int(eng.root_out.cpu()[0])]
    for s in range(steps):
        j = len(emitted) - 1
        depth = D if s % 2 == 0 else int(rng.integers(0, D))
        chain = [emitted[-1]] + ar[j + 1:j + 1 + depth]
        parent = list(range(-1, depth))
        toks = list(chain)
        if depth < D:                         # a wrong child where the chain stops
            parent.append(depth); toks.append((ar[j + 1 + depth] + 1) % wl.vocab)
        while len(toks) < wl.tree_nodes:      # distractor leaves hanging off the root
            cand = int(rng.integers(0, wl.vocab))
            if cand != ar[j + 1] and cand not in toks[1:]:
                parent.append(0); toks.append(cand)
        eng.draft_tree()
        plant(eng, t, 0, toks, parent)
        eng.verify(tree=t)
        eng.accept_compact(tree=t)
        a = int(eng.accept_len.cpu()[0])
        assert a == depth, (s, a, depth)
        path = eng.path.cpu().numpy()[:a + 1]
        emitted += [toks[p] for p in path[1:]] + [int(eng.bonus.cpu()[0])]
    assert emitted == ar[:len(emitted)]
    eng.close()


def test_causality_non_ancestor_rows_bit_identical():
    """Changing one node's token leaves every row not descended from it
    bit-identical (rows see only their ancestors), on the bf16 tensor-core path."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16")
    eng, w = open_engine(wl)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    eng.draft_tree()
    toks, par, dep, mask = tree_numpy(eng.tree, 0)
    N, V = wl.tree_nodes, wl.vocab
    l1 = torch.zeros(N, V, device="cuda")
    eng.verify(logits=l1)
    j = N - 1
    eng.tree.tokens[j] = (int(toks[j]) + 7) % V
    l2 = torch.zeros(N, V, device="cuda")
    eng.verify(logits=l2)
    torch.cuda.synchronize()
    desc = [(int(mask[i, j // 64]) >> (j % 64)) & 1 for i in range(N)]
    for i in range(N):
        if desc[i]:
            assert not torch.equal(l1[i], l2[i])
        else:
            assert torch.equal(l1[i], l2[i]), i
    eng.close()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_linear_matches_torch(dtype):
    """The GEMM building block against a plain PyTorch fp32 product, over ragged
    shapes that span several tiles, a split K and a ragged tail."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype)
    eng, _ = open_engine(wl)
    dt = torch.float32 if dtype == "f32" else torch.bfloat16
    g = torch.Generator(device="cuda").manual_seed(5)
    for (M, K, O) in [(1, 256, 1024), (7, 512, 256), (16, 688, 256), (60, 4096, 384),
                      (129, 256, 200), (300, 1024, 640), (960, 512, 128)]:
        x = torch.randn(M, K, device="cuda", generator=g).to(dt)
        wt = (torch.randn(O, K, device="cuda", generator=g) * 0.02).to(dt)
        y = torch.zeros(M, O, device="cuda")
        eng.linear(x, wt, y)
        ref = x.float() @ wt.float().T
        torch.cuda.synchronize()
        err = (y - ref).abs().max().item()
        assert err <= 1e-4 * max(1.0, ref.abs().max().item()), (M, K, O, err)
        y2 = y.clone()
        eng.linear(x, wt, y2, accumulate=True)
        torch.cuda.synchronize()
        assert (y2 - 2 * ref).abs().max().item() <= 2e-4 * max(1.0, ref.abs().max().item())
        y3 = torch.zeros(M, O, device="cuda")
        eng.linear(x, wt, y3)
        torch.cuda.synchronize()
        assert torch.equal(y, y3)             # deterministic (split-K order is fixed)
    eng.close()


def test_bad_planted_tree_sets_device_status():
    """A planted tree whose root token is not the current root is detected on the
    device; the next call reports MSD_ERR_DEVICE."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="f32")
    eng, _ = open_engine(wl)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    t = msd.Tree(1, wl.tree_nodes)
    root = int(eng.root_out.cpu()[0])
    plant(eng, t, 0, [(root + 1) % wl.vocab], [-1])
    eng.verify(tree=t)
    torch.cuda.synchronize()
    with pytest.raises(msd.MsdError) as e:
        eng.verify(tree=t)
    assert e.value.status == msd.MSD_ERR_DEVICE
    eng.close()


def test_capacity_is_refused_on_the_host():
    wl = synth.WORKLOADS["tiny"].with_(dtype="f32")
    w = synth.make_weights(wl)
    from tests.gpu_support import to_device
    prompts = synth.make_prompts(wl)
    L = prompts[0].length
    cfg = msd.make_config(wl, L + wl.tree_depth + 1 + 2)       # room for about one step
    eng = msd.Engine(cfg, to_device(w))
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng.prefill(ids, lens, vis, offs)
    with pytest.raises(msd.MsdError) as e:
        for _ in range(4):
            eng.step()
    assert e.value.status == msd.MSD_ERR_CAPACITY
    eng.close()
    small = msd.make_config(wl, L)                              # prompt alone does not fit
    eng2 = msd.Engine(small, to_device(w))
    with pytest.raises(msd.MsdError) as e:
        eng2.prefill(ids, lens, vis, offs)
    assert e.value.status == msd.MSD_ERR_CAPACITY
    eng2.close()


def test_step_graph_matches_separate_calls():
    """msd_step (one CUDA graph, recorded once and replayed while the cache
    grows past 512 positions, so attention's split boundaries move between
    replays) gives bit-identical steps to msd_draft_tree + msd_verify +
    msd_accept_compact."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", n_text=(440, 440), steps=24)
    w = synth.make_weights(wl)
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    assert prompts[0].length > 500
    ea, _ = open_engine(wl, w)
    eb, _ = open_engine(wl, w)
    ea.prefill(ids, lens, vis, offs)
    eb.prefill(ids, lens, vis, offs)
    for step in range(wl.steps):
        pa = [t.clone() for t in ea.step()]
        pb = [t.clone() for t in eb.step_calls()]
        torch.cuda.synchronize()
        for x, y in zip(pa, pb):
            assert torch.equal(x, y), step
        assert torch.equal(ea.tree.tokens, eb.tree.tokens)
        assert torch.equal(ea.argmax, eb.argmax)
    sa, sb = ea.state(), eb.state()
    assert torch.equal(sa["seq_len"], sb["seq_len"]) and int(sa["seq_len"][0]) > 512
    L = int(sa["seq_len"][0])
    for name in [n for n in ("target_kv", "target_kv_lo") if n in sa]:   # hi and lo planes
        assert torch.equal(sa[name][..., :L, :], sb[name][..., :L, :]), name
    for name in [n for n in ("draft_kv", "draft_kv_lo") if n in sa]:
        assert torch.equal(sa[name][..., :L - 8, :], sb[name][..., :L - 8, :]), name
    ea.close(); eb.close()
