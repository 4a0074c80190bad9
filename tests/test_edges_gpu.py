"""Edge cases of the decode step on the GPU path, against the oracle: the
degenerate depth-1 tree (no tree-expansion pass), the largest tree the
configuration admits (N = 256 nodes in four mask words, k = 16, 1296
candidates), speculative sampling over that tree (16 children per node), and
the prompts msd_prefill must refuse before any launch."""
import pytest
import torch

import numpy as np

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import open_engine
from tests.parity_support import run_parity
from tests.test_sample_gpu import run_sampling

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_depth_one_tree_matches_oracle(dtype):
    """D = 1: the root slot's top-k are the whole tree (N = 1 + k)."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype, tree_depth=1, tree_nodes=5, steps=3)
    run_parity(wl, wl.steps)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_largest_tree_matches_oracle(dtype):
    """N = 256 (four 64-bit mask words per node, four query-row tiles and four
    tree key tiles per request in attention, a many-row verify GEMM), k = 16,
    D = 6: k + (D-1) k^2 = 1296 candidates ranked for 255 slots."""
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype, tree_nodes=256, tree_depth=6, topk=16, steps=2)
    run_parity(wl, wl.steps)


def test_sampling_over_the_largest_tree_matches_oracle():
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", tree_nodes=256, tree_depth=6, topk=16, steps=2)
    near, _ = run_sampling(wl, 1.0, wl.steps, seed=5)
    assert near <= 1


def test_prefill_refuses_invalid_prompts():
    """Refused on the host with MSD_ERR_INVALID (MSD_ERR_CAPACITY for a prompt
    that leaves no room for a step), before anything is launched."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="f32")
    eng, _ = open_engine(wl)
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    L = lens[0]

    def expect(status, ids_, lens_, vis_=vis, offs_=offs):
        with pytest.raises(msd.MsdError) as e:
            eng.prefill(ids_, lens_, vis_, offs_)
        assert e.value.status == status

    expect(msd.MSD_ERR_INVALID, ids, [0])                                 # empty prompt
    expect(msd.MSD_ERR_INVALID, ids, [L + 1])                             # longer than its row
    vis_end = ids.clone()
    vis_end[0, L - 1] = -1
    expect(msd.MSD_ERR_INVALID, vis_end, lens)                            # ends in a visual slot
    bad = ids.clone()
    bad[0, 3] = wl.vocab
    expect(msd.MSD_ERR_INVALID, bad, lens)                                # token id out of range
    bad[0, 3] = -2
    expect(msd.MSD_ERR_INVALID, bad, lens)
    expect(msd.MSD_ERR_INVALID, ids, lens, None, offs)                    # visual slots, no rows
    eng.close()
    small, _ = open_engine(wl.with_(n_text=(4, 4)), steps=0)
    expect_small = small.cfg.max_seq
    long_ids = torch.zeros(1, expect_small, dtype=torch.int32, device="cuda")
    with pytest.raises(msd.MsdError) as e:
        small.prefill(long_ids, [expect_small], None, [0])
    assert e.value.status == msd.MSD_ERR_CAPACITY                        # no room for a step
    small.close()


def _depth(par, i):
    d, j = 0, par[i]
    while j >= 0:
        d, j = d + 1, par[j]
    return d


def test_tree_complete_derives_depths_and_ancestor_masks():
    """msd_tree_complete (the binding's Engine.plant) derives the depths and the
    ancestor-or-self bitmasks of caller-planted trees on the device: compared
    with the oracle's Tree (a walk of the parent links) for two requests, one
    across a 64-node word boundary, the other a chain; a parent that does not
    precede its node is reported by the next call."""
    wl = synth.WORKLOADS["tiny"].with_(batch=2, tree_nodes=70, tree_depth=6, topk=16, steps=1)
    eng, _ = open_engine(wl)
    t = msd.Tree(2, 70)
    trees = {0: [-1] + [(i - 1) // 2 if i % 5 else i - 1 for i in range(1, 66)],
             1: list(range(-1, 69))}
    for b, par in trees.items():
        eng.plant(t, b, [3] * len(par), par)
    torch.cuda.synchronize()
    W = t.W
    mask = t.mask.cpu().numpy().view(np.uint64).reshape(2, 70, W)
    depth = t.depth.cpu().numpy().reshape(2, 70)
    for b, par in trees.items():
        n = len(par)
        ref = O.Tree(tokens=np.zeros(n, np.int64), parent=np.array(par), depth=np.zeros(n, np.int64))
        np.testing.assert_array_equal(mask[b, :n], ref.mask_words())
        assert not mask[b, n:].any()
        np.testing.assert_array_equal(depth[b, :n], [_depth(par, i) for i in range(n)])
    eng.plant(t, 0, [3, 4, 5], [-1, 2, 0])          # node 1's parent follows it
    torch.cuda.synchronize()
    with pytest.raises(msd.MsdError) as e:
        eng.plant(t, 0, [3], [-1])
    assert e.value.status == msd.MSD_ERR_DEVICE
    eng.close()


def test_bounded_wait_that_runs_out_is_reported():
    """Failure detection without a fault: the library's bounded mbarrier wait,
    given a 1 ms limit on a barrier that nothing arrives at, gives up and sets
    the context's status word; the next call reports MSD_ERR_DEVICE."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", steps=1)
    eng, _ = open_engine(wl)
    eng.test_wait_timeout(1_000_000)
    torch.cuda.synchronize()
    with pytest.raises(msd.MsdError) as e:
        eng.draft_tree()
    assert e.value.status == msd.MSD_ERR_DEVICE
    eng.close()


def test_bf16_context_never_reads_its_borrowed_projection_matrices():
    """A bf16 context packs every projection matrix (the target's and the
    draft's wq, wk, wv, wo, w_gate, w_up, w_down, plus lm_head and draft_fc)
    into copies of its own in msd_create and reads the caller's matrices no
    more: overwriting them with NaN afterwards changes no output of the step."""
    from tests.gpu_support import to_device
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16")
    w = synth.make_weights(wl)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    runs = []
    for poison in (False, True):
        wd = to_device(w)
        eng = msd.Engine(msd.make_config(wl, wl.max_seq(4)), wd)
        if poison:
            for lw in wd["layers"] + [wd["draft"]]:
                for n in synth.LAYER_MATS:
                    lw[n].fill_(float("nan"))
            wd["lm_head"].fill_(float("nan"))
            wd["draft_fc"].fill_(float("nan"))
        eng.prefill(ids, lens, vis, offs)
        out = []
        for _ in range(3):
            path, a, bonus = eng.step()
            out.append([t.clone() for t in (path, a, bonus, eng.tree.tokens, eng.argmax)])
        torch.cuda.synchronize()
        eng.close()
        runs.append(out)
    for s, (x, y) in enumerate(zip(*runs)):
        for p, q in zip(x, y):
            assert torch.equal(p, q), f"step {s}"


def test_single_split_attention_matches_oracle():
    """When the (row tile, head) CTAs of a launch fill a wave by themselves
    (40 requests x 4 heads on the tiny model), attention takes each request's
    whole cache and then its tree keys in one CTA (no cluster, no combine); a
    ragged batch against the oracle. (Batch 1 on the tiny model runs nine
    splits per head, the last one with the tree keys.)"""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", batch=40, n_text=(8, 90), steps=2)
    run_parity(wl, wl.steps, (0, 17, 39))
