"""Plain greedy autoregressive decoding (msd_ar_step), the baseline of the
paper's speedup ratio (Sec. 4.1, Eq. 9: T_p): against the same decoding done
with planted one-node trees through msd_verify / msd_accept_compact, against
the oracle's greedy decode (fp32), on a one-node-tree context (B token rows per
forward), and its effect on the draft state."""
import pytest
import torch

from oracle import msd_oracle as O
from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import open_engine, plant
from tests.oracle_support import oracle_model, prompt_numpy

pytestmark = pytest.mark.gpu


def _ar_tokens(eng, n):
    out = [int(eng.state()["root"].cpu()[0])]     # the prefill's greedy token
    for _ in range(n - 1):
        out.append(int(eng.ar_step().cpu()[0]))
    return out


def _planted_greedy(eng, n):
    out = [int(eng.state()["root"].cpu()[0])]
    t = msd.Tree(1, eng.cfg.tree_nodes)
    for _ in range(n - 1):
        plant(eng, t, 0, [out[-1]], [-1])
        eng.verify(tree=t)
        eng.accept_compact(tree=t)
        out.append(int(eng.bonus.cpu()[0]))
    return out


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_ar_step_matches_planted_greedy_and_oracle(dtype):
    wl = synth.WORKLOADS["tiny"].with_(dtype=dtype)
    n = 24
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng, w = open_engine(wl, steps=n)
    eng.prefill(ids, lens, vis, offs)
    ar = _ar_tokens(eng, n)
    L = int(eng.state()["seq_len"].cpu()[0])
    eng.close()
    assert L == int(lens[0]) + n - 1                  # one position per token
    eng, _ = open_engine(wl, w, steps=n)
    eng.prefill(ids, lens, vis, offs)
    assert ar == _planted_greedy(eng, n)              # the same kernels, bit for bit
    eng.close()
    if dtype == "f32":                                # fp32 reproduces the oracle's greedy decode
        m = oracle_model(wl, w)
        ids_np, vis_np = prompt_numpy(prompts[0])
        assert ar == O.greedy_ar(m, ids_np, vis_np, n)


@pytest.mark.parametrize("name", ["tiny", "llava7b"])
def test_ar_one_node_context_matches(name):
    """A context built for plain decoding (one-node trees: B token rows per
    forward, the shape the speedup ratio times) emits the same tokens as a
    tree context decoding greedily (its other rows masked). 7B width cut to 2
    layers."""
    wl = synth.WORKLOADS[name].with_(dtype="bf16")
    if name != "tiny":
        wl = wl.with_(n_layers=2)
    n = 12
    prompts = synth.make_prompts(wl)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng, w = open_engine(wl, steps=n)
    eng.prefill(ids, lens, vis, offs)
    ref = _ar_tokens(eng, n)
    eng.close()
    one, _ = open_engine(wl.with_(tree_nodes=1, tree_depth=1, topk=1), w, steps=n)
    one.prefill(ids, lens, vis, offs)
    assert _ar_tokens(one, n) == ref
    one.close()


def test_ar_step_marks_draft_stale_until_prefill():
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16")
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng, _ = open_engine(wl, steps=8)
    eng.prefill(ids, lens, vis, offs)
    eng.ar_step()
    for call in (eng.draft_tree, eng.step):
        with pytest.raises(msd.MsdError) as ex:
            call()
        assert ex.value.status == msd.MSD_ERR_INVALID
    eng.prefill(ids, lens, vis, offs)
    eng.step()                                        # a fresh prefill makes the draft usable again
    torch.cuda.synchronize()
    eng.close()
