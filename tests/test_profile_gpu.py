"""The launch stamps of profile mode 2: replayed step graphs that time their
own tensor-core GEMMs and tree-attention launches with %globaltimer leave every
output of the step unchanged, measure each step once, and report spans that fit
inside the steps' elapsed time (the wait-to-exit spans of one stream's kernels
are disjoint); the per-slot breakdown adds up to the totals."""
import pytest
import torch

from paper_2505_14260_gb300 import msd, synth
from tests.gpu_support import open_engine

pytestmark = pytest.mark.gpu

STEPS = 4


def run_steps(wl, w, mode):
    eng, _ = open_engine(wl, w, steps=STEPS + 4)
    ids, lens, vis, offs = msd.upload_prompts(synth.make_prompts(wl))
    eng.prefill(ids, lens, vis, offs)
    if mode:
        eng.profile_enable(mode)
        eng.profile_read()
    out = []
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(STEPS):
        path, a, bonus = eng.step()
        out.append([t.clone() for t in (path, a, bonus, eng.tree.tokens, eng.argmax)])
    e1.record(stream)
    torch.cuda.synchronize()
    prof = eng.profile_read() if mode else None
    if mode:
        prof["slots"] = eng.profile_slots()
        with pytest.raises(msd.MsdError) as e:
            eng.profile_enable(3)
        assert e.value.status == msd.MSD_ERR_INVALID
        eng.profile_enable(0)
    eng.close()
    return out, prof, e0.elapsed_time(e1)


@pytest.mark.parametrize("nodes,depth,k", [(16, 4, 4), (256, 6, 16)], ids=["decode_rows", "many_rows"])
def test_stamped_step_graph_times_its_gemms(nodes, depth, k):
    """N = 16 runs every GEMM on the split-K cluster kernel; N = 256 puts the
    verify GEMMs on the persistent many-row kernel."""
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16", tree_nodes=nodes, tree_depth=depth, topk=k)
    w = synth.make_weights(wl)
    plain, _, _ = run_steps(wl, w, 0)
    stamped, prof, ms = run_steps(wl, w, 2)
    for s, (a, b) in enumerate(zip(plain, stamped)):
        for x, y in zip(a, b):
            assert torch.equal(x, y), f"step {s}: stamping changed an output"
    assert prof["windows"] == STEPS
    n = prof["gemm_launches"]
    assert n > 0 and n % STEPS == 0, n
    assert 0.0 < prof["gemm_critical_ms"] <= prof["gemm_ms"]
    assert prof["gemm_critical_ms"] <= ms, (prof["gemm_critical_ms"], ms)
    assert prof["gemm_bytes"] > prof["gemm_weight_bytes"] > 0
    assert prof["gemm_flops"] <= prof["gemm_mma_flops"] <= 2 * prof["gemm_flops"]
    assert 0 < prof["gemm_prefetch_bytes"] <= prof["gemm_weight_bytes"]   # (capped per launch)
    gemm = [s for s in prof["slots"] if s["kind"] == 0]
    attn = [s for s in prof["slots"] if s["kind"] == 1]
    assert len(gemm) == n // STEPS and len(attn) > 0
    assert all(s["launches"] == STEPS for s in prof["slots"])
    assert all(0.0 < s["critical_ms"] <= s["span_ms"] for s in prof["slots"])
    assert sum(s["critical_ms"] for s in gemm) == pytest.approx(prof["gemm_critical_ms"], rel=1e-9)
    assert sum(s["bytes"] * s["launches"] for s in gemm) == pytest.approx(prof["gemm_bytes"], rel=1e-9)
    assert sum(s["critical_ms"] for s in prof["slots"]) <= ms
    assert all(s["outputs"] == wl.n_heads and s["inner"] == wl.head_dim for s in attn)
