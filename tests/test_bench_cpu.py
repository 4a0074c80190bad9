"""The bench's roofline arithmetic, checked on the CPU against counts taken
from the synthetic models themselves: algorithmic bytes per step = the target's
weights once, the draft's weights (layer, f_down, LM head) once per dependent
draft pass, and the K/V the step's attention reads."""
import pytest

import bench
from paper_2505_14260_gb300 import synth


def _params(shapes):
    return sum(a * b for a, b in shapes)


@pytest.mark.parametrize("name", ["llava7b", "llava13b", "long7b", "tiny"])
def test_step_bytes_counts_every_weight_once_per_dependent_pass(name):
    wl = synth.WORKLOADS[name]
    H, V, NL, D = wl.hidden, wl.vocab, wl.n_layers, wl.tree_depth
    layer = _params(synth.layer_shapes(wl).values())          # q, k, v, o, gate, up, down
    target = NL * layer + V * H                                # layers + LM head (embedding rows are gathered)
    draft = layer + (2 * H) * H + V * H                        # one layer + f_down [H, 2H] + LM head
    L = 700
    kv = (NL + D) * 2 * L * H                                  # K and V of every target layer + the draft's, per pass
    total, parts = bench.step_bytes(wl, [L])
    assert parts["target_weights"] == 2 * target
    assert parts["draft_weights"] == 2 * D * draft
    assert parts["kv"] == 2 * kv
    assert total == 2 * (target + D * draft + kv)


def test_llava7b_step_bytes_near_18_gb():
    total, _ = bench.step_bytes(synth.WORKLOADS["llava7b"], [645])
    assert 17.9e9 < total < 18.2e9


def test_aggregate_rate_is_whole_job_throughput():
    assert bench.aggregate_rate(64, 1, 270.0) == pytest.approx(64 / 0.27)
    assert bench.aggregate_rate(64, 8, 270.0) == pytest.approx(8 * 64 / 0.27)


def test_gemm_traffic_only_for_the_captured_source(monkeypatch):
    assert bench.gemm_traffic(0) is None
    for bound in ("hbm", "tensor"):
        v = bench.gemm_traffic(100.0, bound)
        assert v is None or v == pytest.approx(bench.GEMM_TRAFFIC["ratio"][bound] * 100.0)
    monkeypatch.setitem(bench.GEMM_TRAFFIC, "source_sha1", "0" * 40)
    assert bench.gemm_traffic(100.0) is None


def _prof(windows, crit_ms, entry_ms, byts, flops, launches, pre=0.0):
    return {"windows": windows, "gemm_critical_ms": crit_ms, "gemm_ms": entry_ms, "gemm_bytes": byts,
            "gemm_flops": flops, "gemm_mma_flops": 2 * flops, "gemm_launches": launches,
            "gemm_prefetch_bytes": pre, "gemm_weight_bytes": byts}


def test_gemm_roofline_is_per_step_from_the_critical_spans():
    """Per step: the wait-to-exit spans (not the entry spans) divide the bytes;
    a decode mix (60 flops per byte) is HBM-bound against the copy bandwidth."""
    r = bench.gemm_roofline(_prof(4, 4 * 3.0, 4 * 4.5, 4 * 18e9, 4 * 60 * 18e9, 4 * 165, 4 * 2e9), 6000.0, "m")
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["gemm_ms_per_step"] == pytest.approx(3.0)
    assert r["gemm_ms_per_step_from_entry"] == pytest.approx(4.5)
    assert r["achieved"] == pytest.approx(18e9 / 3e-3 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / 6000.0)
    assert r["frac_nominal"] == pytest.approx(r["achieved"] / bench.NOMINAL_HBM_GBS)
    assert r["achieved_after_wait"] == pytest.approx(16e9 / 3e-3 / 1e9)
    assert r["launches_per_step"] == 165


def test_gemm_roofline_past_the_ridge_is_tensor_bound():
    """A many-row mix (500 flops per byte, above the sustained-bf16 / HBM ridge
    of about 250) reports TFLOP/s against the sustained bf16 rate."""
    tf, _ = bench.tensor_peak()
    r = bench.gemm_roofline(_prof(2, 2 * 18.0, 2 * 20.0, 2 * 27e9, 2 * 500 * 27e9, 2 * 165), 6767.1, "m")
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(500 * 27e9 / 18e-3 / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / tf)
    assert r["frac_issued"] == pytest.approx(2 * r["frac"])


def test_oracle_sample_runs_every_layer_with_two_held():
    """The CPU baseline's oracle step covers all of the target's layers (two
    layers' weights held and alternated, their prefilled caches laid down for
    every layer); nothing is scaled."""
    wl = synth.WORKLOADS["tiny"].with_(n_layers=5)
    w = synth.make_weights(wl, layers=bench.OracleSample.HELD)
    sample = bench.OracleSample(wl, w, synth.make_prompts(wl))
    assert len(sample.m.w["layers"]) == 5 and len(sample.st.K) == 5
    assert sample.m.w["layers"][4] is sample.m.w["layers"][0]
    L0 = sample.st.L
    assert sample.step_seconds() > 0
    assert sample.st.L > L0 and all(k.shape[0] == sample.st.L for k in sample.st.K)
    assert "scaled" not in sample.describe().replace("nothing scaled", "")


def test_weights_with_layers_kept_equal_the_full_set():
    """make_weights(layers=n) draws the whole random stream and keeps the first
    n decoder layers: every kept tensor equals its value in the full set (the
    reference arm's held layers are the workload's own)."""
    import torch
    wl = synth.WORKLOADS["tiny"].with_(n_layers=3)
    full, part = synth.make_weights(wl), synth.make_weights(wl, layers=2)
    assert len(part["layers"]) == 2
    for k, v in full.items():
        if k == "layers":
            for a, b in zip(v[:2], part["layers"]):
                assert a.keys() == b.keys() and all(torch.equal(a[n], b[n]) for n in a)
        elif k == "draft":
            assert all(torch.equal(v[n], part[k][n]) for n in v)
        else:
            assert torch.equal(v, part[k]), k


def test_kernel_breakdown_groups_slots_by_projection():
    """Stamp slots of two steps: the verify q/k/v slots of both layers form one
    group, rates come from the summed wait-to-exit spans, and verify attention
    is charged its requests' prefix and tree keys."""
    wl = synth.WORKLOADS["llava7b"].with_(n_layers=2)
    H, N = wl.hidden, wl.tree_nodes
    R = wl.batch * N

    def slot(kind, rows, outputs, inner, byts, ms):
        return {"kind": kind, "rows": rows, "outputs": outputs, "inner": inner, "launches": 2,
                "bytes": byts, "critical_ms": 2 * ms, "span_ms": 3 * ms}

    qkv = 3 * H * H * 2.0
    slots = [slot(0, R, 3 * H, H, qkv, 0.02), slot(1, R, wl.n_heads, wl.head_dim, 0.0, 0.01),
             slot(0, R, 3 * H, H, qkv, 0.02), slot(0, 10, 3 * H, H, qkv, 0.015)]
    rows = {g["name"]: g for g in bench.kernel_breakdown(slots, wl, [1000.0], 6767.1, 2)}
    v = rows["verify q/k/v + RoPE"]
    assert v["launches_per_step"] == 2 and v["ms_per_step"] == pytest.approx(0.04)
    assert v["us_per_launch"] == pytest.approx(20.0)
    assert v["achieved_gbs"] == pytest.approx(2 * qkv / 0.04e-3 / 1e9)
    assert v["achieved_tflops"] == pytest.approx(2 * 2.0 * R * 3 * H * H / 0.04e-3 / 1e12)
    a = rows["verify tree attention"]
    assert a["bytes_per_step"] == pytest.approx(2 * (1000 + N) * H * 2)
    assert rows["draft q/k/v + RoPE"]["launches_per_step"] == 1
