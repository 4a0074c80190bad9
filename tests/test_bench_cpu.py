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
    v = bench.gemm_traffic(100.0)
    assert v is None or v == pytest.approx(bench.GEMM_TRAFFIC["ratio"] * 100.0)
    monkeypatch.setitem(bench.GEMM_TRAFFIC, "source_sha1", "0" * 40)
    assert bench.gemm_traffic(100.0) is None
