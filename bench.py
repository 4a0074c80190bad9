#!/usr/bin/env python
"""Benchmark of the MSD decode step (draft tree -> verify -> accept/compact).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload llava7b]
                    [--impl msd|reference]

Prints ONE JSON line (rank 0). A step is one draft -> verify -> accept ->
compact pass over the batch. The default workload is the LLaVA-1.5-7B shape
(32 layers, hidden 4096, vocab 32000; 8 text + 576 visual + 56 text prompt
tokens; tree N=60, D=6, k=10; batch 1) with seeded random bf16 weights.

value        steps/s, device-timed with CUDA events over K back-to-back steps
             (inputs resident in HBM; 13+ GB of weights streamed per step, far
             larger than L2, so no flush is needed between steps)
e2e          steps/s through the public API with host buffers: prompt copied
             from pinned host memory, prefill, then every step reads its
             emitted tokens back to pinned host memory and synchronises
roofline     the step's tensor-core GEMMs (gemm_cluster_kernel for decode rows,
             gemm_persist_kernel for many rows; most of the step's kernel time),
             timed INSIDE the replayed step graph: every CTA of every GEMM launch
             stamps %globaltimer (first entry, first return from the wait on the
             previous kernel, last exit) over K_prof steps right after the timed
             region (msd_profile_enable mode 2). achieved = algorithmic bytes (or
             flops) of a step's GEMM launches / their summed wait-to-exit spans
             (disjoint, so they fit in the step);
             bound "hbm" against the measured copy bandwidth while the GEMMs'
             flops per byte stay below the ridge (measured sustained bf16 / HBM),
             else "tensor" against the measured sustained bf16 rate; a nominal
             fraction (8 TB/s, 2.25 PFLOP/s) sits beside the measured one.
             traffic = DRAM bytes per launch from an ncu capture, reported while
             the GEMM source is the one it was captured on
cpu_baseline the CPU oracle's full-depth step on the same shapes (batch 1, every
             target layer run, nothing scaled; host RAM holds two layers'
             weights, which the layers alternate), mean of one or two steps
--impl reference times the same oracle step as the reference arm (timed
             steps stop after REF_BUDGET_S; the line reports the steps timed).

Multi-GPU: the step does not shard; N ranks run N independent replicas and
value = total steps of all ranks / the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "spec-decode steps/s and verified tokens/s at LLaVA-1.5-7B shape; % HBM roofline"
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
NOMINAL_HBM_GBS = 8000.0
NOMINAL_BF16_TFLOPS = 2250.0
REF_BUDGET_S = 60.0          # timed oracle steps of the reference arm stop after this


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=64)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="llava7b")
    ap.add_argument("--impl", default="msd", choices=["msd", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-ar", action="store_true",
                    help="skip the plain greedy decoding baseline (speedup ratio)")
    ap.add_argument("--draft-input", default="embedding", choices=["embedding", "concat", "feature"],
                    help="draft input of visual prefix positions: MSD's embedding (default), the "
                         "Baseline concatenation, or the target feature (the paper's ablation)")
    ap.add_argument("--no-chain", action="store_true",
                    help="skip the chain-draft timing (T_q, T_v(gamma), n-alpha and Eq. 9)")
    ap.add_argument("--no-sampling", action="store_true",
                    help="skip the temperature-1 speculative sampling step timing")
    ap.add_argument("--layers", type=int, default=None,
                    help="cut the target to this many layers (small cases for profiling only)")
    ap.add_argument("--gemm", default=None,
                    help="M,K,O: time the tensor-core GEMM alone on that shape (kernel case)")
    return ap.parse_args()


# DRAM traffic of the GEMMs: ncu dram__bytes_read.sum + dram__bytes_write.sum
# per launch divided by the same launches' algorithmic bytes. Decode
# (gemm_cluster_kernel): the 90 launches of two 2-layer 7B-width steps, 0.9945
# (no re-reads). Many rows (gemm_persist_kernel): the first two many-row
# launches of a 2-layer batch-16 step (the draft's input projection and q/k/v at
# 160 token rows), 0.975 (0.997 and 0.960: part of q/k/v's fp32 output is still
# in L2 when the launch ends). Per launch of a full workload it is the ratio
# times its algorithmic bytes per launch. Valid for the GEMM source with this
# SHA-1 only.
GEMM_TRAFFIC = {"source_sha1": "af8b12bbe0baebb332dc96e69230605bb01a881e",
                "ratio": {"hbm": 0.9945, "tensor": 0.975}}


def gemm_traffic(bytes_per_launch, bound="hbm"):
    import hashlib
    src = os.path.join(ROOT, "paper_2505_14260_gb300", "csrc", "gemm_tc.cu")
    try:
        with open(src, "rb") as f:
            sha = hashlib.sha1(f.read()).hexdigest()
    except OSError:
        return None
    if sha != GEMM_TRAFFIC["source_sha1"] or not bytes_per_launch:
        return None
    return GEMM_TRAFFIC["ratio"][bound] * bytes_per_launch


# Output length and average acceptance lengths the paper reports (Sec. 4): the
# MLLM benchmarks average 85 output tokens; MSD's average τ over its eight
# benchmarks at temperature 0 is 4.45 on LLaVA-1.5-7B and 4.18 on 13B. Used
# only for the labelled projection of the speedup ratio (random-init drafts
# accept nothing here).
PAPER_OUTPUT_LEN = 85
PAPER_TAU = {"llava7b": 4.45, "long7b": 4.45, "batch16": 4.45, "llava13b": 4.18}


def speedup_ratio(n_out, t_p, t_step, tau, t_prof):
    """Eq. 9: (N T_p + T_profiling) / (N (step time / tokens per step) + T_profiling)."""
    from paper_2505_14260_gb300 import metrics
    return metrics.speedup_ratio(n_out, t_p, t_prof, t_step, tau)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def tensor_peak():
    """Sustained dense bf16 TFLOP/s (the GEMMs are timed inside a long step)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["bf16_tflops_sustained"]), "measured sustained"
    except Exception:
        return FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback sustained"


def gemm_roofline(prof, hbm, hbm_kind):
    """The roofline object of the step's GEMMs from in-graph launch stamps.

    A launch's duration is its span from the first return of
    griddepcontrol.wait (the previous kernel's results are visible) to its last
    CTA's exit: these spans are disjoint within the step, so their sum fits in
    the step. Each launch requests its first pipeline stages of weights before
    that wait, overlapping the previous kernel's tail; those bytes
    (prefetch_bytes) stay in the algorithmic bytes, and achieved_after_wait
    gives the rate without them (a lower bound). The span from the first CTA's
    entry is reported too: with programmatic dependent launch a CTA enters
    while the previous kernel still runs, so those spans overlap."""
    w = max(prof["windows"], 1)
    ms = prof["gemm_critical_ms"] / w
    entry_ms = prof["gemm_ms"] / w
    byts, flops = prof["gemm_bytes"] / w, prof["gemm_flops"] / w
    pre = prof["gemm_prefetch_bytes"] / w
    tf, tf_kind = tensor_peak()
    ridge = tf * 1e12 / (hbm * 1e9)                 # flops per byte
    intensity = flops / byts if byts else 0.0
    sec = ms / 1e3
    gbs = byts / sec / 1e9 if sec > 0 else None
    tfs = flops / sec / 1e12 if sec > 0 else None
    launches = prof["gemm_launches"] / w
    r = {"intensity_flop_per_byte": intensity, "ridge_flop_per_byte": ridge,
         "gemm_ms_per_step": ms, "gemm_ms_per_step_from_entry": entry_ms,
         "launches_per_step": launches, "steps": prof["windows"],
         "bytes_per_launch": byts / launches if launches else None,
         "prefetch_bytes_per_launch": pre / launches if launches else None,
         "achieved_gbs": gbs, "achieved_tflops": tfs,
         "issued_tflops": prof["gemm_mma_flops"] / w / sec / 1e12 if sec > 0 else None}
    if intensity > ridge:
        r.update({"bound": "tensor", "achieved": tfs, "peak": tf, "unit": "TFLOP/s",
                  "frac": tfs / tf if tfs else None, "peak_kind": tf_kind,
                  "frac_nominal": tfs / NOMINAL_BF16_TFLOPS if tfs else None,
                  "nominal_peak": NOMINAL_BF16_TFLOPS,
                  "frac_issued": r["issued_tflops"] / tf if tfs else None})
    else:
        after = (byts - pre) / sec / 1e9 if sec > 0 else None
        r.update({"bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s",
                  "frac": gbs / hbm if gbs else None, "peak_kind": hbm_kind,
                  "frac_nominal": gbs / NOMINAL_HBM_GBS if gbs else None,
                  "nominal_peak": NOMINAL_HBM_GBS,
                  "achieved_after_wait": after, "frac_after_wait": after / hbm if after else None})
    return r


def kernel_breakdown(slots, wl, L_mean_per_req, hbm, windows):
    """Per-projection (and attention) breakdown of the replayed step from the
    per-launch stamp slots (msd_profile_slots): launches per step, wait-to-exit
    time per launch and per step, and the achieved rate against the measured
    copy bandwidth. GEMM bytes are each launch's algorithmic bytes; verify
    attention reads every request's visible prefix and tree keys (K and V, 2
    bytes an element, the stamped steps' mean prefix); the draft passes'
    attention is timed only."""
    H, F, V, B, N = wl.hidden, wl.ffn, wl.vocab, wl.batch, wl.tree_nodes
    glu = 128 * ((F + 63) // 64)
    names = {(3 * H, H): "q/k/v + RoPE", (H, H): "O + residual", (glu, H): "gate/up + SwiGLU",
             (H, F): "down + residual", (V, H): "LM head", (H, 2 * H): "input projection"}
    groups = {}
    w = max(windows, 1)
    for sl in slots:
        if sl["launches"] <= 0:
            continue
        phase = "verify" if sl["rows"] == B * N else "draft"
        flops = None
        if sl["kind"] == 0:
            name = f"{phase} {names.get((sl['outputs'], sl['inner']), 'GEMM %dx%d' % (sl['outputs'], sl['inner']))}"
            byts = sl["bytes"]
            flops = 2.0 * sl["rows"] * sl["outputs"] * sl["inner"]
        else:
            name = f"{phase} tree attention"
            byts = sum(2 * (L + N) * H * 2 for L in L_mean_per_req) if phase == "verify" else None
        g = groups.setdefault(name, {"name": name, "launches_per_step": 0.0, "ms_per_step": 0.0,
                                     "bytes_per_step": None if byts is None else 0.0,
                                     "flops_per_step": None if flops is None else 0.0})
        g["launches_per_step"] += sl["launches"] / w
        g["ms_per_step"] += sl["critical_ms"] / w
        if byts is not None:
            g["bytes_per_step"] += byts * sl["launches"] / w
        if flops is not None:
            g["flops_per_step"] += flops * sl["launches"] / w
    out = []
    for g in groups.values():
        sec = g["ms_per_step"] / 1e3
        g["us_per_launch"] = g["ms_per_step"] * 1e3 / g["launches_per_step"]
        if g["bytes_per_step"] is not None and sec > 0:
            g["achieved_gbs"] = g["bytes_per_step"] / sec / 1e9
            g["frac_hbm"] = g["achieved_gbs"] / hbm
        if g["flops_per_step"] is not None and sec > 0:
            g["achieved_tflops"] = g["flops_per_step"] / sec / 1e12
        out.append(g)
    return sorted(out, key=lambda g: -g["ms_per_step"])


# ----------------------------------------------------------------------------
# Algorithmic bytes of a step (weights once per dependent pass + KV read)
# ----------------------------------------------------------------------------
def step_bytes(wl, L_mean_per_req):
    H, F, V, NL, D = wl.hidden, wl.ffn, wl.vocab, wl.n_layers, wl.tree_depth
    layer = 4 * H * H + 3 * H * F
    target_w = 2 * (NL * layer + V * H)
    draft_w = D * 2 * (layer + 2 * H * H + V * H)
    kv = sum(NL * 2 * L * H * 2 + D * 2 * L * H * 2 for L in L_mean_per_req)
    return target_w + draft_w + kv, dict(target_weights=target_w, draft_weights=draft_w, kv=kv)


# ----------------------------------------------------------------------------
# nvidia-smi clock sampling during the timed region
# ----------------------------------------------------------------------------
class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1])); mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------
# CPU oracle sample (cpu_baseline and the reference arm)
# ----------------------------------------------------------------------------
class OracleSample:
    """The oracle's full-depth step on the workload's shapes (batch 1).

    Every one of the target's decoder layers runs in every step; host memory
    holds two layers' weights (the workload's first two), which the layers
    alternate, so a 7B or 13B target fits in a few GB of host RAM. The prompt
    is prefilled through those two layers and its KV caches are then laid
    down for every layer (layer l gets layer l mod 2's cache): a step's cost
    depends on the caches' sizes, not on their values. Nothing is scaled: a
    step's time is the measured time of draft_tree, verify (all layers and the
    LM head), accept and compact."""

    HELD = 2

    def __init__(self, wl, weights, prompts):
        import numpy as np
        from oracle import msd_oracle as O
        from paper_2505_14260_gb300 import synth
        self.O, self.np = O, np
        self.wl = wl
        f = synth.to_numpy_f32
        w = {k: f(v) for k, v in weights.items() if hasattr(v, "dtype") and k != "layers"}
        held = [{n: f(t) for n, t in lw.items()} for lw in weights["layers"][:self.HELD]]
        w["draft"] = {n: f(t) for n, t in weights["draft"].items()}

        def cfg(n_layers):
            return O.OracleConfig(n_layers=n_layers, hidden=wl.hidden, n_heads=wl.n_heads,
                                  head_dim=wl.head_dim, ffn=wl.ffn, vocab=wl.vocab,
                                  tree_nodes=wl.tree_nodes, tree_depth=wl.tree_depth, topk=wl.topk,
                                  rms_eps=wl.rms_eps, rope_base=wl.rope_base,
                                  draft_input=wl.draft_input)
        nh = len(held)
        p = prompts[0]
        st = O.prefill(O.OracleModel(cfg(nh), dict(w, layers=held)), p.ids.astype(np.int64), f(p.vis))
        self.m = O.OracleModel(cfg(wl.n_layers), dict(w, layers=[held[i % nh] for i in range(wl.n_layers)]))
        st.K = [st.K[i % nh].copy() for i in range(wl.n_layers)]
        st.V = [st.V[i % nh].copy() for i in range(wl.n_layers)]
        self.st = st
        try:
            self.cores = len(os.sched_getaffinity(0))
        except Exception:
            self.cores = os.cpu_count()

    def step_seconds(self):
        """Measured seconds of one full-depth oracle step (batch 1)."""
        O = self.O
        t0 = time.perf_counter()
        O.spec_step(self.m, self.st)          # draft_tree, verify, accept, compact
        return time.perf_counter() - t0

    def describe(self):
        wl = self.wl
        return (f"oracle (numpy float64) full-depth step on the {wl.name} shapes, batch 1: all "
                f"{wl.n_layers} target layers, the draft and LM heads in every step, nothing "
                f"scaled; the layers alternate the workload's first {self.HELD} layers' weights "
                f"(host RAM holds {self.HELD}) and start from their prefilled KV caches")


# ----------------------------------------------------------------------------
# Replicas (--gpus N under torchrun): the step does not shard, so each rank runs
# its own copy of the workload; the only collectives are the barriers around
# the timed region and the maximum of the ranks' times.
# ----------------------------------------------------------------------------
def max_over_ranks(ms: float, world: int, device) -> float:
    """The slowest rank's time (ms); every rank gets the same value."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_rate(units_per_rank: float, world: int, ms_max: float) -> float:
    """Whole-job throughput: the units all ranks processed over the slowest
    rank's time (weak scaling: each rank processes the same units)."""
    return world * units_per_rank / (ms_max / 1e3)


def oracle_one_thread(workload: str, steps: int = 3):
    """The oracle's step on one host thread (BLAS pinned to one thread in a
    child process, so the parent's thread pools are untouched): steps/s."""
    code = (
        "import sys, time, json, statistics\n"
        f"sys.path.insert(0, {ROOT!r})\n"
        "import bench\n"
        "from paper_2505_14260_gb300 import synth\n"
        f"wl = synth.WORKLOADS[{workload!r}]\n"
        "w = synth.make_weights(wl)\n"
        "s = bench.OracleSample(wl, w, synth.make_prompts(wl))\n"
        f"est = [s.step_seconds() for _ in range({steps})]\n"
        "print(json.dumps({'value': 1.0 / statistics.mean(est)}))\n")
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    try:
        r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                           timeout=300)
        v = json.loads(r.stdout.strip().splitlines()[-1])["value"]
        return {"value": v, "unit": "steps/s", "cores": 1, "kind": "oracle",
                "sample": f"the same oracle step, BLAS and OpenMP pinned to one thread, mean of {steps} steps"}
    except Exception as ex:
        return {"value": None, "unit": "steps/s", "cores": 1, "kind": "oracle", "sample": f"failed: {ex!r}"}


def make_inputs(wl, device, layers=None):
    from paper_2505_14260_gb300 import synth
    return synth.make_weights(wl, device=device, layers=layers), synth.make_prompts(wl)


# ----------------------------------------------------------------------------
def run_reference(args, rank, world):
    """The reference arm: the float64 oracle's full-depth step on the host
    cores, timed step by step (rank 0 only). Each oracle step takes seconds, so
    at most one warm-up step runs and the timed steps stop once about
    REF_BUDGET_S has been spent (at least one); the line reports the steps it
    timed and the steps requested."""
    import torch
    from paper_2505_14260_gb300 import synth
    if rank != 0:
        return
    t_start = time.perf_counter()
    wl = synth.WORKLOADS[args.workload]
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    w, prompts = make_inputs(wl, dev, layers=OracleSample.HELD)
    w = {k: (v.cpu() if hasattr(v, "cpu") else v) for k, v in w.items() if k not in ("layers", "draft")} | \
        {"layers": [{n: t.cpu() for n, t in lw.items()} for lw in w["layers"]],
         "draft": {n: t.cpu() for n, t in w["draft"].items()}}
    sample = OracleSample(wl, w, prompts)
    t_setup = time.perf_counter() - t_start
    n_warm = min(args.warmup, 1)
    for _ in range(n_warm):
        sample.step_seconds()
    times = []
    while len(times) < max(1, args.steps) and (not times or sum(times) < REF_BUDGET_S):
        times.append(sample.step_seconds())
    n_timed, total = len(times), sum(times)
    v = n_timed / total
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "steps/s", "n_gpus": args.gpus,
            "steps": n_timed, "steps_requested": args.steps, "warmup": n_warm,
            "warmup_requested": args.warmup, "ms_per_step": 1e3 * total / n_timed,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl.name, "batch": 1, "layers": wl.n_layers},
            "cpu_baseline": {"value": v, "unit": "steps/s", "cores": sample.cores, "kind": "oracle",
                             "sample": sample.describe() + f"; {n_timed} timed steps after {n_warm} "
                                       f"warm-up (timed steps stop after ~{REF_BUDGET_S:g} s)"},
            "e2e": {"value": v, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "wall_s": time.perf_counter() - t_start, "setup_s": t_setup}
    print(json.dumps(line), flush=True)


def run_gemm_case(args):
    """One GEMM shape through msd_linear: weights [O,K] bf16 larger than L2 for
    the 7B shapes, timed per launch with CUDA events (a small kernel case for
    ncu captures and tuning)."""
    import torch
    from paper_2505_14260_gb300 import msd, synth
    M, K, O = (int(v) for v in args.gemm.split(","))
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16")
    w = {k: v.cuda() for k, v in synth.make_weights(wl).items() if hasattr(v, "cuda")}
    w["layers"] = [{n: t.cuda() for n, t in lw.items()} for lw in synth.make_weights(wl)["layers"]]
    w["draft"] = {n: t.cuda() for n, t in synth.make_weights(wl)["draft"].items()}
    eng = msd.Engine(msd.make_config(wl, 256), w)
    g = torch.Generator(device="cuda").manual_seed(3)
    x = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    n_w = max(2, (512 << 20) // (O * K * 2) + 1)          # rotate weights: > L2 per pass
    ws = [(torch.randn(O, K, device="cuda", generator=g) * 0.02).to(torch.bfloat16) for _ in range(n_w)]
    y = torch.zeros(M, O, device="cuda")
    for i in range(3):
        eng.linear(x, ws[i % n_w], y)
    torch.cuda.synchronize()
    times = []
    eng.profile_enable(True)
    eng.profile_read()
    for i in range(20):                   # the GEMM launch alone (packing excluded)
        eng.linear(x, ws[i % n_w], y)
        times.append(eng.profile_read()["gemm_ms"])
    eng.profile_enable(False)
    hbm, kind = peaks()
    ms = statistics.median(times)
    byts = O * K * 2 + M * K * 2 + M * O * 4
    print(json.dumps({"case": "gemm", "M": M, "K": K, "O": O, "ms_median": ms, "ms_min": min(times),
                      "gbs": byts / (ms / 1e3) / 1e9, "frac": byts / (ms / 1e3) / 1e9 / hbm,
                      "peak": hbm, "peak_kind": kind}), flush=True)
    eng.close()


def run_msd(args, rank, world, local_rank):
    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2505_14260_gb300 import msd, synth

    torch.cuda.set_device(local_rank)
    wl = synth.WORKLOADS[args.workload].with_(draft_input=args.draft_input)
    if args.layers:
        wl = wl.with_(n_layers=args.layers, name=f"{wl.name}-{args.layers}layers")
    B, N, D, V = wl.batch, wl.tree_nodes, wl.tree_depth, wl.vocab
    weights, prompts = make_inputs(wl, "cuda")
    K, W = args.steps, args.warmup
    K_prof = min(K, 16)
    max_seq = wl.max_prompt + (W + 2 * K + K_prof + 6) * (D + 1) + N + 8
    eng = msd.Engine(msd.make_config(wl, max_seq), weights)
    ids, lens, vis, offs = msd.upload_prompts(prompts)
    eng.prefill(ids, lens, vis, offs)
    for _ in range(W):
        eng.step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    st = eng.state()
    L0 = st["seq_len"].cpu().numpy().astype(np.int64)
    launches0 = eng.profile_read()["kernel_launches"]
    clocks = Clocks(torch.cuda.current_device())
    clocks.start()
    time.sleep(0.3)
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_push("timed")
    e0.record(stream)
    for _ in range(K):
        eng.step()
    e1.record(stream)
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    clk = clocks.stop()
    launches1 = eng.profile_read()["kernel_launches"]
    L1 = eng.state()["seq_len"].cpu().numpy().astype(np.int64)
    tokens = int((L1 - L0).sum())
    # GEMM roofline inside the replayed step graph: launch stamps (mode 2) over
    # K_prof more steps; two steps first record the stamped graphs
    eng.profile_enable(2)
    for _ in range(2):
        eng.step()
    torch.cuda.synchronize()
    eng.profile_read()
    eng.profile_slots()
    Ls0 = eng.state()["seq_len"].cpu().numpy().astype(np.int64)
    e0.record(stream)
    for _ in range(K_prof):
        eng.step()
    e1.record(stream)
    torch.cuda.synchronize()
    ms_stamped = e0.elapsed_time(e1) / K_prof
    prof = eng.profile_read()
    slots = eng.profile_slots()
    Ls1 = eng.state()["seq_len"].cpu().numpy().astype(np.int64)
    eng.profile_enable(0)
    if world > 1:
        dist.barrier()
    ms_max = max_over_ranks(ms, world, "cuda")
    steps_s = aggregate_rate(K, world, ms_max)

    hbm, peak_kind = peaks()
    roof = gemm_roofline(prof, hbm, peak_kind)
    roof["by_kernel"] = kernel_breakdown(slots, wl, [(a + b) / 2 for a, b in zip(Ls0, Ls1)], hbm,
                                         prof["windows"])
    sb, parts = step_bytes(wl, [(a + b) / 2 for a, b in zip(L0, L1)])
    step_gbs = sb / (ms / 1e3 / K) / 1e9

    # ---- end to end through the public API with host buffers --------------
    # (each step is msd_step, a replayed CUDA graph, then the emitted tokens
    # are read back to pinned host memory)
    e2e = None
    if not args.no_e2e:
        ids_h = ids.cpu().pin_memory()
        vis_h = vis.cpu().pin_memory() if vis is not None else None
        out_tok = torch.empty(B * N, dtype=torch.int32).pin_memory()
        out_path = torch.empty(B * (D + 1), dtype=torch.int32).pin_memory()
        out_a = torch.empty(B, dtype=torch.int32).pin_memory()
        out_b = torch.empty(B, dtype=torch.int32).pin_memory()
        torch.cuda.synchronize()
        e0.record(stream)
        ids_d = ids_h.to("cuda", non_blocking=True)
        vis_d = vis_h.to("cuda", non_blocking=True) if vis_h is not None else None
        eng.prefill(ids_d, lens, vis_d, offs)
        for _ in range(K):
            path, alen, bonus = eng.step()
            out_tok.copy_(eng.tree.tokens, non_blocking=True)
            out_path.copy_(path, non_blocking=True)
            out_a.copy_(alen, non_blocking=True)
            out_b.copy_(bonus, non_blocking=True)
            stream.synchronize()
        e1.record(stream)
        torch.cuda.synchronize()
        ms_e2e = e0.elapsed_time(e1)
        ms_e2e = max_over_ranks(ms_e2e, world, "cuda")
        h2d = ids_h.numel() * 4 + (vis_h.numel() * vis_h.element_size() if vis_h is not None else 0)
        d2h = (out_tok.numel() + out_path.numel() + out_a.numel() + out_b.numel()) * 4
        e2e = {"value": aggregate_rate(K, world, ms_e2e), "unit": "steps/s",
               "h2d_bytes_per_step": h2d / K, "d2h_bytes_per_step": d2h,
               "note": "prompt H2D + prefill amortised over the steps; tokens read back every step"}

    # ---- plain greedy decoding on the same kernels: the speedup ratio --------
    # (a context with a one-node tree, so each token is one target forward
    # over B rows; msd_ar_step, a replayed CUDA graph per token)
    speedup = None
    if not args.no_ar:
        wl_ar = wl.with_(tree_nodes=1, tree_depth=1, topk=1)
        K_ar = min(K, 32)
        ar = msd.Engine(msd.make_config(wl_ar, wl.max_prompt + K_ar + 16), weights)
        ar.prefill(ids, lens, vis, offs)             # first call: one-time set-up
        torch.cuda.synchronize()
        e0.record(stream)
        ar.prefill(ids, lens, vis, offs)
        e1.record(stream)
        torch.cuda.synchronize()
        t_prof = e0.elapsed_time(e1)
        for _ in range(3):
            ar.ar_step()
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(K_ar):
            ar.ar_step()
        e1.record(stream)
        torch.cuda.synchronize()
        t_p = e0.elapsed_time(e1) / K_ar
        ar.close()
        tau = tokens / (K * B)
        t_step = ms / K
        speedup = {"ar_ms_per_token": t_p, "prefill_ms": t_prof, "spec_ms_per_step": t_step,
                   "output_len": PAPER_OUTPUT_LEN, "tau_measured": tau,
                   "sr_measured": speedup_ratio(PAPER_OUTPUT_LEN, t_p, t_step, tau, t_prof),
                   "note": "Eq. 9 with the measured times: T_p = msd_ar_step (one-node tree, "
                           f"{K_ar} tokens after 3 warm-up), T_profiling = msd_prefill of the prompt, "
                           "step time / tokens per step from the timed region"}
        if wl.name in PAPER_TAU:
            speedup["sr_projected"] = {
                "tau": PAPER_TAU[wl.name],
                "value": speedup_ratio(PAPER_OUTPUT_LEN, t_p, t_step, PAPER_TAU[wl.name], t_prof),
                "note": "projection: the paper's average acceptance length of trained MSD drafts, "
                        "not measured here"}

    # ---- per-step distribution and per-phase times, after the timed region on
    # a fresh prefill (the timed number above is untouched): K_prof replayed
    # steps each bracketed by events, then K_prof steps as separate calls
    eng.prefill(ids, lens, vis, offs)
    for _ in range(3):
        eng.step()
    torch.cuda.synchronize()
    pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
             for _ in range(K_prof)]
    for a, b in pairs:
        a.record(stream)
        eng.step()
        b.record(stream)
    torch.cuda.synchronize()
    per_step = sorted(a.elapsed_time(b) for a, b in pairs)

    def pct(q):
        return per_step[min(len(per_step) - 1, int(q * (len(per_step) - 1) + 0.5))]

    evp = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    phase = [0.0, 0.0, 0.0]
    for _ in range(K_prof):
        evp[0].record(stream)
        eng.draft_tree()
        evp[1].record(stream)
        eng.verify()
        evp[2].record(stream)
        eng.accept_compact()
        evp[3].record(stream)
        torch.cuda.synchronize()
        for i in range(3):
            phase[i] += evp[i].elapsed_time(evp[i + 1]) / K_prof
    distribution = {"p10_ms": pct(0.1), "p50_ms": pct(0.5), "p90_ms": pct(0.9), "steps": K_prof,
                    "phases_ms": {"draft_tree": phase[0], "verify": phase[1], "accept_compact": phase[2]},
                    "note": "after a fresh prefill: per-step CUDA events around replayed msd_step "
                            f"({K_prof} steps after 3 warm-up); phases from {K_prof} steps run as separate "
                            "calls (msd_draft_tree, msd_verify, msd_accept_compact)"}

    # ---- compaction worst case: a planted chain of the target's own argmax
    # tokens (grown by verifying it one node at a time), accepted in full (a = D)
    worst = None
    if B == 1:
        chain_tree = msd.Tree(B, N)
        toks, par = [int(eng.state()["root"].cpu()[0])], [-1]
        eng.draft_tree()                  # keeps the draft cache caught up
        for d in range(D):
            eng.plant(chain_tree, 0, toks, par)
            eng.verify(tree=chain_tree)
            toks.append(int(eng.argmax[d].cpu()))
            par.append(d)
        eng.plant(chain_tree, 0, toks, par)
        eng.verify(tree=chain_tree)
        torch.cuda.synchronize()
        e0.record(stream)
        eng.accept_compact(tree=chain_tree)
        e1.record(stream)
        torch.cuda.synchronize()
        worst = {"accept_len": int(eng.accept_len.cpu()[0]), "accept_compact_ms": e0.elapsed_time(e1),
                 "note": "msd_accept_compact on a planted chain of the target's argmax tokens "
                         "(D + 1 positions compacted in every layer), one call timed with CUDA events"}

    # ---- speculative sampling at T = 1 (Eq. 6 over the tree): msd_step_sample,
    # a replayed graph of draft, verify and the sampling walk + compaction; the
    # uniforms are inputs, copied device to device into the step's buffer
    sampling = None
    if not args.no_sampling:
        K_s, T_s = min(K, 32), 1.0
        shape = (B, D + 1, wl.topk + 1)
        g_u = torch.Generator(device="cuda").manual_seed(1234)
        u_all = torch.rand((K_s + 3,) + shape, device="cuda", generator=g_u)
        u_buf = torch.empty(shape, device="cuda")
        for i in range(3):
            u_buf.copy_(u_all[i])
            eng.step_sample(T_s, u_buf)
        torch.cuda.synchronize()
        Ls0 = eng.state()["seq_len"].cpu().numpy().astype(np.int64)
        torch.cuda.nvtx.range_push("timed_sample")
        e0.record(stream)
        for i in range(K_s):
            u_buf.copy_(u_all[3 + i], non_blocking=True)
            eng.step_sample(T_s, u_buf)
        e1.record(stream)
        torch.cuda.nvtx.range_pop()
        torch.cuda.synchronize()
        ms_s = e0.elapsed_time(e1)
        Ls1 = eng.state()["seq_len"].cpu().numpy().astype(np.int64)
        tok_s = int((Ls1 - Ls0).sum())
        sampling = {"temperature": T_s, "steps": K_s, "ms_per_step": ms_s / K_s,
                    "steps_per_s": world * K_s / (ms_s / 1e3), "tokens_per_s": world * tok_s / (ms_s / 1e3),
                    "tau": tok_s / (K_s * B),
                    "note": "msd_step_sample: draft tree, verify, speculative sampling over the tree "
                            "(Eq. 6, top-k candidates as point-mass proposals) and compaction, one replayed "
                            "graph per step after 3 warm-up steps; uniforms copied into its buffer before "
                            "each step (inside the timed region)"}

    # ---- chain drafts (top-1 per depth, N = D + 1): the drafting mode of the
    # paper's n-alpha, and Eq. 9 in its own terms: gamma T_q + T_v(gamma) per
    # cycle, omega(gamma, alpha) tokens per cycle
    chain = None
    if not args.no_chain:
        from paper_2505_14260_gb300 import metrics
        wl_c = wl.with_(topk=1, tree_nodes=D + 1)
        K_c = min(K, 32)
        ce = msd.Engine(msd.make_config(wl_c, wl.max_prompt + (2 * K_c + 8) * (D + 1) + 16), weights)
        ce.prefill(ids, lens, vis, offs)
        for _ in range(3):
            ce.step()
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(K_c):
            ce.step()
        e1.record(stream)
        torch.cuda.synchronize()
        t_cycle = e0.elapsed_time(e1) / K_c
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        ph = [0.0, 0.0, 0.0]
        alens = []
        for _ in range(K_c):                # the same step as separate calls, per phase
            ev[0].record(stream)
            ce.draft_tree()
            ev[1].record(stream)
            ce.verify()
            ev[2].record(stream)
            ce.accept_compact()
            ev[3].record(stream)
            torch.cuda.synchronize()
            for i in range(3):
                ph[i] += ev[i].elapsed_time(ev[i + 1]) / K_c
            alens += [int(x) for x in ce.accept_len.cpu().tolist()]
        ce.close()
        alpha = metrics.acceptance_rate(alens, D)
        chain = {"gamma": D, "ms_per_cycle": t_cycle, "t_q_ms": ph[0] / D, "t_v_ms": ph[1],
                 "accept_compact_ms": ph[2], "n_alpha": metrics.n_alpha(alens, D), "alpha": alpha,
                 "tau": metrics.tau(alens),
                 "note": f"N={D + 1}, k=1 context on the same weights; cycle = replayed msd_step over {K_c} "
                         "steps after 3 warm-up; T_q = msd_draft_tree time / gamma and T_v(gamma) = "
                         f"msd_verify time from {K_c} steps run as separate calls (CUDA events)"}
        if speedup is not None and alpha is not None:
            chain["sr_eq9"] = metrics.speedup_ratio(PAPER_OUTPUT_LEN, speedup["ar_ms_per_token"],
                                                    speedup["prefill_ms"], t_cycle, metrics.omega(D, alpha))

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        try:
            sample = OracleSample(wl, weights, prompts)
            est = [sample.step_seconds()]
            if est[0] < 10.0:
                est.append(sample.step_seconds())
            cpu = {"value": 1.0 / statistics.mean(est), "unit": "steps/s", "cores": sample.cores,
                   "kind": "oracle", "sample": sample.describe() + f"; mean of {len(est)} step(s)"}
        except Exception as ex:           # the bench line must still print
            cpu = {"value": None, "unit": "steps/s", "cores": None, "kind": "oracle",
                   "sample": f"failed: {ex!r}"}
        if cpu.get("value") and wl.name == "tiny":
            cpu["one_thread"] = oracle_one_thread(wl.name)



    if rank == 0:
        line = {
            "metric": METRIC, "value": steps_s, "unit": "steps/s", "n_gpus": world, "steps": K,
            "warmup": W, "ms_per_step": ms_max / K, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded random-init weights and prompts of the workload's shapes)",
            "config": {"workload": wl.name, "batch": B, "layers": wl.n_layers, "hidden": wl.hidden,
                       "vocab": V, "prompt": f"{wl.n_sys} text + {wl.n_vis} visual + rest text, "
                                             f"{int(L0.mean())} tokens at the timed start",
                       "tree": f"N={N} D={D} k={wl.topk}", "parallelism": f"replicas x{world}",
                       "draft_input": wl.draft_input,
                       "l2": "inputs larger than L2 (weights streamed every step)"},
            "tokens_per_s": world * tokens / (ms / 1e3),
            "tau": tokens / (K * B),
            "roofline": dict(roof, **{
                "traffic": gemm_traffic(roof["bytes_per_launch"], roof["bound"]),
                "kernel": "gemm_cluster_kernel / gemm_persist_kernel (tcgen05 bf16 GEMMs: 128-row weight "
                          "tiles x token rows, TMA-staged, TMEM accumulators, fused epilogues; all "
                          "projections and LM heads of the step)",
                "measured": f"%globaltimer stamps of every GEMM launch inside the replayed step graph, "
                            f"{prof['windows']} steps right after the timed region; a launch lasts from "
                            "its first return from the wait on the previous kernel to its last CTA's exit "
                            "(disjoint spans, summed per step)",
                "stamped_ms_per_step": ms_stamped}),
            "step_roofline": {"bytes_per_step": sb, "parts": parts, "achieved_gbs": step_gbs,
                              "frac": step_gbs / hbm, "peak": hbm, "peak_kind": peak_kind,
                              "frac_nominal": step_gbs / NOMINAL_HBM_GBS,
                              "gemm_tflops_over_step": (prof["gemm_flops"] / max(prof["windows"], 1))
                              / (ms / K / 1e3) / 1e12,
                              "note": "weights once per dependent pass + KV read at 2 bytes per "
                                      "element (the split caches' lo planes, as many bytes again, "
                                      "are not counted)"},
            "cpu_baseline": cpu,
            "e2e": e2e,
            "speedup": speedup,
            "distribution": distribution,
            "compaction_worst_case": worst,
            "sampling": sampling,
            "chain": chain,
            "gpu_launches": int(launches1 - launches0),
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    eng.close()


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.gemm:
        run_gemm_case(args)
        return
    import torch
    import torch.distributed as dist
    if world > 1:
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    try:
        run_msd(args, rank, world, local_rank)
    finally:
        if world > 1:
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
