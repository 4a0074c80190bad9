"""Helpers for the GPU tests: move synthetic weights to the device, open an
engine, and compare device outputs with the oracle."""
import numpy as np
import torch

from paper_2505_14260_gb300 import msd, synth

# Tolerances against the float64 oracle. bf16 workloads: the stated bound for
# the logits, max |d| <= 3e-2 and relative L2 <= 1e-2, at every width (the
# split-bf16 activations and caches carry each value to about 2^-17, so the
# measured errors sit orders of magnitude below it). fp32: float32 rounding of
# a float64 computation over two layers. KV caches (hi + lo of each entry for
# bf16): relative L2 <= 1e-3 -- a check of our own, not a stated bound.
TOL = {"f32": dict(max_abs=2e-4, rel_l2=1e-5), "bf16": dict(max_abs=3e-2, rel_l2=1e-2)}
KV_REL_L2 = {"f32": 1e-5, "bf16": 1e-3}


def to_device(w: dict, device="cuda") -> dict:
    out = {}
    for k, v in w.items():
        if k == "layers":
            out[k] = [{n: t.to(device) for n, t in lw.items()} for lw in v]
        elif k == "draft":
            out[k] = {n: t.to(device) for n, t in v.items()}
        else:
            out[k] = v.to(device)
    return out


def open_engine(wl, weights_cpu=None, steps=None, batch=None):
    w = synth.make_weights(wl) if weights_cpu is None else weights_cpu
    wd = to_device(w)
    cfg = msd.make_config(wl, wl.max_seq(steps), batch)
    return msd.Engine(cfg, wd), w


def rel_l2(a, b) -> float:
    a = np.asarray(a, np.float64); b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


def abs_bound(ref, tol) -> float:
    """The max |d| bound of a block (absolute)."""
    return tol["max_abs"]


def assert_close(gpu, ref, tol, what=""):
    gpu = np.asarray(gpu, np.float64); ref = np.asarray(ref, np.float64)
    d = float(np.max(np.abs(gpu - ref))) if gpu.size else 0.0
    r = rel_l2(gpu, ref)
    bound = abs_bound(ref, tol)
    assert d <= bound and r <= tol["rel_l2"], f"{what}: max|d|={d:.3e} (bound {bound:.3e}) relL2={r:.3e}"
    return d, r


def top2_margin(row) -> float:
    s = np.sort(np.asarray(row, np.float64))
    return float(s[-1] - s[-2])


def record_buffers(wl, B=None):
    B = wl.batch if B is None else B
    D, k, V = wl.tree_depth, wl.topk, wl.vocab
    return {"logits": torch.zeros(B, D, k, V, device="cuda"),
            "topk_ids": torch.zeros(B, D, k, k, dtype=torch.int32, device="cuda"),
            "topk_logp": torch.zeros(B, D, k, k, device="cuda")}


def tree_numpy(tree: msd.Tree, b: int):
    N = tree.N
    sl = slice(b * N, (b + 1) * N)
    toks = tree.tokens[sl].cpu().numpy().astype(np.int64)
    par = tree.parent[sl].cpu().numpy().astype(np.int64)
    dep = tree.depth[sl].cpu().numpy().astype(np.int64)
    mask = tree.mask.view(torch.int64)[b * N * tree.W:(b + 1) * N * tree.W].cpu().numpy()
    return toks, par, dep, mask.view(np.uint64).reshape(N, tree.W)


def plant(eng: msd.Engine, tree: msd.Tree, b: int, tokens, parent):
    """A caller-planted tree for request b (depths and masks derived by the
    library, msd_tree_complete)."""
    eng.plant(tree, b, [int(x) for x in tokens], [int(x) for x in parent])
