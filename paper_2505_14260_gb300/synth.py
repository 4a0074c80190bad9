"""Seeded synthetic workloads for the MSD decode step.

This module only draws random numbers and shapes them; it holds none of the
method's arithmetic. It is the one piece shared by the CUDA path's tests and
bench and by the oracle harness: both sides receive the very same arrays.

Recipe (shapes from the paper's LLaVA-1.5 setting, Sec. 3.1 and Sec. 5.1; the
paper's benchmark images and trained weights are not available, so seeded
random tensors of the same shapes stand in for them):

* Matrices ~ N(0, 0.02), drawn in a fixed order: embed, then per target layer
  wq, wk, wv, wo, w_gate, w_up, w_down, then lm_head, then the draft layer's
  seven matrices, then draft_fc. RMSNorm gains are drawn afterwards as
  1 + 0.1 * N(0, 1) (target layers in order, final norm, draft layer), so that a
  misapplied gain shows in parity tests.
* bf16 workloads round every weight to bf16 (round-to-nearest-even); the oracle
  reads the rounded values upcast, so weights are identical on both sides.
* Prompts follow the interleaved layout of Eq. 3: ``n_sys`` text tokens, then the
  visual embeddings, then the remaining text tokens. Text ids ~ U[0, V);
  visual embeddings ~ 0.5 * N(0, 1) (rounded to the workload dtype). A visual
  slot is marked by id -1 and the visual rows are consumed in order.
* Prompts use their own CPU generator seeded from the workload seed, so the
  same prompt is produced whichever device the weights are drawn on.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass, field

import numpy as np
import torch

MATRIX_STD = 0.02
NORM_JITTER = 0.1
VISUAL_SCALE = 0.5


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    hidden: int
    n_heads: int
    head_dim: int
    ffn: int
    vocab: int
    tree_nodes: int          # N, including the root
    tree_depth: int          # D, number of draft passes
    topk: int                # k
    batch: int
    n_vis: tuple             # per-request visual-token count choices
    n_text: tuple            # (lo, hi) inclusive range of text-token counts
    n_sys: int               # text tokens placed before the image (Eq. 3)
    seed: int
    steps: int
    dtype: str               # "f32" or "bf16"
    rms_eps: float = 1e-6
    rope_base: float = 10000.0
    draft_input: str = "embedding"   # visual draft input: "embedding" (MSD), "concat", "feature"

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def max_prompt(self) -> int:
        return max(self.n_vis) + self.n_text[1]

    def max_seq(self, steps: int | None = None) -> int:
        s = self.steps if steps is None else steps
        return self.max_prompt + s * (self.tree_depth + 1) + self.tree_nodes + 8


_7B = dict(n_layers=32, hidden=4096, n_heads=32, head_dim=128, ffn=11008,
           vocab=32000, tree_nodes=60, tree_depth=6, topk=10)

WORKLOADS = {
    # Tiny reference model; compared against the oracle on every step.
    "tiny": Workload("tiny", n_layers=2, hidden=256, n_heads=4, head_dim=64,
                     ffn=688, vocab=1024, tree_nodes=16, tree_depth=4, topk=4,
                     batch=1, n_vis=(64,), n_text=(32, 32), n_sys=0, seed=0,
                     steps=8, dtype="f32"),
    # LLaVA-1.5-7B shape, 576 visual tokens + 64 text ids.
    "llava7b": Workload("llava7b", batch=1, n_vis=(576,), n_text=(64, 64),
                        n_sys=8, seed=1, steps=128, dtype="bf16", **_7B),
    # LLaVA-1.5-13B shape.
    "llava13b": Workload("llava13b", n_layers=40, hidden=5120, n_heads=40,
                         head_dim=128, ffn=13824, vocab=32000, tree_nodes=60,
                         tree_depth=6, topk=10, batch=1, n_vis=(576,),
                         n_text=(128, 128), n_sys=8, seed=2, steps=128,
                         dtype="bf16"),
    # Long multimodal prefix: 5 image tiles of 576 tokens + 512 text ids.
    "long7b": Workload("long7b", batch=1, n_vis=(2880,), n_text=(512, 512),
                       n_sys=8, seed=3, steps=256, dtype="bf16", **_7B),
    # Batched serving: 16 ragged requests.
    "batch16": Workload("batch16", batch=16, n_vis=(576, 1152),
                        n_text=(32, 512), n_sys=8, seed=4, steps=128,
                        dtype="bf16", **_7B),
}


def torch_dtype(wl: Workload) -> torch.dtype:
    return torch.float32 if wl.dtype == "f32" else torch.bfloat16


LAYER_MATS = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")
LAYER_NORMS = ("attn_norm", "mlp_norm")


def layer_shapes(wl: Workload) -> dict:
    H, F = wl.hidden, wl.ffn
    return {"wq": (H, H), "wk": (H, H), "wv": (H, H), "wo": (H, H),
            "w_gate": (F, H), "w_up": (F, H), "w_down": (H, F)}


def make_weights(wl: Workload, device="cpu", layers: int | None = None) -> dict:
    """All model weights as tensors of the workload dtype on ``device``.

    Returns {"embed", "lm_head", "final_norm", "draft_fc",
             "layers": [ {name: tensor} * n_layers ], "draft": {name: tensor}}.
    Matrices are [out, in] row-major. With ``layers`` set, only the first
    ``layers`` decoder layers are kept (the others are still drawn, so every
    kept tensor equals its value in the full set).
    """
    device = torch.device(device)
    g = torch.Generator(device=device)
    g.manual_seed(wl.seed)
    dt = torch_dtype(wl)
    H, V = wl.hidden, wl.vocab

    def mat(shape):
        t = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
        t.mul_(MATRIX_STD)
        return t.to(dt)

    def gain():
        t = torch.randn((H,), generator=g, device=device, dtype=torch.float32)
        return (1.0 + NORM_JITTER * t).to(dt)

    shapes = layer_shapes(wl)
    keep = wl.n_layers if layers is None else min(layers, wl.n_layers)
    w = {"embed": mat((V, H)), "layers": []}
    for i in range(wl.n_layers):
        lw = {n: mat(shapes[n]) for n in LAYER_MATS}
        if i < keep:
            w["layers"].append(lw)
        del lw
    w["lm_head"] = mat((V, H))
    w["draft"] = {n: mat(shapes[n]) for n in LAYER_MATS}
    w["draft_fc"] = mat((H, 2 * H))
    for i in range(wl.n_layers):
        g_ = {n: gain() for n in LAYER_NORMS}
        if i < keep:
            w["layers"][i].update(g_)
    w["final_norm"] = gain()
    for n in LAYER_NORMS:
        w["draft"][n] = gain()
    return w


@dataclass
class Prompt:
    ids: np.ndarray          # int32 [L]; -1 marks a visual slot
    vis: torch.Tensor        # [n_vis, H] in the workload dtype (CPU)

    @property
    def length(self) -> int:
        return int(self.ids.shape[0])


def make_prompts(wl: Workload) -> list:
    """One prompt per request, laid out as Eq. 3 (text, image, text)."""
    g = torch.Generator().manual_seed(wl.seed * 1000003 + 17)
    dt = torch_dtype(wl)
    out = []
    for _ in range(wl.batch):
        if len(wl.n_vis) == 1:
            m = wl.n_vis[0]
        else:
            m = wl.n_vis[int(torch.randint(len(wl.n_vis), (1,), generator=g))]
        lo, hi = wl.n_text
        n = lo if lo == hi else int(torch.randint(lo, hi + 1, (1,), generator=g))
        text = torch.randint(0, wl.vocab, (n,), generator=g, dtype=torch.int64)
        vis = (VISUAL_SCALE * torch.randn((m, wl.hidden), generator=g)).to(dt)
        p = min(wl.n_sys, n - 1)
        ids = np.concatenate([text[:p].numpy(), np.full(m, -1, np.int64),
                              text[p:].numpy()]).astype(np.int32)
        out.append(Prompt(ids=ids, vis=vis))
    return out


def to_numpy_f32(t: torch.Tensor) -> np.ndarray:
    """Exact upcast of a (possibly bf16) tensor to a float32 numpy array."""
    return t.detach().to("cpu", torch.float32).numpy()


def weights_to_numpy(w: dict) -> dict:
    """The same weights as float32 numpy arrays (values unchanged)."""
    out = {k: to_numpy_f32(v) for k, v in w.items() if isinstance(v, torch.Tensor)}
    out["layers"] = [{k: to_numpy_f32(v) for k, v in lw.items()} for lw in w["layers"]]
    out["draft"] = {k: to_numpy_f32(v) for k, v in w["draft"].items()}
    return out
