"""Thin ctypes binding of the MSD C ABI (include/msd.h).

Argument marshalling only: every step of the decode path runs in the CUDA
library. PyTorch supplies device memory and the stream. Loading fails loudly
if the library has not been built (``python -m paper_2505_14260_gb300.build``);
there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_char_p, c_float, c_int32, c_int64, c_void_p

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmsd.so")

MSD_OK, MSD_ERR_INVALID, MSD_ERR_CAPACITY, MSD_ERR_OOM, MSD_ERR_CUDA, MSD_ERR_DEVICE = 0, -1, -2, -3, -4, -5
MSD_F32, MSD_BF16 = 0, 1
DRAFT_INPUTS = {"embedding": 0, "concat": 1, "feature": 2}     # MSD_DRAFT_*
STATUS_NAMES = {0: "MSD_OK", -1: "MSD_ERR_INVALID", -2: "MSD_ERR_CAPACITY", -3: "MSD_ERR_OOM",
                -4: "MSD_ERR_CUDA", -5: "MSD_ERR_DEVICE"}


class msd_config(ctypes.Structure):
    _fields_ = [("n_layers", c_int32), ("hidden", c_int32), ("n_heads", c_int32),
                ("head_dim", c_int32), ("ffn", c_int32), ("vocab", c_int32),
                ("rms_eps", c_float), ("rope_base", c_float), ("dtype", c_int32),
                ("max_batch", c_int32), ("max_seq", c_int32), ("tree_nodes", c_int32),
                ("tree_depth", c_int32), ("topk", c_int32), ("draft_input", c_int32)]


LAYER_FIELDS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "w_gate", "w_up", "w_down")


class msd_layer(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in LAYER_FIELDS]


class msd_weights(ctypes.Structure):
    _fields_ = [("embed", c_void_p), ("layers", POINTER(msd_layer)), ("final_norm", c_void_p),
                ("lm_head", c_void_p), ("draft", msd_layer), ("draft_fc", c_void_p)]


class msd_tree(ctypes.Structure):
    _fields_ = [("tokens", c_void_p), ("parent", c_void_p), ("depth", c_void_p),
                ("mask", c_void_p), ("n_nodes", c_void_p)]


class msd_draft_record(ctypes.Structure):
    _fields_ = [("logits", c_void_p), ("topk_ids", c_void_p), ("topk_logp", c_void_p)]


class msd_state_view(ctypes.Structure):
    _fields_ = [("target_kv", c_void_p), ("draft_kv", c_void_p), ("seq_len", c_void_p),
                ("n_pending", c_void_p), ("root", c_void_p), ("elem_bytes", c_int64),
                ("lo_offset", c_int64)]


class msd_profile(ctypes.Structure):
    _fields_ = [("kernel_launches", c_int64), ("gemm_launches", c_int64), ("gemm_ms", ctypes.c_double),
                ("gemm_bytes", ctypes.c_double), ("gemm_weight_bytes", ctypes.c_double),
                ("gemm_critical_ms", ctypes.c_double), ("windows", c_int64),
                ("gemm_flops", ctypes.c_double), ("gemm_mma_flops", ctypes.c_double),
                ("gemm_prefetch_bytes", ctypes.c_double)]


class msd_kernel_slot(ctypes.Structure):
    _fields_ = [("kind", c_int32), ("rows", c_int32), ("outputs", c_int32), ("inner", c_int32),
                ("launches", c_int64), ("bytes", ctypes.c_double), ("critical_ms", ctypes.c_double),
                ("span_ms", ctypes.c_double)]


_SIGNATURES = {
    "msd_create": (c_int32, [POINTER(msd_config), POINTER(msd_weights), POINTER(c_void_p)]),
    "msd_destroy": (c_int32, [c_void_p]),
    "msd_prefill": (c_int32, [c_void_p, c_int32, POINTER(c_int32), c_void_p, c_int32, c_void_p,
                              POINTER(c_int64), c_void_p, c_void_p]),
    "msd_draft_tree": (c_int32, [c_void_p, POINTER(msd_tree), POINTER(msd_draft_record), c_void_p]),
    "msd_verify": (c_int32, [c_void_p, POINTER(msd_tree), c_void_p, c_void_p, c_void_p]),
    "msd_accept_compact": (c_int32, [c_void_p, POINTER(msd_tree), c_void_p, c_void_p, c_void_p,
                                     c_void_p, c_void_p, c_void_p]),
    "msd_accept_sample": (c_int32, [c_void_p, POINTER(msd_tree), c_void_p, c_float, c_void_p,
                                    c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
    "msd_step": (c_int32, [c_void_p, POINTER(msd_tree), c_void_p, c_void_p, c_void_p, c_void_p,
                           c_void_p]),
    "msd_step_sample": (c_int32, [c_void_p, POINTER(msd_tree), c_float, c_void_p, c_void_p, c_void_p,
                                  c_void_p, c_void_p, c_void_p]),
    "msd_ar_step": (c_int32, [c_void_p, c_void_p, c_void_p]),
    "msd_linear": (c_int32, [c_void_p, c_void_p, c_int32, c_int32, c_int32, c_void_p, c_int32,
                             c_void_p, c_int32, c_int32, c_void_p]),
    "msd_linear_noalloc": (c_int32, [c_void_p, c_int32, c_int32, c_int32, c_void_p, c_int32,
                                     c_void_p, c_int32, c_int32, c_void_p]),
    "msd_tree_complete": (c_int32, [c_void_p, POINTER(msd_tree), c_int32, c_void_p]),
    "msd_test_wait_timeout": (c_int32, [c_void_p, c_int64, c_void_p]),
    "msd_profile_enable": (c_int32, [c_void_p, c_int32]),
    "msd_profile_read": (c_int32, [c_void_p, POINTER(msd_profile)]),
    "msd_profile_slots": (c_int32, [c_void_p, POINTER(msd_kernel_slot), c_int32, POINTER(c_int32)]),
    "msd_state": (c_int32, [c_void_p, POINTER(msd_state_view)]),
    "msd_last_error": (c_char_p, [c_void_p]),
}

_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it is missing (no fallback path exists)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"MSD CUDA library not built: {_LIB_PATH} is missing "
                               "(run python -m paper_2505_14260_gb300.build)")
        L = ctypes.CDLL(_LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


class MsdError(RuntimeError):
    def __init__(self, status: int, call: str, msg: str):
        super().__init__(f"{call} -> {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int:
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


class _DevArray:
    """Exposes a raw device pointer to torch.as_tensor (no copy)."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (ptr, False), "version": 3}


def device_view(ptr: int, shape, dtype: torch.dtype) -> torch.Tensor:
    typestr = {torch.int32: "<i4", torch.float32: "<f4", torch.int16: "<i2"}[
        torch.int16 if dtype == torch.bfloat16 else dtype]
    t = torch.as_tensor(_DevArray(ptr, shape, typestr), device="cuda")
    return t.view(torch.bfloat16) if dtype == torch.bfloat16 else t


class Tree:
    """Caller-owned device tree arrays in the layout of include/msd.h."""

    def __init__(self, B: int, N: int, device="cuda"):
        self.B, self.N, self.W = B, N, (N + 63) // 64
        self.tokens = torch.zeros(B * N, dtype=torch.int32, device=device)
        self.parent = torch.full((B * N,), -1, dtype=torch.int32, device=device)
        self.depth = torch.zeros(B * N, dtype=torch.int32, device=device)
        self.mask = torch.zeros(B * N * self.W, dtype=torch.int64, device=device)
        self.n_nodes = torch.full((B,), N, dtype=torch.int32, device=device)

    def c(self) -> msd_tree:
        return msd_tree(_ptr(self.tokens), _ptr(self.parent), _ptr(self.depth), _ptr(self.mask),
                        _ptr(self.n_nodes))

    def set_nodes(self, b: int, tokens, parent):
        """Writes the tokens and parent links of request b (n <= N nodes, node 0
        the root; the rest padded). Depths and ancestor masks are derived by the
        library: Engine.plant (msd_tree_complete)."""
        n = len(tokens)
        if n < 1 or n > self.N or len(parent) != n:
            raise ValueError("a tree needs 1..N nodes and one parent entry per node")
        pad = self.N - n
        sl = slice(b * self.N, (b + 1) * self.N)
        dev = self.tokens.device
        self.tokens[sl] = torch.tensor(list(tokens) + [0] * pad, dtype=torch.int32, device=dev)
        self.parent[sl] = torch.tensor(list(parent) + [-1] * pad, dtype=torch.int32, device=dev)
        self.n_nodes[b] = n


class Engine:
    """One context of the C ABI plus the caller-owned buffers of a step."""

    def __init__(self, cfg: msd_config, weights: dict):
        self.cfg = cfg
        self.w = weights             # keeps the borrowed device tensors alive
        L = lib()
        self._layers = (msd_layer * cfg.n_layers)(
            *[msd_layer(*[_ptr(lw[n]) for n in LAYER_FIELDS]) for lw in weights["layers"]])
        d = weights["draft"]
        self._weights = msd_weights(_ptr(weights["embed"]), self._layers, _ptr(weights["final_norm"]),
                                    _ptr(weights["lm_head"]),
                                    msd_layer(*[_ptr(d[n]) for n in LAYER_FIELDS]),
                                    _ptr(weights["draft_fc"]))
        ctx = c_void_p()
        st = L.msd_create(ctypes.byref(cfg), ctypes.byref(self._weights), ctypes.byref(ctx))
        if st != MSD_OK:
            raise MsdError(st, "msd_create", "invalid configuration or allocation failure")
        self.ctx = ctx
        B, N, D = cfg.max_batch, cfg.tree_nodes, cfg.tree_depth
        self.tree = Tree(B, N)
        self.argmax = torch.zeros(B * N, dtype=torch.int32, device="cuda")
        self.path = torch.zeros(B * (D + 1), dtype=torch.int32, device="cuda")
        self.accept_len = torch.zeros(B, dtype=torch.int32, device="cuda")
        self.bonus = torch.zeros(B, dtype=torch.int32, device="cuda")
        self.index_map = torch.zeros(B * (D + 1), dtype=torch.int32, device="cuda")
        self.root_out = torch.zeros(B, dtype=torch.int32, device="cuda")

    def close(self):
        if getattr(self, "ctx", None) is not None and self.ctx.value:
            lib().msd_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _check(self, st: int, call: str):
        if st != MSD_OK:
            msg = lib().msd_last_error(self.ctx)
            raise MsdError(st, call, msg.decode() if msg else "")

    # -- the five calls ------------------------------------------------------
    def prefill(self, ids: torch.Tensor, lengths, vis: torch.Tensor | None, vis_off, stream=None):
        """ids: int32 [B, stride] on the device (-1 = visual slot)."""
        B = len(lengths)
        lens = (c_int32 * B)(*[int(x) for x in lengths])
        offs = (c_int64 * B)(*[int(x) for x in vis_off])
        st = lib().msd_prefill(self.ctx, B, lens, _ptr(ids), ids.shape[1], _ptr(vis), offs,
                               _ptr(self.root_out), _stream(stream))
        self._check(st, "msd_prefill")
        return self.root_out

    def draft_tree(self, record: dict | None = None, tree: Tree | None = None, stream=None):
        t = self.tree if tree is None else tree
        rec = None
        if record is not None:
            rec = msd_draft_record(_ptr(record.get("logits")), _ptr(record.get("topk_ids")),
                                   _ptr(record.get("topk_logp")))
        st = lib().msd_draft_tree(self.ctx, ctypes.byref(t.c()),
                                  ctypes.byref(rec) if rec is not None else None, _stream(stream))
        self._check(st, "msd_draft_tree")
        return t

    def verify(self, tree: Tree | None = None, logits: torch.Tensor | None = None, stream=None):
        t = self.tree if tree is None else tree
        st = lib().msd_verify(self.ctx, ctypes.byref(t.c()), _ptr(self.argmax), _ptr(logits),
                              _stream(stream))
        self._check(st, "msd_verify")
        return self.argmax

    def accept_compact(self, tree: Tree | None = None, stream=None):
        t = self.tree if tree is None else tree
        st = lib().msd_accept_compact(self.ctx, ctypes.byref(t.c()), _ptr(self.argmax),
                                      _ptr(self.path), _ptr(self.accept_len), _ptr(self.bonus),
                                      _ptr(self.index_map), _stream(stream))
        self._check(st, "msd_accept_compact")
        return self.path, self.accept_len, self.bonus

    def accept_sample(self, temperature: float, u: torch.Tensor, logits: torch.Tensor | None = None,
                      tree: Tree | None = None, stream=None):
        """Speculative sampling at temperature T > 0 + compaction (msd_accept_sample).
        u: fp32 [B, D+1, k+1] uniforms on the device; logits: the tensor given to
        verify(), or None if verify() kept them in the context."""
        t = self.tree if tree is None else tree
        st = lib().msd_accept_sample(self.ctx, ctypes.byref(t.c()), _ptr(logits), float(temperature),
                                     _ptr(u), _ptr(self.path), _ptr(self.accept_len), _ptr(self.bonus),
                                     _ptr(self.index_map), _stream(stream))
        self._check(st, "msd_accept_sample")
        return self.path, self.accept_len, self.bonus

    def step_sample(self, temperature: float, u: torch.Tensor, stream=None):
        """draft -> verify -> sample/compact at temperature T as one replayed
        CUDA graph (msd_step_sample); u is read when the step runs."""
        st = lib().msd_step_sample(self.ctx, ctypes.byref(self.tree.c()), float(temperature), _ptr(u),
                                   _ptr(self.argmax), _ptr(self.path), _ptr(self.accept_len),
                                   _ptr(self.bonus), _stream(stream))
        self._check(st, "msd_step_sample")
        return self.path, self.accept_len, self.bonus

    def step(self, stream=None):
        """draft -> verify -> accept/compact as one replayed CUDA graph (msd_step)."""
        st = lib().msd_step(self.ctx, ctypes.byref(self.tree.c()), _ptr(self.argmax),
                            _ptr(self.path), _ptr(self.accept_len), _ptr(self.bonus),
                            _stream(stream))
        self._check(st, "msd_step")
        return self.path, self.accept_len, self.bonus

    def step_calls(self, stream=None):
        """The same step as three separate calls (no graph)."""
        self.draft_tree(stream=stream)
        self.verify(stream=stream)
        return self.accept_compact(stream=stream)

    def ar_step(self, out: torch.Tensor | None = None, stream=None):
        """One plain greedy decode step (msd_ar_step): the next token of every request."""
        if out is None:
            if getattr(self, "_ar_out", None) is None:
                self._ar_out = torch.zeros(self.cfg.max_batch, dtype=torch.int32, device="cuda")
            out = self._ar_out
        st = lib().msd_ar_step(self.ctx, _ptr(out), _stream(stream))
        self._check(st, "msd_ar_step")
        return out

    def linear(self, x: torch.Tensor, w: torch.Tensor, y: torch.Tensor, accumulate=False,
               stream=None):
        """y (=|+=) x @ w.T through the library's GEMM (x, w in the model dtype)."""
        st = lib().msd_linear(self.ctx, _ptr(x), x.stride(0), x.shape[0], x.shape[1], _ptr(w),
                              w.shape[0], _ptr(y), y.stride(0), int(accumulate), _stream(stream))
        self._check(st, "msd_linear")
        return y

    def plant(self, tree: Tree, b: int, tokens, parent, stream=None):
        """A caller-planted tree for request b: tokens and parent links are
        copied, depths and ancestor masks derived on the device
        (msd_tree_complete; a parent that does not precede its node is reported
        by the next call as MSD_ERR_DEVICE)."""
        tree.set_nodes(b, tokens, parent)
        st = lib().msd_tree_complete(self.ctx, ctypes.byref(tree.c()), int(b), _stream(stream))
        self._check(st, "msd_tree_complete")
        return tree

    def test_wait_timeout(self, limit_ns: int, stream=None):
        """Test hook: a bounded wait that runs out and sets the status word."""
        st = lib().msd_test_wait_timeout(self.ctx, int(limit_ns), _stream(stream))
        self._check(st, "msd_test_wait_timeout")

    def profile_enable(self, mode=True):
        """0/False off, 1/True CUDA events around separate launches, 2 launch
        stamps inside the replayed step graphs."""
        self._check(lib().msd_profile_enable(self.ctx, int(mode)), "msd_profile_enable")

    def profile_read(self) -> dict:
        p = msd_profile()
        self._check(lib().msd_profile_read(self.ctx, ctypes.byref(p)), "msd_profile_read")
        return {n: getattr(p, n) for n, _ in msd_profile._fields_}

    def profile_slots(self, max_slots: int = 4096) -> list:
        """Per-launch sums of the stamped step graphs since the last call
        (mode 2): GEMM slots in launch order, then the attention launches."""
        buf = (msd_kernel_slot * max_slots)()
        n = c_int32(0)
        self._check(lib().msd_profile_slots(self.ctx, buf, max_slots, ctypes.byref(n)), "msd_profile_slots")
        return [{f: getattr(buf[i], f) for f, _ in msd_kernel_slot._fields_} for i in range(n.value)]

    # -- state ---------------------------------------------------------------
    def state(self) -> dict:
        v = msd_state_view()
        self._check(lib().msd_state(self.ctx, ctypes.byref(v)), "msd_state")
        c = self.cfg
        dt = torch.bfloat16 if c.dtype == MSD_BF16 else torch.float32
        B, nh, S, hd = c.max_batch, c.n_heads, c.max_seq, c.head_dim
        out = {
            "target_kv": device_view(v.target_kv, (c.n_layers, 2, B, nh, S, hd), dt),
            "draft_kv": device_view(v.draft_kv, (2, B, nh, S, hd), dt),
            "seq_len": device_view(v.seq_len, (B,), torch.int32),
            "n_pending": device_view(v.n_pending, (B,), torch.int32),
            "root": device_view(v.root, (B,), torch.int32),
            "lo_offset": int(v.lo_offset),
        }
        if v.lo_offset:     # bf16: the lo planes of the split cache entries
            eb = int(v.elem_bytes)
            out["target_kv_lo"] = device_view(v.target_kv + v.lo_offset * eb, (c.n_layers, 2, B, nh, S, hd), dt)
            out["draft_kv_lo"] = device_view(v.draft_kv + v.lo_offset * eb, (2, B, nh, S, hd), dt)
        return out


def make_config(wl, max_seq: int, batch: int | None = None) -> msd_config:
    """msd_config of a synth.Workload."""
    return msd_config(n_layers=wl.n_layers, hidden=wl.hidden, n_heads=wl.n_heads,
                      head_dim=wl.head_dim, ffn=wl.ffn, vocab=wl.vocab, rms_eps=wl.rms_eps,
                      rope_base=wl.rope_base,
                      dtype=MSD_BF16 if wl.dtype == "bf16" else MSD_F32,
                      max_batch=wl.batch if batch is None else batch, max_seq=max_seq,
                      tree_nodes=wl.tree_nodes, tree_depth=wl.tree_depth, topk=wl.topk,
                      draft_input=DRAFT_INPUTS[wl.draft_input])


def upload_prompts(prompts, device="cuda"):
    """Packs synth prompts into the msd_prefill layout: ids [B, stride] int32,
    lengths, concatenated visual rows and their per-request offsets."""
    B = len(prompts)
    stride = max(p.length for p in prompts)
    ids = torch.full((B, stride), 0, dtype=torch.int32)
    vis_rows, offs, off = [], [], 0
    for b, p in enumerate(prompts):
        ids[b, :p.length] = torch.from_numpy(p.ids)
        offs.append(off)
        vis_rows.append(p.vis)
        off += p.vis.shape[0]
    vis = torch.cat(vis_rows, 0).to(device) if off > 0 else None
    return ids.to(device), [p.length for p in prompts], vis, offs
