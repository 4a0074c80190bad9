"""The C-ABI library builds for sm_103a, loads, and exports every entry point
declared in include/msd.h; argument validation that needs no GPU works."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libmsd():
    from paper_2505_14260_gb300 import build, msd
    build.build()
    return msd.lib()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "msd.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(msd_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for n in ["msd_create", "msd_prefill", "msd_draft_tree", "msd_verify", "msd_accept_compact"]:
        assert n in names


def test_library_exports_every_declared_symbol(libmsd):
    for n in declared_symbols():
        assert hasattr(libmsd, n), n


def test_create_rejects_bad_configs_before_touching_the_gpu(libmsd):
    from paper_2505_14260_gb300 import msd, synth
    ctx = ctypes.c_void_p()
    assert libmsd.msd_create(None, None, ctypes.byref(ctx)) == msd.MSD_ERR_INVALID
    wl = synth.WORKLOADS["tiny"]
    good = msd.make_config(wl, 256)
    w = msd.msd_weights()
    cases = [dict(head_dim=96), dict(n_heads=3), dict(topk=0), dict(topk=17),
             dict(tree_nodes=300), dict(tree_depth=0), dict(max_batch=0), dict(dtype=7),
             dict(tree_nodes=64, tree_depth=2, topk=2),     # k + (D-1)k^2 = 6 < 63
             dict(draft_input=3), dict(draft_input=-1)]
    for kw in cases:
        cfg = msd.make_config(wl, 256)
        for k, v in kw.items():
            setattr(cfg, k, v)
        assert libmsd.msd_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(ctx)) == \
            msd.MSD_ERR_INVALID, kw
    # a valid config with null weights is rejected too
    assert libmsd.msd_create(ctypes.byref(good), ctypes.byref(w), ctypes.byref(ctx)) == \
        msd.MSD_ERR_INVALID


def test_null_context_calls_fail_cleanly(libmsd):
    from paper_2505_14260_gb300 import msd
    assert libmsd.msd_last_error(None) == b"null context"
    assert libmsd.msd_destroy(None) == msd.MSD_OK
    assert libmsd.msd_verify(None, None, None, None, None) == msd.MSD_ERR_INVALID
    assert libmsd.msd_state(None, None) == msd.MSD_ERR_INVALID


def test_binding_fails_loudly_without_the_library(tmp_path, monkeypatch):
    from paper_2505_14260_gb300 import msd
    monkeypatch.setattr(msd, "_LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(msd, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        msd.lib()


def test_tree_set_nodes_copies_tokens_and_parents_only():
    """The binding only copies a planted tree's tokens and parent links (and its
    node count); depths and masks are derived by the library
    (msd_tree_complete, tested on the GPU)."""
    from paper_2505_14260_gb300 import msd
    N = 70
    t = msd.Tree(2, N, device="cpu")
    n = 66
    parent = [-1] + [(i - 1) // 2 for i in range(1, n)]
    t.set_nodes(1, list(range(100, 100 + n)), parent)
    assert t.tokens[N:2 * N].tolist() == list(range(100, 100 + n)) + [0] * (N - n)
    assert t.parent[N:2 * N].tolist() == parent + [-1] * (N - n)
    assert int(t.n_nodes[1]) == n and int(t.n_nodes[0]) == N
    assert t.parent[:N].tolist() == [-1] * N              # request 0 untouched
    assert not t.depth.any() and not t.mask.any()         # left to the library
    with pytest.raises(ValueError):
        t.set_nodes(0, [1, 2], [-1])                      # one parent entry per node
    with pytest.raises(ValueError):
        t.set_nodes(0, list(range(N + 1)), [-1] * (N + 1))


def _header_struct_fields(name):
    import re
    text = open(os.path.join(ROOT, "include", "msd.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    body = re.search(r"typedef struct\s*\{([^}]*)\}\s*" + name + r"\s*;", text, flags=re.S).group(1)
    fields = []
    for decl in body.split(";"):
        decl = decl.strip()
        if decl:
            fields += [n.strip().lstrip("*") for n in decl.split(None, 1)[1].split(",")]
    return fields


@pytest.mark.parametrize("cname,pyname", [("msd_profile", "msd_profile"), ("msd_state_view", "msd_state_view"),
                                          ("msd_kernel_slot", "msd_kernel_slot")])
def test_binding_structs_match_the_header(cname, pyname):
    """The ctypes mirrors of the header's output structs list the same fields
    in the same order (the library writes them by position)."""
    from paper_2505_14260_gb300 import msd
    assert [f for f, _ in getattr(msd, pyname)._fields_] == _header_struct_fields(cname)


def test_profile_enable_rejects_a_null_context(libmsd):
    from paper_2505_14260_gb300 import msd
    assert libmsd.msd_profile_enable(None, 2) == msd.MSD_ERR_INVALID


def test_profile_slots_rejects_bad_arguments(libmsd):
    import ctypes
    from paper_2505_14260_gb300 import msd
    n = ctypes.c_int32(7)
    assert libmsd.msd_profile_slots(None, None, 0, ctypes.byref(n)) == msd.MSD_ERR_INVALID
