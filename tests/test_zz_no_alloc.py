"""The allocation-free GEMM entry point (msd_linear_noalloc).

It serves callers that cannot allocate device memory: a host program whose
device memory is all owned by its own pool allocator, code running where an
allocation would synchronise the device or is not permitted, or a plug-in that
is handed buffers but no allocator. Its split-K scratch is a static device
array inside the library instead of context memory.

The test calls it through the C ABI twice in a row (the array keeps the last
call's contents, so the second call must not be disturbed by the first) and
compares each result with the context entry point msd_linear on the same
inputs, within the GEMM tolerance used by the other GPU tests. It also checks
that a shape whose scratch would not fit the array is refused. It runs last in
the suite and also passes on its own in a fresh process.
"""
import ctypes

import pytest
import torch

from paper_2505_14260_gb300 import build, msd, synth
from tests.gpu_support import open_engine

pytestmark = pytest.mark.gpu


def _noalloc(x, w, y, accumulate=False):
    stream = torch.cuda.current_stream().cuda_stream
    return msd.lib().msd_linear_noalloc(x.data_ptr(), x.stride(0), x.shape[0], x.shape[1],
                                        w.data_ptr(), w.shape[0], y.data_ptr(), y.stride(0),
                                        int(accumulate), ctypes.c_void_p(stream))


def test_noalloc_linear_matches_context_linear_on_two_calls():
    build.build()
    wl = synth.WORKLOADS["tiny"].with_(dtype="bf16")
    eng, _ = open_engine(wl)
    g = torch.Generator(device="cuda").manual_seed(11)
    # decode-shaped products; each splits K (8 to 16 ways), so the scratch is in use
    for (M, K, O) in [(60, 4096, 1024), (7, 512, 256), (16, 688, 384)]:
        xs = [torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16) for _ in range(2)]
        w = (torch.randn(O, K, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
        for call, x in enumerate(xs):              # two calls in a row, different inputs
            y_ref = torch.zeros(M, O, device="cuda")
            eng.linear(x, w, y_ref)
            y = torch.full((M, O), float("nan"), device="cuda")
            assert _noalloc(x, w, y) == msd.MSD_OK
            torch.cuda.synchronize()
            scale = max(1.0, y_ref.abs().max().item())
            err = (y - y_ref).abs().max().item()
            assert err <= 1e-4 * scale, (M, K, O, call, err)
        y2 = y.clone()
        assert _noalloc(xs[-1], w, y2, accumulate=True) == msd.MSD_OK
        torch.cuda.synchronize()
        assert (y2 - 2 * y_ref).abs().max().item() <= 2e-4 * scale
    eng.close()


def test_noalloc_linear_refuses_shapes_beyond_its_scratch():
    build.build()
    M, K, O = 256, 8192, 2048       # 9-way split-K partials of 18 MiB > the 16 MiB array
    x = torch.zeros(M, K, device="cuda", dtype=torch.bfloat16)
    w = torch.zeros(O, K, device="cuda", dtype=torch.bfloat16)
    y = torch.zeros(M, O, device="cuda")
    assert _noalloc(x, w, y) == msd.MSD_ERR_CAPACITY
    assert _noalloc(x[:, :12], w[:, :12], y) == msd.MSD_ERR_INVALID   # k not a multiple of 8
