"""The allocation-free GEMM entry point (msd_linear_noalloc).

It serves callers that cannot allocate device memory: a host program whose
device memory is all owned by its own pool allocator, code running where an
allocation would synchronise the device or is not permitted, or a plug-in that
is handed buffers but no allocator. Its split-K scratch is a static device
array inside the library instead of context memory.

The tests call it through the C ABI twice in a row (the array keeps the last
call's contents, so the second call must not be disturbed by the first) and
compare each result with the context entry point msd_linear on the same inputs
and with the fp32 product x.float() @ w.float().T, within the GEMM tolerance
used by the other GPU tests. A shape whose best split would not fit the array
runs with fewer splits and still matches; a bounded wait that runs out is
reported by the next call. The file runs last in the suite and also passes on
its own in a fresh process.
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


def _close(y, ref, tol=1e-4):
    scale = max(1.0, ref.abs().max().item())
    err = (y - ref).abs().max().item()
    return err <= tol * scale, err


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
            ok, err = _close(y, y_ref)
            assert ok, (M, K, O, call, err)
            ok, err = _close(y, x.float() @ w.float().T)
            assert ok, (M, K, O, call, "vs fp32 product", err)
        y2 = y.clone()
        assert _noalloc(xs[-1], w, y2, accumulate=True) == msd.MSD_OK
        torch.cuda.synchronize()
        assert _close(y2, 2 * y_ref, 2e-4)[0]
    eng.close()


def test_noalloc_linear_splits_within_its_scratch():
    """A product whose best split-K would need more partials than the 16 MiB
    array runs with fewer splits instead of being refused, and matches the fp32
    product; bad strides are still refused."""
    build.build()
    g = torch.Generator(device="cuda").manual_seed(12)
    M, K, O = 256, 8192, 2048
    x = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(O, K, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    for _ in range(2):
        y = torch.full((M, O), float("nan"), device="cuda")
        assert _noalloc(x, w, y) == msd.MSD_OK
        torch.cuda.synchronize()
        ok, err = _close(y, x.float() @ w.float().T)
        assert ok, err
    assert _noalloc(x[:, :12], w[:, :12], y) == msd.MSD_ERR_INVALID   # k not a multiple of 8


def test_noalloc_linear_reports_a_bounded_wait_that_ran_out():
    """The status word in the static array: a bounded wait given a 1 ms limit on
    a barrier that nothing arrives at records a timeout there; the next call
    reports MSD_ERR_DEVICE (launching nothing) and clears it, and the call after
    that computes normally."""
    build.build()
    g = torch.Generator(device="cuda").manual_seed(13)
    x = torch.randn(16, 512, device="cuda", generator=g).to(torch.bfloat16)
    w = (torch.randn(256, 512, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    y = torch.zeros(16, 256, device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert msd.lib().msd_test_wait_timeout(None, 1_000_000, stream) == msd.MSD_OK
    assert _noalloc(x, w, y) == msd.MSD_ERR_DEVICE
    assert _noalloc(x, w, y) == msd.MSD_OK
    torch.cuda.synchronize()
    assert _close(y, x.float() @ w.float().T)[0]
