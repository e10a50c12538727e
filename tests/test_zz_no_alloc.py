"""fpo_cosine_noalloc: the cosine reduction for callers that cannot allocate
device memory (its scratch is a static device array inside libfpo instead of a
caller workspace).  Called through the C ABI and compared with fpo_cosine, the
workspace-based entry point: the header promises the same bits (same kernels,
block count and summation order), on two calls in a row, and after a larger call
that left more partial sums in the shared array than the next call uses.  This
file sorts last so that a run stopping at the first failure has already run every
other test."""
import ctypes
import os

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FPO_ERR_NULL, FPO_ERR_SHAPE, FPO_ERR_DTYPE, FPO_ERR_ALIGN = 1, 2, 3, 4


@pytest.fixture(scope="module")
def noalloc(fpo):
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so"))
    f = lib.fpo_cosine_noalloc
    f.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                  ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int32
    return f


def _pair(n, dtype, seed=5):
    X = synth.normal((n,), seed=seed, tensor="noise", layer=1, device="cuda").to(dtype)
    Y = (X.float() + 1.3 * synth.normal((n,), seed=seed, tensor="noise", layer=2,
                                        device="cuda")).to(dtype)
    return X, Y


def _call(fpo, noalloc, X, Y, code):
    out = torch.full((4,), float("nan"), dtype=torch.float64, device="cuda")
    rc = noalloc(X.numel(), code, X.data_ptr(), Y.data_ptr(), out.data_ptr(),
                 torch.cuda.current_stream().cuda_stream)
    assert rc == 0, fpo.status_string(rc)
    return out


@pytest.mark.parametrize("dtype,code", [(torch.bfloat16, 1), (torch.float32, 0)])
@pytest.mark.parametrize("n", [7, 1000003, 50331648])
def test_noalloc_cosine_matches_workspace_entry_point(fpo, noalloc, dtype, code, n):
    X, Y = _pair(n, dtype)
    ref = fpo.cosine(X, Y)
    for _ in range(2):  # the shared static scratch keeps the previous call's partials
        got = _call(fpo, noalloc, X, Y, code)
        assert torch.equal(got, ref), (got.cpu().numpy(), ref.cpu().numpy())


@pytest.mark.parametrize("dtype,code", [(torch.bfloat16, 1), (torch.float32, 0)])
def test_noalloc_cosine_after_a_larger_call(fpo, noalloc, dtype, code):
    """A large call fills every partial-sum slot a launch can use; a following small call
    launches fewer blocks and must read only the slots it wrote itself."""
    Xb, Yb = _pair(50331648, dtype, seed=9)
    Xs, Ys = _pair(4099, dtype, seed=10)
    ref_b, ref_s = fpo.cosine(Xb, Yb), fpo.cosine(Xs, Ys)
    for _ in range(2):
        assert torch.equal(_call(fpo, noalloc, Xb, Yb, code), ref_b)
        assert torch.equal(_call(fpo, noalloc, Xs, Ys, code), ref_s)


def test_noalloc_cosine_empty_and_bad_arguments(fpo, noalloc):
    stream = torch.cuda.current_stream().cuda_stream
    out = torch.full((4,), float("nan"), dtype=torch.float64, device="cuda")
    assert noalloc(0, 1, None, None, out.data_ptr(), stream) == 0
    assert np.all(out.cpu().numpy() == 0.0)
    assert noalloc(-1, 1, None, None, out.data_ptr(), stream) == FPO_ERR_SHAPE
    assert noalloc(8, 7, None, None, out.data_ptr(), stream) == FPO_ERR_DTYPE
    assert noalloc(8, 1, None, None, out.data_ptr(), stream) == FPO_ERR_NULL
    X = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    # inputs off their 16-byte boundary, and an output off its 8-byte boundary: rejected
    # before anything is enqueued
    assert noalloc(8, 1, X.data_ptr() + 2, X.data_ptr(), out.data_ptr(), stream) == FPO_ERR_ALIGN
    assert noalloc(8, 1, X.data_ptr(), X.data_ptr() + 8, out.data_ptr(), stream) == FPO_ERR_ALIGN
    assert noalloc(8, 1, X.data_ptr(), X.data_ptr(), out.data_ptr() + 4, stream) == FPO_ERR_ALIGN
    assert np.all(out.cpu().numpy() == 0.0)  # untouched by the rejected calls
