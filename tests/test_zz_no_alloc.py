"""fpo_cosine_noalloc: the cosine reduction for callers that cannot allocate
device memory (its scratch is a static device array inside libfpo instead of a
caller workspace).  Called through the C ABI and compared with fpo_cosine, the
workspace-based entry point, on two calls in a row.  This file sorts last so
that a run stopping at the first failure has already run every other test."""
import ctypes
import os

import numpy as np
import pytest
import torch

from paper_2608_14563_gb300 import synth

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def noalloc(fpo):
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so"))
    f = lib.fpo_cosine_noalloc
    f.argtypes = [ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                  ctypes.c_void_p, ctypes.c_void_p]
    f.restype = ctypes.c_int32
    return f


@pytest.mark.parametrize("dtype,code", [(torch.bfloat16, 1), (torch.float32, 0)])
@pytest.mark.parametrize("n", [7, 1000003, 50331648])
def test_noalloc_cosine_matches_workspace_entry_point(fpo, noalloc, dtype, code, n):
    X = synth.normal((n,), seed=5, tensor="noise", layer=1, device="cuda").to(dtype)
    Y = (X.float() + 1.3 * synth.normal((n,), seed=5, tensor="noise", layer=2,
                                        device="cuda")).to(dtype)
    ref = fpo.cosine(X, Y).cpu().numpy()
    stream = torch.cuda.current_stream().cuda_stream
    for _ in range(2):  # the shared static scratch keeps the previous call's partials
        out = torch.full((4,), float("nan"), dtype=torch.float64, device="cuda")
        rc = noalloc(n, code, X.data_ptr(), Y.data_ptr(), out.data_ptr(), stream)
        assert rc == 0, fpo.status_string(rc)
        got = out.cpu().numpy()
        for k in range(3):
            assert abs(got[k] - ref[k]) <= 1e-5 * abs(ref[k]) + 1e-9
        assert abs(got[3] - ref[3]) < 1e-6


def test_noalloc_cosine_empty_and_bad_arguments(fpo, noalloc):
    stream = torch.cuda.current_stream().cuda_stream
    out = torch.full((4,), float("nan"), dtype=torch.float64, device="cuda")
    assert noalloc(0, 1, None, None, out.data_ptr(), stream) == 0
    assert np.all(out.cpu().numpy() == 0.0)
    assert noalloc(-1, 1, None, None, out.data_ptr(), stream) == 2   # FPO_ERR_SHAPE
    assert noalloc(8, 7, None, None, out.data_ptr(), stream) == 3    # FPO_ERR_DTYPE
    assert noalloc(8, 1, None, None, out.data_ptr(), stream) == 1    # FPO_ERR_NULL
