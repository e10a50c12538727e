"""The tcgen05 GEMM core alone, through fpo_testing_gemm_bf16, against an fp64
host matmul of the same bf16 values, for the three operand layouts the FPO
step uses (K-major x K-major, K-major x MN-major, MN-major x MN-major) on
shapes that span several tiles and end in ragged tails in M, N and K."""
import ctypes
import os

import numpy as np
import pytest
import torch

from helpers import f64, rel_frob

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", params=[0, 1, 2], ids=["cta", "cta_pair", "cta_pair_wide"])
def tlib(fpo, request):
    """The test entry points, with the GEMM kernel variant selected (single CTA, CTA pair, CTA
    pair with 256 x 512 tiles)."""
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so"))
    vp = ctypes.c_void_p
    lib.fpo_testing_gemm_bf16.argtypes = [ctypes.c_int64] * 3 + [ctypes.c_int32] * 2 + [vp] * 4 + [
        ctypes.c_size_t, vp]
    lib.fpo_testing_gemm_bf16.restype = ctypes.c_int32
    lib.fpo_testing_set_gemm_variant.argtypes = [ctypes.c_int32]
    lib.fpo_testing_set_gemm_variant.restype = ctypes.c_int32
    prev = lib.fpo_testing_set_gemm_variant(request.param)
    yield lib
    lib.fpo_testing_set_gemm_variant(prev)


def gemm(tlib, fpo, M, N, K, a_mn, b_mn, seed=0):
    g = torch.Generator(device="cpu").manual_seed(seed)
    A = torch.randn((K, M) if a_mn else (M, K), generator=g).to(torch.bfloat16)
    B = torch.randn((K, N) if b_mn else (N, K), generator=g).to(torch.bfloat16)
    Ad, Bd = A.cuda(), B.cuda()
    C = torch.full((M, N), float("nan"), device="cuda")
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    rc = tlib.fpo_testing_gemm_bf16(M, N, K, a_mn, b_mn, Ad.data_ptr(), Bd.data_ptr(), C.data_ptr(),
                                    ws.data_ptr(), 256, torch.cuda.current_stream().cuda_stream)
    assert rc == 0, fpo.status_string(rc)
    assert fpo.get_device_status(ws) == 0
    a = f64(A).T if a_mn else f64(A)
    b = f64(B) if b_mn else f64(B).T
    return f64(C), a @ b


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 1)])
def test_single_tile(tlib, fpo, a_mn, b_mn):
    got, ref = gemm(tlib, fpo, 128, 256, 64, a_mn, b_mn)
    assert np.all(np.isfinite(got))
    assert rel_frob(got, ref) < 1e-5


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 1)])
def test_many_tiles_ragged(tlib, fpo, a_mn, b_mn):
    got, ref = gemm(tlib, fpo, 296, 600, 520, a_mn, b_mn, seed=1)
    assert np.all(np.isfinite(got))
    assert rel_frob(got, ref) < 1e-5
    assert np.max(np.abs(got - ref)) < 1e-3


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 1)])
def test_persistent_many_tiles_long_k(tlib, fpo, a_mn, b_mn):
    # more tiles than SMs (persistent loop, both TMEM buffers) and a long K ring
    got, ref = gemm(tlib, fpo, 1536, 2816, 1040, a_mn, b_mn, seed=2)
    assert rel_frob(got, ref) < 1e-5


@pytest.mark.parametrize("M", [256, 384, 136])
def test_pair_row_halves(tlib, fpo, M):
    # a tile pair whose second half is partly or wholly outside M
    got, ref = gemm(tlib, fpo, M, 512, 192, 0, 0, seed=4)
    assert rel_frob(got, ref) < 1e-5


def test_tiny_all_overhang(tlib, fpo):
    got, ref = gemm(tlib, fpo, 8, 8, 8, 0, 0, seed=3)
    assert rel_frob(got, ref) < 1e-5
    got, ref = gemm(tlib, fpo, 8, 8, 8, 1, 1, seed=3)
    assert rel_frob(got, ref) < 1e-5
