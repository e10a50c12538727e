"""Failure detection without a GPU fault: a bounded wait inside a kernel runs out
on a barrier nothing arrives on, the kernel reports FPO_ERR_TIMEOUT through the
workspace status word and returns, and the context keeps working."""
import ctypes
import os
import time

import pytest
import torch

from paper_2608_14563_gb300 import synth

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def tlib(fpo):
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so"))
    lib.fpo_testing_wait_timeout.argtypes = [ctypes.c_uint64, ctypes.c_void_p, ctypes.c_size_t,
                                             ctypes.c_void_p]
    lib.fpo_testing_wait_timeout.restype = ctypes.c_int32
    return lib


def test_bounded_wait_times_out_and_reports(fpo, tlib):
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    t0 = time.perf_counter()
    assert tlib.fpo_testing_wait_timeout(20_000_000, ws.data_ptr(), 256, stream) == 0  # 20 ms
    assert fpo.get_device_status(ws) == 9  # FPO_ERR_TIMEOUT
    elapsed = time.perf_counter() - t0
    assert 0.015 < elapsed < 5.0
    assert fpo.get_device_status(ws) == 0  # read-and-clear
    assert tlib.fpo_testing_wait_timeout(0, ws.data_ptr(), 256, stream) == 10  # FPO_ERR_ARG


def test_context_usable_after_timeout(fpo, tlib):
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
    tlib.fpo_testing_wait_timeout(5_000_000, ws.data_ptr(), 256,
                                  torch.cuda.current_stream().cuda_stream)
    assert fpo.get_device_status(ws) == 9
    X = synth.normal((4099,), seed=2, tensor="noise", device="cuda").to(torch.bfloat16)
    out = fpo.cosine(X, X).cpu()
    assert abs(out[3].item() - 1.0) < 1e-6
    wl = synth.Workload("after-timeout", T=64, d=64, d_ff=64, V=256, layers=1)
    inp = synth.make_all(wl, device="cuda")
    g = torch.empty_like(inp["h"])
    ws2 = fpo.error_signal(inp["h"], inp["w"], inp["W_U"], inp["y"], g)
    assert fpo.get_device_status(ws2) == 0
    assert torch.isfinite(g.float()).all()
