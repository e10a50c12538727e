"""Failure detection without a GPU fault: a bounded wait inside a kernel runs out
on a barrier nothing arrives on, the kernel reports FPO_ERR_TIMEOUT through the
workspace status word and returns, and the context keeps working.

The tensor-core GEMMs' own abort path is driven the same way: with the wait limit
set to a microsecond (fpo_set_wait_limit_ns), the epilogue's wait for a tile whose
mainloop takes tens of microseconds runs out; every role of the kernel stops, the
copies and MMAs already issued are awaited with the teardown's own fixed limit, TMEM
is freed, and the status word reports the timeout.  With the default limit restored,
the same calls give the same bits as before."""
import ctypes
import os
import time

import pytest
import torch

import oracle
import synth
from helpers import cos, f64, rel_frob

DEFAULT_WAIT_LIMIT_NS = 2_000_000_000  # fpo_set_wait_limit_ns default (include/fpo.h)
SHORT_WAIT_LIMIT_NS = 1_000

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def tlib(fpo):
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so"))
    lib.fpo_testing_wait_timeout.argtypes = [ctypes.c_uint64, ctypes.c_void_p, ctypes.c_size_t,
                                             ctypes.c_void_p]
    lib.fpo_testing_wait_timeout.restype = ctypes.c_int32
    return lib


@pytest.fixture
def short_wait(fpo):
    """Sets the 1 us wait limit for the block and always restores the default after it."""
    class _Limit:
        def __enter__(self):
            fpo.set_wait_limit_ns(SHORT_WAIT_LIMIT_NS)

        def __exit__(self, *exc):
            fpo.set_wait_limit_ns(DEFAULT_WAIT_LIMIT_NS)
    try:
        yield _Limit()
    finally:
        fpo.set_wait_limit_ns(DEFAULT_WAIT_LIMIT_NS)


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


@pytest.fixture(scope="module")
def gemm_lib(fpo):
    lib = ctypes.CDLL(os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so"))
    vp = ctypes.c_void_p
    lib.fpo_testing_gemm_bf16.argtypes = [ctypes.c_int64] * 3 + [ctypes.c_int32] * 2 + [vp] * 4 + [
        ctypes.c_size_t, vp]
    lib.fpo_testing_gemm_bf16.restype = ctypes.c_int32
    lib.fpo_testing_set_gemm_variant.argtypes = [ctypes.c_int32]
    lib.fpo_testing_set_gemm_variant.restype = ctypes.c_int32
    return lib


@pytest.mark.parametrize("variant", [0, 1, 2], ids=["cta", "cta_pair", "cta_pair_wide"])
@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 1)])
def test_gemm_abort_path_reports_timeout_then_recovers(fpo, gemm_lib, short_wait, variant, a_mn,
                                                         b_mn):
    # 513 k-blocks per tile: a mainloop of a hundred microseconds or more, far longer than
    # the 1 us limit plus however long one try_wait may suspend its thread
    M, N, K = 1000, 2056, 32776
    gen = torch.Generator(device="cuda").manual_seed(17)
    A = torch.randn((K, M) if a_mn else (M, K), generator=gen, device="cuda").to(torch.bfloat16)
    B = torch.randn((K, N) if b_mn else (N, K), generator=gen, device="cuda").to(torch.bfloat16)
    stream = torch.cuda.current_stream().cuda_stream
    prev = gemm_lib.fpo_testing_set_gemm_variant(variant)
    try:
        def call():
            C = torch.full((M, N), float("nan"), device="cuda")
            ws = torch.zeros(256, dtype=torch.uint8, device="cuda")
            rc = gemm_lib.fpo_testing_gemm_bf16(M, N, K, a_mn, b_mn, A.data_ptr(), B.data_ptr(),
                                                C.data_ptr(), ws.data_ptr(), 256, stream)
            assert rc == 0, fpo.status_string(rc)
            return C, fpo.get_device_status(ws)

        C0, st0 = call()
        assert st0 == 0
        with short_wait:
            for _ in range(2):
                _, st = call()
                assert st == 9  # FPO_ERR_TIMEOUT
        C1, st1 = call()
        assert st1 == 0
        assert torch.equal(C0, C1)
    finally:
        gemm_lib.fpo_testing_set_gemm_variant(prev)
    a = A.double().T if a_mn else A.double()
    b = B.double() if b_mn else B.double().T
    # exact products of the bf16 values summed in fp64; the kernel's fp32 accumulation
    # over K = 32776 terms drifts by ~sqrt(K) 2^-24 ~ 1e-5 relative (a plain fp32 matmul
    # of the same values differed from it by 3.8e-5)
    assert rel_frob(f64(C1), f64(a @ b)) < 1e-4


def test_step_after_gemm_timeouts_matches_oracle(fpo, short_wait):
    """A whole bf16 step (error signal, grouped update; d = 8192) under the 1 us limit
    reports the timeout; the step after it, with the default limit, equals the step before bit for
    bit and matches the oracle."""
    wl = synth.Workload("abort-step", T=300, d=8192, d_ff=520, V=2056, layers=2,
                        targets="zipf", lr=1e-2, seed=3)
    inp = synth.make_all(wl, device="cuda")

    def step():
        g = torch.empty_like(inp["h"])
        ws = fpo.error_signal(inp["h"], inp["w"], inp["W_U"], inp["y"], g, eps=wl.eps,
                              min_rms=wl.min_rms)
        st_es = fpo.get_device_status(ws)
        Wm = [W.clone() for W in inp["W"]]
        Go = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device="cuda")
              for _ in range(wl.layers)]
        ws2 = fpo.layer_update_grouped(g, inp["A"], wl.lr, W_masters=Wm, G_outs=Go)
        st_up = fpo.get_device_status(ws2)
        return g, Wm, Go, st_es, st_up

    g0, W0, G0, s0, u0 = step()
    assert (s0, u0) == (0, 0)
    with short_wait:
        _, _, _, s1, u1 = step()
    assert s1 == 9  # the logits pass alone runs 128 k-blocks per tile
    assert u1 in (0, 9)
    g2, W2, G2, s2, u2 = step()
    assert (s2, u2) == (0, 0)
    assert torch.equal(g0, g2)
    for a, b in zip(W0 + G0, W2 + G2):
        assert torch.equal(a, b)
    ref = oracle.error_signal(synth.to_numpy_exact(inp["h"]), synth.to_numpy_exact(inp["w"]),
                              synth.to_numpy_exact(inp["W_U"]), inp["y"].cpu().numpy(),
                              eps=wl.eps, min_rms=wl.min_rms, s=wl.loss_scale)
    assert rel_frob(f64(g2), ref["g_tilde"]) < 2e-2 and cos(f64(g2), ref["g_tilde"]) >= 0.9995
    for l in range(wl.layers):
        G_ref = oracle.pseudograd(ref["g_tilde"], synth.to_numpy_exact(inp["A"][l]))
        assert rel_frob(f64(G2[l]), G_ref) < 2e-2, f"layer {l}"
