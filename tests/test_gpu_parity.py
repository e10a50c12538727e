"""GPU path (through the C ABI) against the fp64 oracle on identical seeded inputs.

Tolerances (Sec. 3.1 / App. A quantities):
* bf16 path: relative Frobenius error <= 2e-2 on g~, G_l and the updated
  weights (and on the step dW = W' - W), cos(G_gpu, G_oracle) >= 0.9995.
* fp32 path: relative Frobenius error <= 1e-5 on the same quantities.
"""

import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu

BF16_TOL = 2e-2
BF16_COS = 0.9995
F32_TOL = 1e-5


def gpu_step(fpo, wl, inp, *, t_chunk=0, lr=None, grouped=True, algo=0):
    """One FPO step on the GPU: error signal, then the update of every layer."""
    lr = wl.lr if lr is None else lr
    h, w, W_U, y = (inp[k].cuda() for k in ("h", "w", "W_U", "y"))
    T, d = h.shape
    g = torch.empty_like(h)
    lse = torch.empty(T, dtype=torch.float32, device="cuda")
    loss = torch.empty(1, dtype=torch.float32, device="cuda")
    ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms,
                          loss_scale=wl.loss_scale, t_chunk=t_chunk, lse_out=lse, loss_out=loss,
                          algo=algo)
    assert fpo.get_device_status(ws) == fpo.OK
    A = [a.cuda() for a in inp["A"]]
    Wm = [W.cuda().clone() for W in inp["W"]]
    Wo = [torch.empty(W.shape, dtype=h.dtype, device="cuda") for W in inp["W"]]
    Go = [torch.empty(W.shape, dtype=h.dtype, device="cuda") for W in inp["W"]]
    if grouped:
        ws2 = fpo.layer_update_grouped(g, A, lr, W_masters=Wm, W_outs=Wo, G_outs=Go)
        assert fpo.get_device_status(ws2) == fpo.OK
    else:
        for l in range(len(A)):
            ws2 = fpo.layer_update(g, A[l], lr, W_master=Wm[l], W_out=Wo[l], G_out=Go[l])
            assert fpo.get_device_status(ws2) == fpo.OK
    torch.cuda.synchronize()
    return {"g": g, "lse": lse, "loss": loss, "W": Wm, "W_out": Wo, "G": Go}


def oracle_step(wl, inp, lr=None):
    lr = wl.lr if lr is None else lr
    h, w, W_U = (synth.to_numpy_exact(inp[k]) for k in ("h", "w", "W_U"))
    y = inp["y"].numpy()
    es = oracle.error_signal(h, w, W_U, y, eps=wl.eps, min_rms=wl.min_rms, s=wl.loss_scale)
    G = [oracle.pseudograd(es["g_tilde"], synth.to_numpy_exact(a)) for a in inp["A"]]
    upd = [oracle.sgd_update(W.numpy(), Gl, lr) for W, Gl in zip(inp["W"], G)]
    return {"g": es["g_tilde"], "lse": es["lse"], "loss": oracle.mean_ce(es["lse"], es["zy"]),
            "G": G, "W": [u[0] for u in upd], "W_bf16": [u[1] for u in upd]}


def check(gpu, ref, inp, lr, tol, cos_min=None):
    assert rel_frob(f64(gpu["g"]), ref["g"]) < tol
    assert abs(float(gpu["loss"].item()) - ref["loss"]) < max(tol, 1e-6) * abs(ref["loss"]) + 1e-6
    assert np.max(np.abs(f64(gpu["lse"]) - ref["lse"])) < max(tol, 1e-6) * 10
    for l in range(len(ref["G"])):
        G = f64(gpu["G"][l])
        assert rel_frob(G, ref["G"][l]) < tol, f"layer {l}"
        if cos_min is not None:
            assert cos(G, ref["G"][l]) >= cos_min
        W0 = inp["W"][l].numpy().astype(np.float64)
        assert rel_frob(f64(gpu["W"][l]), ref["W"][l]) < tol
        if lr != 0:
            # dW read back from fp32 W' is resolved only to fp32 ulps of W' (both sides round
            # W' to fp32), so the bound adds that storage resolution to the tolerance.
            d_ref = ref["W"][l].astype(np.float64) - W0
            ulp = np.spacing(np.abs(ref["W"][l]).astype(np.float32)).astype(np.float64)
            q = np.linalg.norm(ulp) / max(np.linalg.norm(d_ref), 1e-300)
            assert rel_frob(f64(gpu["W"][l]) - W0, d_ref) < tol + q
        assert rel_frob(f64(gpu["W_out"][l]), oracle.bf16_bits_to_f64(ref["W_bf16"][l])
                        if gpu["W_out"][l].dtype == torch.bfloat16 else ref["W"][l]) < tol


def test_tiny_fp32_workload_matches_oracle(fpo):
    wl = synth.WORKLOADS["tiny"]
    inp = synth.make_all(wl)
    gpu = gpu_step(fpo, wl, inp)
    ref = oracle_step(wl, inp)
    check(gpu, ref, inp, wl.lr, F32_TOL)


RAGGED = Workload("ragged-bf16", T=300, d=520, d_ff=600, V=1000, layers=2, targets="zipf", lr=1e-2)


@pytest.fixture(scope="module")
def ragged():
    inp = synth.make_all(RAGGED)
    return inp, oracle_step(RAGGED, inp)


def test_bf16_ragged_matches_oracle(fpo, ragged):
    inp, ref = ragged
    gpu = gpu_step(fpo, RAGGED, inp)
    check(gpu, ref, inp, RAGGED.lr, BF16_TOL, BF16_COS)


@pytest.mark.parametrize("algo", [1, 2])  # FPO_ES_RECOMPUTE, FPO_ES_STORED_LOGITS
def test_bf16_both_algorithms_match_oracle(fpo, ragged, algo):
    inp, ref = ragged
    gpu = gpu_step(fpo, RAGGED, inp, algo=algo)
    check(gpu, ref, inp, RAGGED.lr, BF16_TOL, BF16_COS)


@pytest.mark.parametrize("wl_name", ["tiny", "ragged"])
def test_algorithms_and_chunkings_are_bitwise_identical(fpo, ragged, wl_name):
    wl, inp = (RAGGED, ragged[0]) if wl_name == "ragged" else (
        synth.WORKLOADS["tiny"], synth.make_all(synth.WORKLOADS["tiny"]))
    runs = [gpu_step(fpo, wl, inp, algo=a, t_chunk=c)
            for a in (1, 2) for c in (0, 128, 37)]
    for r in runs[1:]:
        assert torch.equal(runs[0]["g"], r["g"])
        assert torch.equal(runs[0]["lse"], r["lse"])
        assert torch.equal(runs[0]["loss"], r["loss"])


def test_grouped_update_equals_per_layer_calls(fpo, ragged):
    inp, _ = ragged
    a = gpu_step(fpo, RAGGED, inp, grouped=True)
    b = gpu_step(fpo, RAGGED, inp, grouped=False)
    for l in range(RAGGED.layers):
        assert torch.equal(a["G"][l], b["G"][l])
        assert torch.equal(a["W"][l], b["W"][l])
        assert torch.equal(a["W_out"][l], b["W_out"][l])


def test_repeat_runs_are_bitwise_identical(fpo, ragged):
    inp, _ = ragged
    a = gpu_step(fpo, RAGGED, inp)
    b = gpu_step(fpo, RAGGED, inp)
    assert torch.equal(a["g"], b["g"]) and torch.equal(a["loss"], b["loss"])
    for l in range(RAGGED.layers):
        assert torch.equal(a["W"][l], b["W"][l])


def test_lr_zero_leaves_master_bit_identical_and_step_is_linear(fpo, ragged):
    inp, _ = ragged
    z = gpu_step(fpo, RAGGED, inp, lr=0.0)
    for l in range(RAGGED.layers):
        assert torch.equal(z["W"][l].cpu(), inp["W"][l])
        assert torch.equal(z["W_out"][l].cpu(), inp["W"][l].to(torch.bfloat16))
    a = gpu_step(fpo, RAGGED, inp, lr=1e-2)
    b = gpu_step(fpo, RAGGED, inp, lr=2e-2)
    for l in range(RAGGED.layers):
        W0 = inp["W"][l].double().numpy()
        da, db = f64(a["W"][l]) - W0, f64(b["W"][l]) - W0
        assert rel_frob(db, 2 * da) < 1e-3


@pytest.mark.parametrize("shape", [(1, 8, 8, 8), (5, 16, 24, 40), (129, 64, 264, 136)])
def test_bf16_small_and_degenerate_shapes(fpo, shape):
    T, d, V, d_ff = shape
    wl = Workload("edge", T=T, d=d, d_ff=d_ff, V=V, layers=1, targets="uniform", lr=1e-2)
    inp = synth.make_all(wl)
    gpu = gpu_step(fpo, wl, inp)
    ref = oracle_step(wl, inp)
    check(gpu, ref, inp, wl.lr, BF16_TOL)


@pytest.mark.parametrize("shape", [(5, 7, 13, 9), (70, 33, 129, 65), (1, 1, 1, 1)])
def test_fp32_odd_shapes(fpo, shape):
    T, d, V, d_ff = shape
    wl = Workload("edge32", T=T, d=d, d_ff=d_ff, V=V, layers=2, dtype="f32", targets="uniform",
                  lr=1e-2)
    inp = synth.make_all(wl)
    gpu = gpu_step(fpo, wl, inp)
    ref = oracle_step(wl, inp)
    check(gpu, ref, inp, wl.lr, F32_TOL)


def test_min_rms_clamp_on_device(fpo):
    wl = Workload("clamp", T=64, d=128, d_ff=64, V=256, layers=1, dtype="f32", lr=1e-2)
    inp = synth.make_all(wl)
    inp["h"][::3] *= 0.2  # rho ~ 0.2 on every third token: the clamp is active there
    gpu = gpu_step(fpo, wl, inp)
    ref = oracle_step(wl, inp)
    check(gpu, ref, inp, wl.lr, F32_TOL)


def test_min_rms_clamp_in_the_fused_projection_epilogue(fpo):
    """bf16, direct algorithm: the final-norm VJP runs in the projection's epilogue (and in
    its split-tail fixup); tokens with rho ~ 0.2 < min_rms take the clamped prefactor
    while x^ keeps the true rho, as the oracle defines it.  T = 4096, d = 4096: one chunk
    has 128 projection tiles of 256 x 512, 1.7 waves of pair clusters, so its last wave is
    split and the tail goes through the fixup kernel; chunks of 256 tokens have whole
    tiles only."""
    wl = Workload("clamp-bf16", T=4096, d=4096, d_ff=136, V=1032, layers=1, lr=1e-2)
    inp = synth.make_all(wl)
    inp["h"] = inp["h"].float()
    inp["h"][::3] *= 0.2
    inp["h"] = inp["h"].to(torch.bfloat16)
    ref = oracle_step(wl, inp)
    for t_chunk in (0, 256):
        gpu = gpu_step(fpo, wl, inp, t_chunk=t_chunk)
        check(gpu, ref, inp, wl.lr, BF16_TOL, BF16_COS)
        g, G = f64(gpu["g"]), ref["g"]
        rows = np.arange(0, wl.T, 3)  # every clamped token on its own
        for t in rows:
            assert rel_frob(g[t], G[t]) < BF16_TOL and cos(g[t], G[t]) >= BF16_COS, t


def test_eps0_orthogonality_through_the_fused_vjp(fpo):
    """bf16, direct algorithm, eps = 0: <g~_t, h_t> = 0 for every token up to the bf16
    rounding of g~ (a relative size of ~2^-9 / sqrt(d)), with the VJP's row term taken
    through the logits in the projection's epilogue."""
    wl = Workload("eps0-bf16", T=300, d=1024, d_ff=64, V=4104, layers=1, eps=0.0)
    inp = synth.make_all(wl)
    gpu = gpu_step(fpo, wl, inp)
    g, h = f64(gpu["g"]), f64(inp["h"])
    rel = np.abs(np.sum(g * h, axis=1)) / (np.linalg.norm(g, axis=1) * np.linalg.norm(h, axis=1))
    assert np.max(rel) < 1e-3
    ref = oracle_step(wl, inp)
    assert rel_frob(g, ref["g"]) < BF16_TOL


def test_eps0_vjp_orthogonal_to_h_on_device(fpo):
    wl = Workload("eps0", T=96, d=256, d_ff=64, V=512, layers=1, dtype="f32", eps=0.0)
    inp = synth.make_all(wl)
    gpu = gpu_step(fpo, wl, inp)
    g, h = f64(gpu["g"]), inp["h"].double().numpy()
    rel = np.abs(np.sum(g * h, axis=1)) / (np.linalg.norm(g, axis=1) * np.linalg.norm(h, axis=1))
    assert np.max(rel) < 1e-5


def test_empty_token_batch(fpo):
    wl = Workload("empty", T=0, d=64, d_ff=128, V=256, layers=1)
    inp = synth.make_all(wl)
    gpu = gpu_step(fpo, wl, inp)
    assert gpu["loss"].item() == 0.0
    assert torch.equal(gpu["W"][0].cpu(), inp["W"][0])
    assert torch.equal(gpu["W_out"][0].cpu(), inp["W"][0].to(torch.bfloat16))
    assert torch.count_nonzero(gpu["G"][0]).item() == 0


def test_out_of_range_target_sets_device_status(fpo):
    wl = Workload("badtarget", T=64, d=64, d_ff=64, V=256, layers=1)
    inp = synth.make_all(wl)
    h, w, W_U, y = (inp[k].cuda() for k in ("h", "w", "W_U", "y"))
    y[5] = wl.V
    g = torch.empty_like(h)
    ws = fpo.error_signal(h, w, W_U, y, g)
    assert fpo.get_device_status(ws) == 8  # FPO_ERR_TARGET_RANGE
    y[5] = -3
    fpo.error_signal(h, w, W_U, y, g, workspace=ws)
    assert fpo.get_device_status(ws) == 8
    y[5] = 0
    fpo.error_signal(h, w, W_U, y, g, workspace=ws)
    assert fpo.get_device_status(ws) == fpo.OK  # the context stays usable


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("n", [0, 5, 1000003])
def test_cosine_matches_oracle(fpo, dtype, n):
    X = synth.normal((n,), seed=1, tensor="noise", layer=1).to(dtype)
    Y = (X.float() + 0.7 * synth.normal((n,), seed=1, tensor="noise", layer=2)).to(dtype)
    out = fpo.cosine(X.cuda(), Y.cuda())
    out2 = fpo.cosine(X.cuda(), Y.cuda())
    assert torch.equal(out, out2)  # fixed reduction order
    got = out.cpu().numpy()
    if n == 0:
        assert np.all(got == 0)
        return
    ref = oracle.cosine(synth.to_numpy_exact(X), synth.to_numpy_exact(Y))
    for k in range(3):
        assert abs(got[k] - ref[k]) <= 1e-5 * abs(ref[k]) + 1e-9
    assert abs(got[3] - ref[3]) < 1e-6


def test_layer_update_standalone_matches_oracle(fpo):
    # synthetic g~ (not produced by the GPU) and several layers, more tiles than SMs
    T, d, d_ff, L = 1000, 384, 1048, 3
    g = synth.normal((T, d), std=1e-3, seed=3, tensor="h").to(torch.bfloat16)
    wl = Workload("upd", T=T, d=d, d_ff=d_ff, V=8, layers=L, lr=0.5)
    A = [synth.make_A(wl, l) for l in range(L)]
    W = [synth.make_W_master(wl, l) for l in range(L)]
    Wm = [x.cuda() for x in W]
    Wo = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    Go = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    ws = fpo.layer_update_grouped(g.cuda(), [a.cuda() for a in A], wl.lr, W_masters=Wm, W_outs=Wo,
                                  G_outs=Go)
    assert fpo.get_device_status(ws) == fpo.OK
    gn = synth.to_numpy_exact(g)
    for l in range(L):
        Gr = oracle.pseudograd(gn, synth.to_numpy_exact(A[l]))
        Wn, _ = oracle.sgd_update(W[l].numpy(), Gr, wl.lr)
        assert rel_frob(f64(Go[l]), Gr) < BF16_TOL and cos(f64(Go[l]), Gr) >= BF16_COS
        W0 = W[l].double().numpy()
        assert rel_frob(f64(Wm[l]) - W0, Wn.astype(np.float64) - W0) < BF16_TOL
