"""The direct error-matrix algorithm (FPO_ES_DIRECT, the bf16 default) against
the fp64 oracle, including the rows it hands to its fp32 fixup kernel.

The direct algorithm never forms E = s (softmax(z) - 1_y) (Sec. 3.1 step 2):
with the anchor c_t = z_{t, y_t} it stores p~ = exp(z - c_t) (target column 0)
and projects g_t = s e^{c_t - lse_t} (p~_t W_U - S'_t W_U[y_t]), S'_t = sum of
row t of p~.  Rows whose S'_t leaves [2^-80, 2^80] are recomputed, anchored at
lse_t, before the projection.

The fixup input is built so that every normalised hidden state is exact in bf16
(h = +-1, eps = 0: rho = 1 and yhat = norm_w (.) h), so the oracle's logits and
the GPU's differ only by fp32 accumulation, even at logit scales of ~100:
  * rows 0-49    anti-aligned with W_U[y=0]: cross-entropy ~160 nats (S' overflows)
  * rows 50-99   aligned with W_U[y=0]: 1 - p_target ~ e^-110 (S' underflows)
  * rows 100-149 partly aligned, y = 0: confident, 1 - p_target ~ e^-17 (inside)
  * rows 150-    random signs, random targets (inside)
"""
import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu

TOL = 2e-2
COS_MIN = 0.9995

RAGGED = Workload("ragged-bf16", T=300, d=520, d_ff=600, V=1000, layers=1, targets="zipf")


def run(fpo, h, w, W_U, y, *, eps, algo, t_chunk=0, loss_scale=None):
    h, w, W_U, y = h.cuda(), w.cuda(), W_U.cuda(), y.cuda()
    g = torch.empty_like(h)
    lse = torch.empty(h.shape[0], dtype=torch.float32, device="cuda")
    loss = torch.empty(1, dtype=torch.float32, device="cuda")
    ws = fpo.error_signal(h, w, W_U, y, g, eps=eps, min_rms=0.5, loss_scale=loss_scale,
                          t_chunk=t_chunk, lse_out=lse, loss_out=loss, algo=algo)
    assert fpo.get_device_status(ws) == fpo.OK
    fixed = fpo.direct_fixup_rows(h, W_U, ws, t_chunk=t_chunk, algo=algo)
    return {"g": g, "lse": lse, "loss": loss, "fixed": fixed}


def reference(h, w, W_U, y, *, eps, s):
    return oracle.error_signal(synth.to_numpy_exact(h), synth.to_numpy_exact(w),
                               synth.to_numpy_exact(W_U), y.numpy(), eps=eps, min_rms=0.5, s=s)


@pytest.fixture(scope="module")
def ragged():
    inp = synth.make_all(RAGGED)
    ref = reference(inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps,
                    s=RAGGED.loss_scale)
    return inp, ref


def test_direct_matches_oracle(fpo, ragged):
    inp, ref = ragged
    out = run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps, algo=fpo.ES_DIRECT)
    g = f64(out["g"])
    assert rel_frob(g, ref["g_tilde"]) < TOL and cos(g, ref["g_tilde"]) >= COS_MIN
    assert np.max(np.abs(f64(out["lse"]) - ref["lse"])) < 1e-2
    ce = oracle.mean_ce(ref["lse"], ref["zy"])
    assert abs(out["loss"].item() - ce) < 1e-3 * ce
    assert out["fixed"] == 0


def test_auto_is_direct_for_bf16(fpo, ragged):
    inp, _ = ragged
    a = run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps, algo=fpo.ES_AUTO)
    b = run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps, algo=fpo.ES_DIRECT)
    assert torch.equal(a["g"], b["g"]) and torch.equal(a["loss"], b["loss"])


def test_direct_is_bitwise_identical_across_token_chunks(fpo, ragged):
    """Whole tiles only at this size (the projection's split-K tail needs at least one
    wave of tiles; with it, split tiles depend on the chunk: see the split-K tail test)."""
    inp, _ = ragged
    runs = [run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps,
                algo=fpo.ES_DIRECT, t_chunk=c) for c in (0, 128, 37)]
    for r in runs[1:]:
        assert torch.equal(runs[0]["g"], r["g"])
        assert torch.equal(runs[0]["lse"], r["lse"])
        assert torch.equal(runs[0]["loss"], r["loss"])


def test_direct_is_bitwise_identical_across_gemm_kernels(fpo, ragged):
    inp, _ = ragged
    prev = fpo.set_gemm_variant(0)
    outs = []
    try:
        for v in (0, 1, 2):
            fpo.set_gemm_variant(v)
            outs.append(run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps,
                            algo=fpo.ES_DIRECT))
    finally:
        fpo.set_gemm_variant(prev)
    for o in outs[1:]:
        assert torch.equal(outs[0]["g"], o["g"]) and torch.equal(outs[0]["lse"], o["lse"])


def test_direct_agrees_with_stored_logits(fpo, ragged):
    inp, _ = ragged
    a = run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps, algo=fpo.ES_DIRECT)
    b = run(fpo, inp["h"], inp["w"], inp["W_U"], inp["y"], eps=RAGGED.eps,
            algo=fpo.ES_STORED_LOGITS)
    # the direct algorithm takes lse = c + log(1 + S') from its bf16-rounded
    # probabilities (S' off by at most 2^-9 relative), stored logits from fp32 sums
    assert torch.max(torch.abs(a["lse"] - b["lse"])).item() < 2.0 ** -9
    assert rel_frob(f64(a["g"]), f64(b["g"])) < 1e-2


def _window_input():
    """h = +-1 rows of four kinds (module docstring), W_U x 16 (exact in bf16)."""
    T, d, V = 300, 520, 1000
    wl = Workload("window", T=T, d=d, d_ff=8, V=V, layers=1, targets="uniform", eps=0.0)
    w = synth.make_norm_w(wl)
    W_U = synth.make_W_U(wl) * 16
    align = torch.sign(W_U[0].float() * w.float())
    align[align == 0] = 1.0
    rnd = torch.sign(synth.normal((T, d), seed=3, tensor="h"))
    rnd[rnd == 0] = 1.0
    h = rnd.clone()
    h[0:50] = -align
    h[50:100] = align
    part = torch.arange(d) < int(0.3 * d)
    h[100:150] = torch.where(part, align, rnd[100:150])
    y = synth.make_targets(wl)
    y[0:150] = 0
    return h.to(torch.bfloat16), w, W_U, y


def test_rows_outside_the_anchor_window_are_fixed(fpo):
    h, w, W_U, y = _window_input()
    T = h.shape[0]
    ref = reference(h, w, W_U, y, eps=0.0, s=1.0 / T)
    ce = ref["lse"] - ref["zy"]
    # the input is as intended: log2 S'_t from fp64 logits of the exact yhat = w (.) h
    z = (f64(h) * f64(w)[None, :]) @ f64(W_U).T
    zy = z[np.arange(T), y.numpy()]
    zo = z.copy()
    zo[np.arange(T), y.numpy()] = -np.inf
    mo = zo.max(axis=1)
    log2_S = (mo - zy + np.log(np.exp(zo - mo[:, None]).sum(axis=1))) / np.log(2.0)
    assert np.all(log2_S[0:50] > 100) and np.all(log2_S[50:100] < -100)
    assert np.all(np.abs(log2_S[100:]) < 70)
    outs = [run(fpo, h, w, W_U, y, eps=0.0, algo=fpo.ES_DIRECT, t_chunk=c) for c in (0, 64)]
    assert outs[0]["fixed"] == 100
    assert torch.equal(outs[0]["g"], outs[1]["g"]) and torch.equal(outs[0]["loss"], outs[1]["loss"])
    g = f64(outs[0]["g"])
    G = ref["g_tilde"]
    for lo, hi in ((0, 50), (100, 150), (150, T)):
        assert rel_frob(g[lo:hi], G[lo:hi]) < TOL, (lo, hi)
        assert cos(g[lo:hi], G[lo:hi]) >= COS_MIN, (lo, hi)
    # confident rows: the error signal itself is ~1e-8 of a typical row and still exact
    # to bf16 rounding (no 1 - p cancellation), row by row
    for t in range(100, 150):
        assert rel_frob(g[t], G[t]) < TOL, t
    # rows with 1 - p_target ~ e^-110: the signal is below fp32 range
    assert np.max(np.abs(g[50:100] - G[50:100])) < 1e-30
    assert np.max(np.abs(f64(outs[0]["lse"]) - ref["lse"]) / np.maximum(1, np.abs(ref["lse"]))) < 1e-5
    assert abs(outs[0]["loss"].item() - oracle.mean_ce(ref["lse"], ref["zy"])) < 1e-4 * np.mean(ce)


@pytest.mark.parametrize("variant", [0, 1, 2])
@pytest.mark.parametrize("algo", [1, 2, 3])  # recompute, stored logits, direct
def test_results_do_not_depend_on_workspace_contents(fpo, ragged, variant, algo):
    """Every workspace byte a call reads it writes first: a workspace full of 0xFF (NaN
    bit patterns) gives the same bits as a zeroed one, for every kernel variant."""
    inp, _ = ragged
    h, w, W_U, y = (inp[k].cuda() for k in ("h", "w", "W_U", "y"))
    prev = fpo.set_gemm_variant(variant)
    try:
        desc = fpo.error_signal_desc(*h.shape, W_U.shape[0], fpo.BF16, algo=algo, t_chunk=128)
        n = fpo.error_signal_workspace(desc)
        outs = []
        for fill in (0x00, 0xFF):
            ws = torch.full((n,), fill, dtype=torch.uint8, device="cuda")
            g = torch.empty_like(h)
            loss = torch.empty(1, dtype=torch.float32, device="cuda")
            fpo.error_signal(h, w, W_U, y, g, loss_out=loss, workspace=ws, algo=algo, t_chunk=128)
            assert fpo.get_device_status(ws) == fpo.OK
            outs.append((g, loss))
    finally:
        fpo.set_gemm_variant(prev)
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_many_rows_outside_the_window(fpo):
    """Logits ~30x the usual scale (exact +-1 hidden states, W_U x 64): most tokens have
    cross-entropy far beyond the window and go through the tensor-core fixup (several
    256-row tiles of gathered rows, a partial last one); the rows match the oracle and the
    count matches the fp64 window test of S'_t."""
    T, d, V = 1000, 512, 4096
    wl = Workload("many-fixed", T=T, d=d, d_ff=8, V=V, layers=1, targets="uniform", eps=0.0)
    w = synth.make_norm_w(wl)
    W_U = synth.make_W_U(wl) * 64
    h = torch.sign(synth.normal((T, d), seed=5, tensor="h"))
    h[h == 0] = 1.0
    h = h.to(torch.bfloat16)
    y = synth.make_targets(wl)
    z = (f64(h) * f64(w)[None, :]) @ f64(W_U).T
    zo = z.copy()
    zo[np.arange(T), y.numpy()] = -np.inf
    mo = zo.max(axis=1)
    log2_S = (mo - z[np.arange(T), y.numpy()] + np.log(np.exp(zo - mo[:, None]).sum(axis=1))) \
        / np.log(2.0)
    sure = int(np.sum(np.abs(log2_S) > 80.5))
    maybe = int(np.sum(np.abs(log2_S) > 79.5))
    assert sure > T // 2
    out = run(fpo, h, w, W_U, y, eps=0.0, algo=fpo.ES_DIRECT)
    assert sure <= out["fixed"] <= maybe
    ref = reference(h, w, W_U, y, eps=0.0, s=1.0 / T)
    g, G = f64(out["g"]), ref["g_tilde"]
    assert rel_frob(g, G) < TOL and cos(g, G) >= COS_MIN
    for t in range(0, T, 37):
        assert rel_frob(g[t], G[t]) < TOL, t
    assert np.max(np.abs(f64(out["lse"]) - ref["lse"]) / np.maximum(1, np.abs(ref["lse"]))) < 1e-5


@pytest.mark.parametrize("algo", [2, 3])  # stored logits, direct
def test_projection_split_k_tail(fpo, algo):
    """A projection of 20 x 8 tiles of 256 x 512 (T 5120, d 4096): 160 tiles are not a whole
    number of waves of the pair clusters, so the tiles of the last partial wave are split
    into k-block ranges and summed by the fixup kernel.  Checked against whole tiles (the
    256 x 256 kernel), against the oracle, across chunkings and for repeatability."""
    wl = Workload("sk", T=5120, d=4096, d_ff=8, V=2048, layers=1, targets="zipf")
    inp = synth.make_all(wl)
    h, w, W_U, y = inp["h"], inp["w"], inp["W_U"], inp["y"]
    prev = fpo.set_gemm_variant(2)
    try:
        a = run(fpo, h, w, W_U, y, eps=wl.eps, algo=algo)
        a2 = run(fpo, h, w, W_U, y, eps=wl.eps, algo=algo)
        ac = run(fpo, h, w, W_U, y, eps=wl.eps, algo=algo, t_chunk=1000)
        fpo.set_gemm_variant(1)
        b = run(fpo, h, w, W_U, y, eps=wl.eps, algo=algo)
    finally:
        fpo.set_gemm_variant(prev)
    assert torch.equal(a["g"], a2["g"])  # deterministic
    ga, gb, gc = f64(a["g"]), f64(b["g"]), f64(ac["g"])
    # g~ is bf16: summing a cut tile's two fp32 parts reassociates the K sum, which flips
    # the bf16 rounding of a few elements (a wrong part would be off by O(1) on a tile)
    for x, y_ in ((ga, gb), (gc, ga)):
        assert rel_frob(x, y_) < 2e-4
        row_err = np.linalg.norm(x - y_, axis=1) / np.linalg.norm(y_, axis=1)
        assert np.max(row_err) < 5e-3
    ref = reference(h, w, W_U, y, eps=wl.eps, s=wl.loss_scale)
    assert rel_frob(ga, ref["g_tilde"]) < TOL and cos(ga, ref["g_tilde"]) >= COS_MIN


@pytest.mark.parametrize("shape", [(700, 320, 840, 3), (1024, 512, 768, 2), (300, 1024, 264, 4)])
def test_update_is_bitwise_identical_across_gemm_kernels(fpo, shape):
    """The grouped update (G_l, the fp32 master step, the bf16 weights) computes the same
    sums in the same order per element under every GEMM kernel variant: single CTA and CTA
    pair (ragged T and d)."""
    T, d, d_ff, L = shape
    gen = torch.Generator(device="cuda").manual_seed(T + d)
    g = (torch.randn(T, d, device="cuda", generator=gen) * 1e-2).to(torch.bfloat16)
    A = [torch.randn(T, d_ff, device="cuda", generator=gen).to(torch.bfloat16) for _ in range(L)]
    W0 = [0.02 * torch.randn(d, d_ff, device="cuda", generator=gen) for _ in range(L)]
    prev = fpo.set_gemm_variant(0)
    outs = []
    try:
        for v in (0, 1, 2):
            fpo.set_gemm_variant(v)
            Wm = [w.clone() for w in W0]
            Wo = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(L)]
            Go = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(L)]
            ws = fpo.layer_update_grouped(g, A, 1e-3, W_masters=Wm, W_outs=Wo, G_outs=Go)
            assert fpo.get_device_status(ws) == fpo.OK
            outs.append(Wm + Wo + Go)
    finally:
        fpo.set_gemm_variant(prev)
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            assert torch.equal(a, b)
