"""Layer-specific signals (Sec. 3.1 step 4, Sec. 3.2, App. E): the post-feedforward and / or
pre-MLP RMSNorm Jacobians composed per target layer in one launch (fpo_layer_signals),
against the oracle's composition, and the step of a pre-MLP family (Qwen3-like) through
fpo_layer_update_grouped_signals."""
import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu

MODES = {"post": (True, False), "pre": (False, True), "both": (True, True)}


def _case(wl, layers):
    g = synth.normal((wl.T, wl.d), std=1e-3, seed=7, tensor="h", layer=5).to(wl.torch_dtype)
    m = [synth.make_mlp_out(wl, l) for l in range(layers)]
    gp = [synth.make_post_norm_w(wl, l) for l in range(layers)]
    x = [synth.make_pre_norm_in(wl, l) for l in range(layers)]
    gq = [synth.make_pre_norm_w(wl, l) for l in range(layers)]
    return g, m, gp, x, gq


def _run(fpo, g, m, gp, x, gq, post, pre, *, eps=1e-6, min_rms=0.5):
    outs = [torch.empty(g.shape, dtype=g.dtype, device="cuda") for _ in m]
    cu = lambda ts: [t.cuda() for t in ts]
    fpo.layer_signals(g.cuda(), outs, m=cu(m) if post else None, gamma_post=cu(gp) if post else None,
                      x=cu(x) if pre else None, gamma_pre=cu(gq) if pre else None, eps=eps,
                      min_rms=min_rms)
    torch.cuda.synchronize()
    return outs


def _ref(g, m, gp, x, gq, post, pre, l, *, eps=1e-6, min_rms=0.5):
    e = synth.to_numpy_exact
    return oracle.layer_signal(e(g), e(m[l]) if post else None, e(gp[l]) if post else None,
                               e(x[l]) if pre else None, e(gq[l]) if pre else None, eps=eps,
                               min_rms=min_rms)


# bf16 rows: d <= 2048 / 4096 / 8192 take the block-per-row kernel with 8 / 16 / 32
# elements per thread, longer rows and fp32 the warp-per-row kernel (three passes).
@pytest.mark.parametrize("mode", list(MODES))
@pytest.mark.parametrize("dtype,T,d,tol", [("bf16", 300, 520, 2e-2), ("bf16", 37, 4096, 2e-2),
                                            ("bf16", 5, 8192, 2e-2), ("bf16", 9, 12288, 2e-2),
                                            ("f32", 77, 33, 1e-5), ("f32", 50, 256, 1e-5)])
def test_layer_signals_match_oracle(fpo, mode, dtype, T, d, tol):
    post, pre = MODES[mode]
    wl = Workload("sig", T=T, d=d, d_ff=8, V=8, layers=3, dtype=dtype)
    g, m, gp, x, gq = _case(wl, 3)
    outs = _run(fpo, g, m, gp, x, gq, post, pre)
    for l in range(3):
        ref = _ref(g, m, gp, x, gq, post, pre, l)
        got = f64(outs[l])
        assert rel_frob(got, ref) < tol
        for t in range(T):  # every row: clamped rows (every 64th m row, x row 32 mod 64) too
            assert rel_frob(got[t], ref[t]) < 2 * tol


@pytest.mark.parametrize("dtype,d", [("bf16", 520), ("bf16", 12288), ("f32", 33), ("f32", 256)])
def test_single_norm_is_bitwise_fpo_rmsnorm_vjp(fpo, dtype, d):
    """One norm: the same arithmetic, in the same order, as fpo_rmsnorm_vjp at that norm."""
    wl = Workload("one", T=70, d=d, d_ff=8, V=8, layers=2, dtype=dtype)
    g, m, gp, x, gq = _case(wl, 2)
    for post, pre, inp, w in ((True, False, m, gp), (False, True, x, gq)):
        outs = _run(fpo, g, m, gp, x, gq, post, pre)
        for l in range(2):
            one = torch.empty_like(outs[l])
            fpo.rmsnorm_vjp(g.cuda(), inp[l].cuda(), w[l].cuda(), one, eps=1e-6, min_rms=0.5)
            assert torch.equal(one, outs[l])


@pytest.mark.parametrize("d", [33, 256])
def test_fp32_composition_is_bitwise_two_calls(fpo, d):
    """fp32: the fused composition keeps u in fp32 exactly as one fpo_rmsnorm_vjp call
    stores it, so post-FFN then pre-MLP equals the two calls in sequence, bit for bit."""
    wl = Workload("two", T=50, d=d, d_ff=8, V=8, layers=2, dtype="f32")
    g, m, gp, x, gq = _case(wl, 2)
    outs = _run(fpo, g, m, gp, x, gq, True, True)
    for l in range(2):
        u = torch.empty_like(outs[l])
        two = torch.empty_like(outs[l])
        fpo.rmsnorm_vjp(g.cuda(), m[l].cuda(), gp[l].cuda(), u, eps=1e-6, min_rms=0.5)
        fpo.rmsnorm_vjp(u, x[l].cuda(), gq[l].cuda(), two, eps=1e-6, min_rms=0.5)
        assert torch.equal(two, outs[l])


def test_repeated_entries_and_empty_tokens(fpo):
    wl = Workload("rep", T=40, d=256, d_ff=8, V=8, layers=1)
    g, m, gp, x, gq = _case(wl, 1)
    outs = [torch.empty((wl.T, wl.d), dtype=torch.bfloat16, device="cuda") for _ in range(4)]
    fpo.layer_signals(g.cuda(), outs, m=[m[0].cuda()] * 4, gamma_post=[gp[0].cuda()] * 4,
                      x=[x[0].cuda()] * 4, gamma_pre=[gq[0].cuda()] * 4)
    for o in outs[1:]:
        assert torch.equal(o, outs[0])
    e = torch.empty((0, 256), dtype=torch.bfloat16, device="cuda")
    fpo.layer_signals(e, [e.clone()], m=[e], gamma_post=[gp[0].cuda()])   # T = 0: no work


def test_argument_errors(fpo):
    wl = Workload("err", T=16, d=64, d_ff=8, V=8, layers=1)
    g, m, gp, x, gq = (t[0] if isinstance(t, list) else t for t in _case(wl, 1))
    g, m, gp, x, gq = (t.cuda() for t in (g, m, gp, x, gq))
    out = torch.empty_like(g)
    codes = {}
    for name, kw in {"none": {}, "half_post": {"m": [m]}, "half_pre": {"gamma_pre": [gq]}}.items():
        with pytest.raises(fpo.FpoError) as e:
            fpo.layer_signals(g, [out], **kw)
        codes[name] = e.value.code
    assert codes == {"none": 10, "half_post": 10, "half_pre": 10}       # FPO_ERR_ARG
    buf = torch.empty(wl.T * wl.d + 8, dtype=torch.bfloat16, device="cuda")
    mis = buf[1:1 + wl.T * wl.d].view(wl.T, wl.d)
    with pytest.raises(fpo.FpoError) as e:
        fpo.layer_signals(g, [out], x=[mis], gamma_pre=[gq])
    assert e.value.code == 4                                             # FPO_ERR_ALIGN
    g12 = torch.zeros((4, 12), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(fpo.FpoError) as e:
        fpo.layer_signals(g12, [torch.empty_like(g12)], x=[g12], gamma_pre=[g12[0]])
    assert e.value.code == 2                                             # FPO_ERR_SHAPE


PRE = Workload("pre-mlp-bf16", T=300, d=520, d_ff=600, V=1000, layers=3, targets="zipf",
               lr=1e-2)


@pytest.mark.parametrize("post", [False, True])
def test_pre_mlp_step_matches_oracle(fpo, post):
    """Qwen3 (pre-MLP only) and Gemma 3 (post-FFN, then pre-MLP) steps: error signal,
    layer signals, grouped update with per-layer signals, against the oracle chain."""
    wl = PRE
    inp = synth.make_all(wl)
    _, m, gp, x, gq = _case(wl, wl.layers)
    h, w, W_U, y = (inp[k].cuda() for k in ("h", "w", "W_U", "y"))
    g = torch.empty_like(h)
    ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms)
    assert fpo.get_device_status(ws) == fpo.OK
    gl = [torch.empty_like(g) for _ in range(wl.layers)]
    fpo.layer_signals(g, gl, m=[t.cuda() for t in m] if post else None,
                      gamma_post=[t.cuda() for t in gp] if post else None,
                      x=[t.cuda() for t in x], gamma_pre=[t.cuda() for t in gq], eps=wl.eps,
                      min_rms=wl.min_rms)
    Wm = [W.cuda() for W in inp["W"]]
    Go = [torch.empty(W.shape, dtype=torch.bfloat16, device="cuda") for W in inp["W"]]
    ws2 = fpo.layer_update_grouped_signals(gl, [a.cuda() for a in inp["A"]], wl.lr, W_masters=Wm,
                                           G_outs=Go)
    assert fpo.get_device_status(ws2) == fpo.OK
    e = synth.to_numpy_exact
    es = oracle.error_signal(e(inp["h"]), e(inp["w"]), e(inp["W_U"]), inp["y"].numpy(),
                             eps=wl.eps, min_rms=wl.min_rms, s=wl.loss_scale)
    for l in range(wl.layers):
        gref = oracle.layer_signal(es["g_tilde"], e(m[l]) if post else None,
                                   e(gp[l]) if post else None, e(x[l]), e(gq[l]), eps=wl.eps,
                                   min_rms=wl.min_rms)
        assert rel_frob(f64(gl[l]), gref) < 2e-2
        G = oracle.pseudograd(gref, e(inp["A"][l]))
        assert rel_frob(f64(Go[l]), G) < 2e-2 and cos(f64(Go[l]), G) >= 0.9995
        Wn, _ = oracle.sgd_update(inp["W"][l].numpy(), G, wl.lr)
        W0 = inp["W"][l].double().numpy()
        assert rel_frob(f64(Wm[l]) - W0, Wn.astype(np.float64) - W0) < 2e-2


@pytest.mark.slow
@pytest.mark.parametrize("post", [False, True])
def test_layer_signals_full_size_sampled_rows(fpo, post):
    """Qwen3-8B-shaped layers (T = 16384, d = 4096, 9 target layers; with the post-FFN
    norm the Gemma-3 layout), one launch for all layers, 12 sampled rows of every layer's
    signal (clamped rows 32 + 64 k of x and 64 k of m included) against the oracle."""
    wl = synth.WORKLOADS["qwen"]
    g = synth.normal((wl.T, wl.d), std=1e-4, seed=8, tensor="h", layer=11, device="cuda").to(
        torch.bfloat16)
    x = [synth.make_pre_norm_in(wl, l, device="cuda") for l in range(wl.layers)]
    gq = [synth.make_pre_norm_w(wl, l, device="cuda") for l in range(wl.layers)]
    m = [synth.make_mlp_out(wl, l, device="cuda") for l in range(wl.layers)] if post else None
    gp = [synth.make_post_norm_w(wl, l, device="cuda") for l in range(wl.layers)] if post else None
    outs = [torch.empty_like(g) for _ in range(wl.layers)]
    fpo.layer_signals(g, outs, m=m, gamma_post=gp, x=x, gamma_pre=gq)
    torch.cuda.synchronize()
    rows = [0, 1, 32, 64, 96, 8191, 8192, 12345, 16352, wl.T - 2, wl.T - 1, 5000]
    e = synth.to_numpy_exact
    for l in range(wl.layers):
        ref = oracle.layer_signal(e(g[rows]), e(m[l][rows]) if post else None,
                                  e(gp[l]) if post else None, e(x[l][rows]), e(gq[l]))
        got = f64(outs[l][rows])
        for r in range(len(rows)):
            assert rel_frob(got[r], ref[r]) < 2e-2
