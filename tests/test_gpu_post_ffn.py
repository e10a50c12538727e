"""Post-feedforward RMSNorm composition (OLMo-2 / Gemma 3, Sec. 3.2, App. E): the
closed-form VJP at each layer's cached MLP output (fpo_rmsnorm_vjp) and the grouped
update with one signal per layer (fpo_layer_update_grouped_signals), against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype,T,d,tol", [("bf16", 300, 520, 2e-2), ("f32", 77, 33, 1e-5),
                                            ("bf16", 1, 8, 2e-2)])
def test_rmsnorm_vjp_matches_oracle(fpo, dtype, T, d, tol):
    wl = Workload("vjp", T=T, d=d, d_ff=8, V=8, layers=1, dtype=dtype)
    g = synth.normal((T, d), std=1e-3, seed=5, tensor="h", layer=3).to(wl.torch_dtype)
    x = synth.make_mlp_out(wl, 0)
    gam = synth.make_post_norm_w(wl, 0)
    out = torch.empty((T, d), dtype=wl.torch_dtype, device="cuda")
    fpo.rmsnorm_vjp(g.cuda(), x.cuda(), gam.cuda(), out, eps=1e-6, min_rms=0.5)
    ref = oracle.rmsnorm_vjp(synth.to_numpy_exact(g), synth.to_numpy_exact(x),
                             synth.to_numpy_exact(gam), eps=1e-6, min_rms=0.5)
    got = f64(out)
    assert rel_frob(got, ref) < tol
    for t in range(T):  # every row, clamped outlier rows (every 64th) included
        assert rel_frob(got[t], ref[t]) < 2 * tol


POST = Workload("post-ffn-bf16", T=300, d=520, d_ff=600, V=1000, layers=3, targets="zipf",
                lr=1e-2)


def test_post_ffn_step_matches_oracle(fpo):
    wl = POST
    inp = synth.make_all(wl)
    m = [synth.make_mlp_out(wl, l) for l in range(wl.layers)]
    gp = [synth.make_post_norm_w(wl, l) for l in range(wl.layers)]
    h, w, W_U, y = (inp[k].cuda() for k in ("h", "w", "W_U", "y"))
    g = torch.empty_like(h)
    ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms)
    assert fpo.get_device_status(ws) == fpo.OK
    gl = [torch.empty_like(g) for _ in range(wl.layers)]
    for l in range(wl.layers):
        fpo.rmsnorm_vjp(g, m[l].cuda(), gp[l].cuda(), gl[l], eps=wl.eps, min_rms=wl.min_rms)
    Wm = [W.cuda() for W in inp["W"]]
    Go = [torch.empty(W.shape, dtype=torch.bfloat16, device="cuda") for W in inp["W"]]
    ws2 = fpo.layer_update_grouped_signals(gl, [a.cuda() for a in inp["A"]], wl.lr, W_masters=Wm,
                                           G_outs=Go)
    assert fpo.get_device_status(ws2) == fpo.OK
    es = oracle.error_signal(synth.to_numpy_exact(inp["h"]), synth.to_numpy_exact(inp["w"]),
                             synth.to_numpy_exact(inp["W_U"]), inp["y"].numpy(), eps=wl.eps,
                             min_rms=wl.min_rms, s=wl.loss_scale)
    for l in range(wl.layers):
        gref = oracle.rmsnorm_vjp(es["g_tilde"], synth.to_numpy_exact(m[l]),
                                  synth.to_numpy_exact(gp[l]), eps=wl.eps, min_rms=wl.min_rms)
        assert rel_frob(f64(gl[l]), gref) < 2e-2
        G = oracle.pseudograd(gref, synth.to_numpy_exact(inp["A"][l]))
        assert rel_frob(f64(Go[l]), G) < 2e-2 and cos(f64(Go[l]), G) >= 0.9995
        Wn, _ = oracle.sgd_update(inp["W"][l].numpy(), G, wl.lr)
        W0 = inp["W"][l].double().numpy()
        assert rel_frob(f64(Wm[l]) - W0, Wn.astype(np.float64) - W0) < 2e-2


def test_grouped_signals_with_one_signal_equals_grouped(fpo):
    wl = Workload("same", T=260, d=256, d_ff=520, V=8, layers=3)
    g = synth.normal((wl.T, wl.d), std=1e-2, seed=6, tensor="h").to(torch.bfloat16).cuda()
    A = [synth.make_A(wl, l).cuda() for l in range(wl.layers)]
    Ga = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device="cuda") for _ in A]
    Gb = [torch.empty_like(x) for x in Ga]
    fpo.layer_update_grouped(g, A, 0.0, G_outs=Ga)
    fpo.layer_update_grouped_signals([g] * wl.layers, A, 0.0, G_outs=Gb)
    for a, b in zip(Ga, Gb):
        assert torch.equal(a, b)


def test_rmsnorm_vjp_full_size_sampled_rows(fpo):
    # OLMo-2-7B-shaped post-FFN VJP for one layer, synthetic upstream signal
    wl = synth.WORKLOADS["olmo"]
    g = synth.normal((wl.T, wl.d), std=1e-4, seed=7, tensor="h", layer=9, device="cuda").to(
        torch.bfloat16)
    x = synth.make_mlp_out(wl, 0, device="cuda")
    gam = synth.make_post_norm_w(wl, 0, device="cuda")
    out = torch.empty_like(g)
    fpo.rmsnorm_vjp(g, x, gam, out)
    rows = [0, 64, 1, 8191, wl.T - 1, 12345]  # 0 and 64 are clamped outliers
    ref = oracle.rmsnorm_vjp(synth.to_numpy_exact(g[rows]), synth.to_numpy_exact(x[rows]),
                             synth.to_numpy_exact(gam))
    got = f64(out[rows])
    for r in range(len(rows)):
        assert rel_frob(got[r], ref[r]) < 2e-2
