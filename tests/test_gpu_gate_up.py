"""Gate / up (W1 / W2) updates through the cached W3_init feedback (Sec. 3.1 step 5,
Eq. errh) on a SwiGLU MLP: fpo_gate_up_signals and the grouped update of W1, W2 against
the oracle."""
import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu


def _inputs(wl, layer=0, device="cpu"):
    g = synth.normal((wl.T, wl.d), std=1e-3, seed=wl.seed, tensor="h", layer=7,
                     device=device).to(wl.torch_dtype)
    W3 = synth.make_W_master(wl, layer, device).to(wl.torch_dtype)  # W3_init in the working dtype
    a, b = synth.make_gate_up(wl, layer, device)
    return g, W3, a, b


@pytest.mark.parametrize("dtype,shape,tol", [("bf16", (300, 136, 264), 2e-2),
                                             ("f32", (70, 33, 65), 1e-5),
                                             ("bf16", (1, 8, 8), 2e-2)])
def test_gate_up_signals_match_oracle(fpo, dtype, shape, tol):
    T, d, d_ff = shape
    wl = Workload("gu", T=T, d=d, d_ff=d_ff, V=8, layers=1, dtype=dtype, seed=3)
    g, W3, a, b = _inputs(wl)
    dA = torch.empty((T, d_ff), dtype=wl.torch_dtype, device="cuda")
    dB = torch.empty_like(dA)
    ws = fpo.gate_up_signals(g.cuda(), W3.cuda(), a.cuda(), b.cuda(), dA, dB)
    assert fpo.get_device_status(ws) == fpo.OK
    rA, rB = oracle.gate_up_signals(*(synth.to_numpy_exact(t) for t in (g, W3, a, b)))
    assert rel_frob(f64(dA), rA) < tol and rel_frob(f64(dB), rB) < tol


def test_gate_up_weight_update_matches_oracle(fpo):
    wl = Workload("gu-step", T=300, d=136, d_ff=264, V=8, layers=2, lr=0.5, seed=4)
    sig, acts, W1m, W2m, refs = [], [], [], [], []
    for l in range(wl.layers):
        g, W3, a, b = _inputs(wl, l)
        x = synth.make_mlp_in(wl, l)
        dA = torch.empty((wl.T, wl.d_ff), dtype=torch.bfloat16, device="cuda")
        dB = torch.empty_like(dA)
        fpo.gate_up_signals(g.cuda(), W3.cuda(), a.cuda(), b.cuda(), dA, dB)
        W1, W2 = synth.make_gate_up_master(wl, l)
        sig += [dA, dB]
        acts += [x.cuda(), x.cuda()]
        W1m.append(W1.cuda())
        W2m.append(W2.cuda())
        rA, rB = oracle.gate_up_signals(*(synth.to_numpy_exact(t) for t in (g, W3, a, b)))
        xn = synth.to_numpy_exact(x)
        refs.append((W1, oracle.pseudograd(rA, xn)))
        refs.append((W2, oracle.pseudograd(rB, xn)))
    masters = [m for pair in zip(W1m, W2m) for m in pair]
    Go = [torch.empty(m.shape, dtype=torch.bfloat16, device="cuda") for m in masters]
    ws = fpo.layer_update_grouped_signals(sig, acts, wl.lr, W_masters=masters, G_outs=Go)
    assert fpo.get_device_status(ws) == fpo.OK
    for k, (W0, G) in enumerate(refs):
        assert G.shape == (wl.d_ff, wl.d)
        assert rel_frob(f64(Go[k]), G) < 2e-2 and cos(f64(Go[k]), G) >= 0.9995
        Wn, _ = oracle.sgd_update(W0.numpy(), G, wl.lr)
        w0 = W0.double().numpy()
        assert rel_frob(f64(masters[k]) - w0, Wn.astype(np.float64) - w0) < 2e-2


def test_gate_up_signals_full_size_sampled_rows(fpo):
    wl = synth.WORKLOADS["olmo"]
    g, W3, a, b = _inputs(wl, 0, device="cuda")
    dA = torch.empty((wl.T, wl.d_ff), dtype=torch.bfloat16, device="cuda")
    dB = torch.empty_like(dA)
    ws = fpo.gate_up_signals(g, W3, a, b, dA, dB)
    assert fpo.get_device_status(ws) == fpo.OK
    rows = [0, 1, 4097, wl.T - 1]
    sel = lambda t: synth.to_numpy_exact(t[rows])
    rA, rB = oracle.gate_up_signals(sel(g), synth.to_numpy_exact(W3), sel(a), sel(b))
    for r in range(len(rows)):
        assert rel_frob(f64(dA[rows[r]]), rA[r]) < 2e-2
        assert rel_frob(f64(dB[rows[r]]), rB[r]) < 2e-2
