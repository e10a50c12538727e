"""Parity at the full sizes of the four bf16 workloads (OLMo-2-7B, Qwen3-8B and
Falcon3-7B shapes, and the 36-layer diagnostic sweep), in the launch
configuration bench.py times (one error-signal call over all T tokens, one
grouped update over every target layer).

* fpo_error_signal: sampled tokens against the oracle, token by token
  (tokens are independent until the contraction over T).
* fpo_layer_update_grouped: a seeded synthetic g~ (not produced by the GPU)
  and every layer's A_l; sampled entries of G_l and of the updated master
  against the oracle's sums over all T tokens.
* diagnostic sweep: G_l for 36 layers from the GPU path, synthetic 'true'
  gradients G_l + sigma_l |G_l| Z / sqrt(n), and the cosine reduction checked
  against its closed-form expectation 1/sqrt(1 + sigma_l^2) (Sec. 2.2).
"""
import math

import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
from paper_2608_14563_gb300 import synth
from paper_2608_14563_gb300.synth import WORKLOADS

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

TOL = 2e-2
COS_MIN = 0.9995


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _sample_rows(T, k, seed):
    g = torch.Generator().manual_seed(seed)
    rows = torch.randperm(T, generator=g)[: k - 2].tolist()
    return sorted(set([0, T - 1] + rows))


@pytest.mark.parametrize("name", ["olmo", "qwen", "falcon", "diag"])
def test_error_signal_sampled_tokens_full_size(fpo, name):
    wl = WORKLOADS[name]
    dev = torch.device("cuda")
    h, w, W_U, y = (synth.make_h(wl, dev), synth.make_norm_w(wl, dev), synth.make_W_U(wl, dev),
                    synth.make_targets(wl, dev))
    g = torch.empty_like(h)
    lse = torch.empty(wl.T, dtype=torch.float32, device=dev)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms, lse_out=lse,
                          loss_out=loss)
    assert fpo.get_device_status(ws) == fpo.OK
    rows = _sample_rows(wl.T, 10, seed=sum(map(ord, name)))
    ref = oracle.error_signal(synth.to_numpy_exact(h[rows]), synth.to_numpy_exact(w),
                              synth.to_numpy_exact(W_U), y[rows].cpu().numpy(), eps=wl.eps,
                              min_rms=wl.min_rms, s=wl.loss_scale)
    got = f64(g[rows])
    for r in range(len(rows)):
        assert rel_frob(got[r], ref["g_tilde"][r]) < TOL, f"token {rows[r]}"
        assert cos(got[r], ref["g_tilde"][r]) >= COS_MIN
    assert np.max(np.abs(f64(lse[rows]) - ref["lse"])) < 1e-2
    assert math.isfinite(loss.item()) and loss.item() > 0
    del h, w, W_U, y, g, ws
    _free()


@pytest.mark.parametrize("name", ["olmo", "qwen", "falcon"])
def test_layer_update_sampled_entries_full_size(fpo, name):
    wl = WORKLOADS[name]
    dev = torch.device("cuda")
    g = synth.normal((wl.T, wl.d), std=1e-2, seed=11, tensor="h", device=dev).to(torch.bfloat16)
    A = [synth.make_A(wl, l, dev) for l in range(wl.layers)]
    W0 = [synth.make_W_master(wl, l, dev) for l in range(wl.layers)]
    Wm = [x.clone() for x in W0]
    Wo = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(wl.layers)]
    Go = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(wl.layers)]
    ws = fpo.layer_update_grouped(g, A, wl.lr, W_masters=Wm, W_outs=Wo, G_outs=Go)
    assert fpo.get_device_status(ws) == fpo.OK
    gen = torch.Generator().manual_seed(7)
    ii = torch.randint(0, wl.d, (48,), generator=gen)
    jj = torch.randint(0, wl.d_ff, (48,), generator=gen)
    ii[0], jj[0] = wl.d - 1, wl.d_ff - 1  # last tile corner
    ui, inv_i = torch.unique(ii, return_inverse=True)
    uj, inv_j = torch.unique(jj, return_inverse=True)
    g_cols = synth.to_numpy_exact(g[:, ui.to(dev)].contiguous())
    for l in (0, wl.layers // 2, wl.layers - 1):
        a_cols = synth.to_numpy_exact(A[l][:, uj.to(dev)].contiguous())
        G_ref = oracle.pseudograd(g_cols, a_cols, pairs=(inv_i.numpy(), inv_j.numpy()))
        G_got = f64(Go[l][ii.to(dev), jj.to(dev)])
        assert rel_frob(G_got, G_ref) < TOL and cos(G_got, G_ref) >= COS_MIN, f"layer {l}"
        w0 = f64(W0[l][ii.to(dev), jj.to(dev)])
        w1 = f64(Wm[l][ii.to(dev), jj.to(dev)])
        d_ref = -wl.lr * G_ref
        ulp = np.spacing(np.abs(w1).astype(np.float32)).astype(np.float64)
        assert rel_frob(w1 - w0, d_ref) < TOL + np.linalg.norm(ulp) / np.linalg.norm(d_ref)
        wo = f64(Wo[l][ii.to(dev), jj.to(dev)])
        assert np.all(np.abs(wo - w1) <= np.abs(w1) * 2.0 ** -8)  # bf16 cast of the master
    del g, A, W0, Wm, Wo, Go, ws
    _free()


def test_diagnostic_sweep_cosines_match_closed_form(fpo):
    wl = WORKLOADS["diag"]
    dev = torch.device("cuda")
    h, w, W_U, y = (synth.make_h(wl, dev), synth.make_norm_w(wl, dev), synth.make_W_U(wl, dev),
                    synth.make_targets(wl, dev))
    g = torch.empty_like(h)
    ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms)
    assert fpo.get_device_status(ws) == fpo.OK
    del h, W_U
    L = wl.layers
    n = wl.d * wl.d_ff
    A = [synth.make_A(wl, l, dev) for l in range(L)]
    G = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    ws2 = fpo.layer_update_grouped(g, A, 0.0, G_outs=G)  # G only: no master, no step
    assert fpo.get_device_status(ws2) == fpo.OK
    del A
    _free()
    for l in range(L):
        sigma = 4.0 - 2.5 * l / (L - 1)
        Gf = G[l].float().reshape(-1)
        scale = sigma * torch.linalg.vector_norm(Gf).item() / math.sqrt(n)
        Z = synth.make_noise(n, seed=wl.seed, layer=l, device=dev)
        G_true = (Gf + scale * Z).to(torch.bfloat16)
        out = fpo.cosine(G[l].reshape(-1), G_true).cpu().numpy()
        assert abs(out[3] - 1.0 / math.sqrt(1.0 + sigma * sigma)) < 2e-3, f"layer {l}"
        del Gf, Z, G_true
    del G, g, ws, ws2
    _free()
