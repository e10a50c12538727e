"""Parity at the full sizes of the four bf16 workloads (OLMo-2-7B, Qwen3-8B and
Falcon3-7B shapes, and the 36-layer diagnostic sweep), in the launch
configuration bench.py times (one error-signal call over all T tokens in the
default 8192-token chunks, one grouped update over every target layer), the
GPU's own g~ feeding the GPU's own update as in a step.

* fpo_error_signal: 64 sampled tokens against the oracle, token by token (tokens
  are independent until the contraction over T): both ends, both sides of every
  token-chunk boundary, and tokens whose target is the most frequent Zipf id.
* fpo_layer_update_grouped, every layer: whole rows of G_l (all d_ff entries) and
  of the updated fp32 master against the oracle's sums over all T tokens of the
  GPU's g~ (the contraction checked on the exact input the kernel saw).
* the chain from scratch: the GPU update restricted to the sampled tokens (the
  GPU's g~ rows) against the oracle's pseudogradient of the oracle's own g~ of
  those tokens.
* diagnostic sweep: whole rows and columns of G_l for four of the 36 layers
  against the oracle on the GPU's g~; the cosine reduction of every layer against
  the oracle's cosine of the same bf16 G_l and synthetic 'true' gradient
  G_l + sigma_l |G_l| Z / sqrt(n), and against its closed-form expectation
  1/sqrt(1 + sigma_l^2) (Sec. 2.2); the same G_l and cosines from the one-GEMM form
  (fpo_layer_grad_cosine_grouped) against those.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import synth
from helpers import cos, f64, rel_frob
from synth import WORKLOADS

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

TOL = 2e-2
COS_MIN = 0.9995
T_CHUNK = 8192  # the library's default token chunk (FPO_AUTO_T_CHUNK)


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def _sample_tokens(wl, y_host, k=64, seed=0):
    """k token indices: 0 and T-1, the last and first token of every chunk boundary,
    up to 8 tokens whose target is id 0 (the most frequent Zipf rank), then random."""
    fixed = {0, wl.T - 1}
    for b in range(T_CHUNK, wl.T, T_CHUNK):
        fixed |= {b - 1, b}
    top = np.flatnonzero(y_host == 0)[:8].tolist()
    fixed |= set(top)
    rng = np.random.default_rng(seed)
    rest = [int(t) for t in rng.permutation(wl.T) if int(t) not in fixed]
    return sorted(fixed | set(rest[: max(0, k - len(fixed))])), top


def _error_signal(fpo, wl, dev):
    h, w, W_U, y = (synth.make_h(wl, dev), synth.make_norm_w(wl, dev), synth.make_W_U(wl, dev),
                    synth.make_targets(wl, dev))
    g = torch.empty_like(h)
    lse = torch.empty(wl.T, dtype=torch.float32, device=dev)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms, lse_out=lse,
                          loss_out=loss)
    assert fpo.get_device_status(ws) == fpo.OK
    return h, w, W_U, y, g, lse, loss


def _check_sampled_tokens(wl, h, w, W_U, y, g, lse, rows):
    ref = oracle.error_signal(synth.to_numpy_exact(h[rows]), synth.to_numpy_exact(w),
                              synth.to_numpy_exact(W_U), y[rows].cpu().numpy(), eps=wl.eps,
                              min_rms=wl.min_rms, s=wl.loss_scale)
    got = f64(g[rows])
    for r in range(len(rows)):
        assert rel_frob(got[r], ref["g_tilde"][r]) < TOL, f"token {rows[r]}"
        assert cos(got[r], ref["g_tilde"][r]) >= COS_MIN, f"token {rows[r]}"
    assert np.max(np.abs(f64(lse[rows]) - ref["lse"])) < 1e-2
    return ref


@pytest.mark.parametrize("name", ["olmo", "qwen", "falcon"])
def test_full_step_full_size(fpo, name):
    wl = WORKLOADS[name]
    dev = torch.device("cuda")
    h, w, W_U, y, g, lse, loss = _error_signal(fpo, wl, dev)
    assert math.isfinite(loss.item()) and loss.item() > 0
    y_host = y.cpu().numpy()
    rows, top = _sample_tokens(wl, y_host, seed=sum(map(ord, name)))
    assert len(rows) >= 64
    if wl.targets == "zipf":
        assert len(top) > 0  # the most frequent target is among the sampled tokens
    ref = _check_sampled_tokens(wl, h, w, W_U, y, g, lse, rows)
    del h, W_U
    _free()

    A = [synth.make_A(wl, l, dev) for l in range(wl.layers)]
    W0 = [synth.make_W_master(wl, l, dev) for l in range(wl.layers)]
    Wm = [x.clone() for x in W0]
    Wo = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(wl.layers)]
    Go = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(wl.layers)]
    ws = fpo.layer_update_grouped(g, A, wl.lr, W_masters=Wm, W_outs=Wo, G_outs=Go)
    assert fpo.get_device_status(ws) == fpo.OK

    # whole rows of G_l and of the stepped master, every layer, on the GPU's own g~
    rng = np.random.default_rng(7)
    g_rows = sorted({0, wl.d - 1, *rng.integers(1, wl.d - 1, size=2).tolist()})
    gi = torch.tensor(g_rows, device=dev)
    g_cols = synth.to_numpy_exact(g[:, gi].contiguous())  # [T, rows] of g~
    for l in range(wl.layers):
        G_ref = oracle.pseudograd(g_cols, synth.to_numpy_exact(A[l]))  # [rows, d_ff]
        G_got = f64(Go[l][gi])
        assert rel_frob(G_got, G_ref) < TOL and cos(G_got, G_ref) >= COS_MIN, f"layer {l}"
        for r in range(len(g_rows)):
            assert cos(G_got[r], G_ref[r]) >= COS_MIN, f"layer {l} row {g_rows[r]}"
        w0, w1 = f64(W0[l][gi]), f64(Wm[l][gi])
        d_ref = -wl.lr * G_ref
        ulp = np.spacing(np.abs(w1).astype(np.float32)).astype(np.float64)
        assert rel_frob(w1 - w0, d_ref) < TOL + np.linalg.norm(ulp) / np.linalg.norm(d_ref)
        assert np.all(np.abs(f64(Wo[l][gi]) - w1) <= np.abs(w1) * 2.0 ** -8)  # bf16 cast

    # the chain from scratch on the sampled tokens: oracle g~ -> oracle G, against the GPU
    # g~ rows -> the GPU update kernel
    ti = torch.tensor(rows, device=dev)
    g_s = g[ti].contiguous()
    A_s = [A[l][ti].contiguous() for l in (0, wl.layers - 1)]
    G_s = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in A_s]
    ws2 = fpo.layer_update_grouped(g_s, A_s, 0.0, G_outs=G_s)
    assert fpo.get_device_status(ws2) == fpo.OK
    for k in range(len(A_s)):
        G_ref = oracle.pseudograd(ref["g_tilde"], synth.to_numpy_exact(A_s[k]))
        G_got = f64(G_s[k])
        assert rel_frob(G_got, G_ref) < TOL and cos(G_got, G_ref) >= COS_MIN
    del g, A, W0, Wm, Wo, Go, ws, ws2, g_s, A_s, G_s
    _free()


def test_diagnostic_sweep_full_size(fpo):
    wl = WORKLOADS["diag"]
    dev = torch.device("cuda")
    h, w, W_U, y, g, lse, _ = _error_signal(fpo, wl, dev)
    rows, _ = _sample_tokens(wl, y.cpu().numpy(), seed=11)
    _check_sampled_tokens(wl, h, w, W_U, y, g, lse, rows)
    del h, W_U
    _free()
    L = wl.layers
    n = wl.d * wl.d_ff
    A = [synth.make_A(wl, l, dev) for l in range(L)]
    G = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    ws2 = fpo.layer_update_grouped(g, A, 0.0, G_outs=G)  # G only: no master, no step
    assert fpo.get_device_status(ws2) == fpo.OK

    # whole rows and columns of G_l for four layers, on the GPU's own g~
    g_np = synth.to_numpy_exact(g)
    ri, cj = [0, 1234, wl.d - 1], [0, 5555, wl.d_ff - 1]
    for l in (0, 11, 24, L - 1):
        A_np = synth.to_numpy_exact(A[l])
        G_rows = oracle.pseudograd(np.ascontiguousarray(g_np[:, ri]), A_np)
        G_cols = oracle.pseudograd(g_np, np.ascontiguousarray(A_np[:, cj]))
        got_r, got_c = f64(G[l][ri]), f64(G[l][:, cj])
        assert rel_frob(got_r, G_rows) < TOL and cos(got_r, G_rows) >= COS_MIN, f"layer {l}"
        assert rel_frob(got_c, G_cols) < TOL and cos(got_c, G_cols) >= COS_MIN, f"layer {l}"

    G_true = []
    for l in range(L):
        sigma = 4.0 - 2.5 * l / (L - 1)
        Gf = G[l].float().reshape(-1)
        scale = sigma * torch.linalg.vector_norm(Gf).item() / math.sqrt(n)
        Z = synth.make_noise(n, seed=wl.seed, layer=l, device=dev)
        G_true.append((Gf + scale * Z).to(torch.bfloat16).view(wl.d, wl.d_ff))
        del Gf, Z
    # the same G_l with the cosines formed in the update GEMM's epilogue
    G2 = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(L)]
    fused = fpo.layer_grad_cosine_grouped(g, A, G_true, G2).cpu().numpy()
    del A
    _free()

    for l in range(L):
        sigma = 4.0 - 2.5 * l / (L - 1)
        assert torch.equal(G2[l], G[l]), f"layer {l}"
        out = fpo.cosine(G[l].reshape(-1), G_true[l].reshape(-1)).cpu().numpy()
        for k in range(3):
            assert abs(fused[l, k] - out[k]) <= 1e-5 * math.sqrt(out[1] * out[2]), (l, k)
        assert abs(fused[l, 3] - out[3]) < 1e-5, f"layer {l}"
        assert abs(out[3] - 1.0 / math.sqrt(1.0 + sigma * sigma)) < 2e-3, f"layer {l}"
        ref = oracle.cosine(synth.to_numpy_exact(G[l].reshape(-1)),
                            synth.to_numpy_exact(G_true[l].reshape(-1)))
        assert abs(out[3] - ref[3]) < 1e-4, f"layer {l}"
        # fp32 runs of a few hundred elements per thread, fp64 after that
        assert abs(out[0] - ref[0]) <= 1e-5 * math.sqrt(ref[1] * ref[2]), f"layer {l}"
        assert abs(out[1] - ref[1]) <= 1e-5 * ref[1] and abs(out[2] - ref[2]) <= 1e-5 * ref[2]
    del G, G2, G_true, g, ws2
    _free()
