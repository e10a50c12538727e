"""fpo_cosine_grouped (Sec. 2.2, Eq. (cosine) for every target layer in one launch pair)
against the oracle's cosine, per layer, on the same seeded inputs."""
import math

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


def _pairs(L, n, dtype, seed=3):
    X, Y = [], []
    for l in range(L):
        x = synth.normal((n,), seed=seed, tensor="noise", layer=2 * l)
        y = x * (0.5 + 0.1 * l) + synth.normal((n,), seed=seed, tensor="noise", layer=2 * l + 1)
        X.append(x.to(dtype).cuda())
        Y.append(y.to(dtype).cuda())
    return X, Y


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("n", [1, 7, 8, 1000, 1000003])
def test_cosine_grouped_matches_oracle(fpo, dtype, n):
    X, Y = _pairs(4, n, dtype)
    out = fpo.cosine_grouped(X, Y).cpu().numpy()
    for l in range(4):
        ref = oracle.cosine(synth.to_numpy_exact(X[l].cpu()), synth.to_numpy_exact(Y[l].cpu()))
        for k in range(4):
            assert abs(out[l, k] - ref[k]) <= 1e-6 * max(abs(ref[k]), 1e-30) + 1e-12, (l, k)
    assert torch.equal(fpo.cosine_grouped(X, Y).cpu(), torch.from_numpy(out))


def test_cosine_grouped_agrees_with_single_and_zero_norms(fpo):
    X, Y = _pairs(3, 123457, torch.bfloat16, seed=9)
    X[1] = torch.zeros_like(X[1])
    out = fpo.cosine_grouped(X, Y).cpu().numpy()
    assert out[1, 3] == 0.0 and out[1, 1] == 0.0
    for l in (0, 2):
        single = fpo.cosine(X[l], Y[l]).cpu().numpy()
        assert np.allclose(out[l], single, rtol=1e-6, atol=0)


def test_cosine_grouped_diagnostic_closed_form(fpo):
    """36 Qwen-sized layers at once: noise of relative size sigma_l gives
    E[cos] = 1 / sqrt(1 + sigma_l^2) (the diagnostic's synthetic check)."""
    n = 4096 * 12288
    L = 36
    G, Gt, sig = [], [], []
    for l in range(L):
        base = synth.normal((n,), seed=1, tensor="noise", layer=1000 + l, device="cuda")
        sigma = 4.0 - 2.5 * l / (L - 1)
        Z = synth.make_noise(n, seed=1, layer=l, device="cuda")
        scale = sigma * torch.linalg.vector_norm(base).item() / math.sqrt(n)
        G.append(base.to(torch.bfloat16))
        Gt.append((base + scale * Z).to(torch.bfloat16))
        sig.append(sigma)
        del base, Z
    out = fpo.cosine_grouped(G, Gt).cpu().numpy()
    for l in range(L):
        assert abs(out[l, 3] - 1.0 / math.sqrt(1.0 + sig[l] ** 2)) < 2e-3, l
    del G, Gt
    torch.cuda.empty_cache()


def _grad_inputs(T, d, d_ff, L, dtype, seed=5):
    gen = torch.Generator(device="cuda").manual_seed(seed)
    g = (torch.randn(T, d, device="cuda", generator=gen) * 1e-2).to(dtype)
    A = [torch.randn(T, d_ff, device="cuda", generator=gen).to(dtype) for _ in range(L)]
    Y = [torch.randn(d, d_ff, device="cuda", generator=gen).to(dtype) for _ in range(L)]
    return g, A, Y


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("shape", [(700, 320, 840, 3), (1024, 512, 768, 2), (300, 1032, 264, 4)])
def test_layer_grad_cosine_matches_update_and_oracle(fpo, dtype, shape):
    """The pseudogradients with the diagnostic's cosine in one GEMM (the sums formed in its
    epilogue for bf16): G_l identical to the grouped update's, and each layer's sums and
    cosine against the oracle's cosine of the same stored G_l and Y_l (ragged d, d_ff, T)."""
    T, d, d_ff, L = shape
    g, A, Y = _grad_inputs(T, d, d_ff, L, dtype)
    G = [torch.full((d, d_ff), float("nan"), device="cuda").to(dtype) for _ in range(L)]
    out = fpo.layer_grad_cosine_grouped(g, A, Y, G).cpu().numpy()
    G_ref = [torch.empty(d, d_ff, device="cuda", dtype=dtype) for _ in range(L)]
    ws = fpo.layer_update_grouped(g, A, 0.0, G_outs=G_ref)
    assert fpo.get_device_status(ws) == fpo.OK
    for l in range(L):
        assert torch.equal(G[l], G_ref[l]), f"layer {l}"
        ref = oracle.cosine(synth.to_numpy_exact(G[l].reshape(-1).cpu()),
                            synth.to_numpy_exact(Y[l].reshape(-1).cpu()))
        assert abs(out[l, 0] - ref[0]) <= 2e-5 * math.sqrt(ref[1] * ref[2]), l
        assert abs(out[l, 1] - ref[1]) <= 2e-5 * ref[1] and abs(out[l, 2] - ref[2]) <= 2e-5 * ref[2]
        assert abs(out[l, 3] - ref[3]) <= 2e-5, l
    again = fpo.layer_grad_cosine_grouped(g, A, Y, G).cpu().numpy()
    assert np.array_equal(out, again)  # deterministic


def test_layer_grad_cosine_same_bits_under_every_kernel_variant(fpo):
    """Single-CTA and CTA-pair tiles give the same per-(32-row x 256-column) partial sums,
    so the cosines agree bit for bit, as G does."""
    g, A, Y = _grad_inputs(640, 704, 520, 3, torch.bfloat16, seed=8)
    outs = []
    prev = fpo.set_gemm_variant(0)
    try:
        for v in (0, 1, 2):
            fpo.set_gemm_variant(v)
            G = [torch.empty(704, 520, device="cuda", dtype=torch.bfloat16) for _ in range(3)]
            outs.append((fpo.layer_grad_cosine_grouped(g, A, Y, G).cpu(), G))
    finally:
        fpo.set_gemm_variant(prev)
    for o, G in outs[1:]:
        assert torch.equal(o, outs[0][0])
        for a, b in zip(G, outs[0][1]):
            assert torch.equal(a, b)


def test_layer_grad_cosine_empty_tokens(fpo):
    g, A, Y = _grad_inputs(0, 64, 128, 2, torch.bfloat16)
    G = [torch.full((64, 128), 1.0, device="cuda").to(torch.bfloat16) for _ in range(2)]
    out = fpo.layer_grad_cosine_grouped(g, A, Y, G).cpu().numpy()
    for l in range(2):
        assert torch.count_nonzero(G[l]).item() == 0
        assert out[l, 0] == 0.0 and out[l, 1] == 0.0 and out[l, 3] == 0.0
        assert out[l, 2] > 0.0
