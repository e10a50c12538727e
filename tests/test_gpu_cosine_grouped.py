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
