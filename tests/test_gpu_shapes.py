"""A seeded sweep of ragged shapes through the whole bf16 step (error signal + grouped
update) against the fp64 oracle, for every error-matrix algorithm and GEMM kernel
variant: tile overhangs in M, N and K of all three GEMMs, and the vocabulary tails of the
logits pass."""
import numpy as np
import pytest
import torch

import oracle
from helpers import cos, f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu

TOL = 2e-2


def _shapes(n, seed=2024):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        T = int(rng.integers(1, 700))
        d = 8 * int(rng.integers(1, 90))
        V = 8 * int(rng.integers(1, 260))
        d_ff = 8 * int(rng.integers(1, 90))
        out.append((T, d, V, d_ff))
    return out


SHAPES = _shapes(12)


@pytest.mark.parametrize("variant", [0, 1, 2])
@pytest.mark.parametrize("algo", [1, 2, 3])  # recompute, stored logits, direct
@pytest.mark.parametrize("shape", SHAPES, ids=[f"T{t}d{d}V{v}f{f}" for t, d, v, f in SHAPES])
def test_random_ragged_shapes(fpo, shape, algo, variant):
    T, d, V, d_ff = shape
    wl = Workload("sweep", T=T, d=d, d_ff=d_ff, V=V, layers=2, targets="zipf", lr=1e-2,
                  seed=T + d)
    inp = synth.make_all(wl)
    h, w, W_U, y = (inp[k].cuda() for k in ("h", "w", "W_U", "y"))
    prev = fpo.set_gemm_variant(variant)
    try:
        g = torch.empty_like(h)
        ws = fpo.error_signal(h, w, W_U, y, g, eps=wl.eps, min_rms=wl.min_rms, algo=algo,
                              t_chunk=(T + 1) // 2)
        assert fpo.get_device_status(ws) == fpo.OK
        A = [a.cuda() for a in inp["A"]]
        Go = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
        ws2 = fpo.layer_update_grouped(g, A, 0.0, G_outs=Go)
        assert fpo.get_device_status(ws2) == fpo.OK
    finally:
        fpo.set_gemm_variant(prev)
    es = oracle.error_signal(synth.to_numpy_exact(inp["h"]), synth.to_numpy_exact(inp["w"]),
                             synth.to_numpy_exact(inp["W_U"]), inp["y"].numpy(), eps=wl.eps,
                             min_rms=wl.min_rms, s=wl.loss_scale)
    gg = f64(g)
    assert rel_frob(gg, es["g_tilde"]) < TOL and cos(gg, es["g_tilde"]) >= 0.9995
    for l in range(2):
        G = oracle.pseudograd(es["g_tilde"], synth.to_numpy_exact(inp["A"][l]))
        Gg = f64(Go[l])
        assert rel_frob(Gg, G) < TOL and cos(Gg, G) >= 0.9995, l
