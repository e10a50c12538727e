"""fpo_norm_ratio (App. C update-magnitude ratio ||G_l|| / ||W_l|| and the SGD rate of a
relative step, Sec. C.2) against the oracle on the same seeded inputs."""
import math

import pytest
import torch

import oracle
import synth
from synth import WORKLOADS

pytestmark = pytest.mark.gpu


def _exact(t):
    return synth.to_numpy_exact(t.cpu())


def _check(got, ref, tol):
    got = got.cpu().numpy()
    assert got.shape == ref.shape
    for l in range(ref.shape[0]):
        for k in range(4):
            assert abs(got[l, k] - ref[l, k]) <= tol * abs(ref[l, k]), (l, k, got[l, k], ref[l, k])


@pytest.mark.parametrize("gd,wd", [(torch.bfloat16, torch.float32), (torch.float32, torch.float32),
                                   (torch.bfloat16, torch.bfloat16), (torch.float32, torch.bfloat16)])
@pytest.mark.parametrize("n", [1, 5, 8, 13, 4099, 1000003])
def test_norm_ratio_matches_oracle(fpo, gd, wd, n):
    L = 3
    G = [(synth.normal((n,), std=10.0 ** (-2 - l), seed=5, tensor="noise", layer=l)).to(gd).cuda()
         for l in range(L)]
    W = [synth.normal((n,), std=0.02, seed=5, tensor="W", layer=l).to(wd).cuda() for l in range(L)]
    out = fpo.norm_ratio(G, W, rel_step=0.01)
    ref = oracle.norm_ratio([_exact(g) for g in G], [_exact(w) for w in W], rel=0.01)
    _check(out, ref, 1e-6)
    again = fpo.norm_ratio(G, W, rel_step=0.01)
    assert torch.equal(out, again)  # fixed reduction order


def test_norm_ratio_empty_and_zero_cases(fpo):
    z = [torch.zeros(0, dtype=torch.bfloat16, device="cuda")]
    out = fpo.norm_ratio(z, [torch.zeros(0, dtype=torch.float32, device="cuda")]).cpu().numpy()
    assert out[0, 0] == 0.0 and out[0, 1] == 0.0 and math.isnan(out[0, 2])
    G = [torch.zeros(64, dtype=torch.bfloat16, device="cuda")]
    W = [torch.ones(64, dtype=torch.float32, device="cuda")]
    out = fpo.norm_ratio(G, W).cpu().numpy()
    assert out[0, 2] == 0.0 and math.isinf(out[0, 3]) and out[0, 1] == 64.0


@pytest.mark.slow
def test_norm_ratio_of_a_full_size_update(fpo):
    """G_l from the grouped update at the OLMo-2-7B shape against the fp32 masters."""
    wl = WORKLOADS["olmo"]
    dev = torch.device("cuda")
    g = synth.normal((wl.T, wl.d), std=1e-2, seed=11, tensor="h", device=dev).to(torch.bfloat16)
    A = [synth.make_A(wl, l, dev) for l in range(wl.layers)]
    Wm = [synth.make_W_master(wl, l, dev) for l in range(wl.layers)]
    Go = [torch.empty(wl.d, wl.d_ff, dtype=torch.bfloat16, device=dev) for _ in range(wl.layers)]
    ws = fpo.layer_update_grouped(g, A, 0.0, G_outs=Go)
    assert fpo.get_device_status(ws) == fpo.OK
    del A
    out = fpo.norm_ratio(Go, Wm, rel_step=0.01)
    ref = oracle.norm_ratio([_exact(x) for x in Go], [x.cpu().numpy() for x in Wm], rel=0.01)
    _check(out, ref, 1e-6)
    del g, Wm, Go, ws
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
