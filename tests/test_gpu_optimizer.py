"""Optimizer row (Sec. 3.1 AdamW / SGD with momentum, App. A relative clip) through
fpo_layer_optimize_grouped against the oracle's optimizer step on the oracle's G."""
import numpy as np
import pytest
import torch

import oracle
from helpers import f64, rel_frob
import synth
from synth import Workload

pytestmark = pytest.mark.gpu

KINDS = {"sgd": 0, "sgdm": 1, "adamw": 2}
CLIPS = {"none": 0, "step": 1, "grad": 2}


def _case(dtype, seed):
    if dtype == "bf16":
        wl = Workload("opt-bf16", T=300, d=136, d_ff=264, V=8, layers=2, seed=seed)
    else:
        wl = Workload("opt-f32", T=70, d=33, d_ff=65, V=8, layers=2, dtype="f32", seed=seed)
    gs = [synth.normal((wl.T, wl.d), std=1e-2, seed=seed, tensor="h", layer=l).to(wl.torch_dtype)
          for l in range(wl.layers)]
    A = [synth.make_A(wl, l) for l in range(wl.layers)]
    W = [synth.make_W_master(wl, l) for l in range(wl.layers)]
    return wl, gs, A, W


def _states(wl, Gs, kind, t):
    """Optimizer state before step t (zero at t = 1, synthetic and consistent otherwise)."""
    s1, s2 = [], []
    for l, G in enumerate(Gs):
        sc = float(np.sqrt(np.mean(G * G)))
        if t == 1:
            s1.append(np.zeros(G.shape, np.float32))
            s2.append(np.zeros(G.shape, np.float32))
        else:
            a = synth.normal(G.shape, std=sc, seed=wl.seed, tensor="noise", layer=10 + l).numpy()
            b = synth.normal(G.shape, std=1.0, seed=wl.seed, tensor="noise", layer=20 + l).numpy()
            s1.append(a.astype(np.float32))
            s2.append((sc * sc * (0.5 + np.abs(b))).astype(np.float32))
    return s1, s2


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("kind", list(KINDS))
@pytest.mark.parametrize("clip", list(CLIPS))
def test_optimizer_step_matches_oracle(fpo, dtype, kind, clip):
    wl, gs, A, W = _case(dtype, seed=40 + 3 * KINDS[kind] + CLIPS[clip])
    Gs = [oracle.pseudograd(synth.to_numpy_exact(g), synth.to_numpy_exact(a)) for g, a in zip(gs, A)]
    t = 1 if kind == "sgdm" else 3
    s1, s2 = _states(wl, Gs, kind, t)
    lr = {"sgd": 0.5, "sgdm": 0.05, "adamw": 2e-3}[kind]
    opt = fpo.optimizer_desc(KINDS[kind], lr=lr, clip=CLIPS[clip], step=t)
    Wm = [w.cuda() for w in W]
    Wo = [torch.empty(w.shape, dtype=wl.torch_dtype, device="cuda") for w in W]
    S1 = [torch.from_numpy(x).cuda() for x in s1] if kind != "sgd" else None
    S2 = [torch.from_numpy(x).cuda() for x in s2] if kind == "adamw" else None
    ws = fpo.layer_optimize_grouped([g.cuda() for g in gs], [a.cuda() for a in A], opt, Wm,
                                    W_outs=Wo, states1=S1, states2=S2)
    assert fpo.get_device_status(ws) == fpo.OK
    tol = 2e-2 if dtype == "bf16" else 1e-5
    for l in range(wl.layers):
        ref = oracle.optimizer_step(W[l].numpy(), Gs[l], kind=KINDS[kind], lr=lr, t=t,
                                    clip=CLIPS[clip], s1=s1[l], s2=s2[l])
        W0 = W[l].double().numpy()
        d_ref = ref["W"].astype(np.float64) - W0
        ulp = np.spacing(np.abs(ref["W"]).astype(np.float32)).astype(np.float64)
        q = np.linalg.norm(ulp) / np.linalg.norm(d_ref)
        d_got = f64(Wm[l]) - W0
        assert rel_frob(d_got, d_ref) < tol + q, f"layer {l}"
        if clip != "none" and ref["scale"] < 1.0:
            # an active clip pins the step (or the gradient) at 1% of ||W||
            if clip == "step":
                assert abs(np.linalg.norm(d_got) / (0.01 * np.linalg.norm(W0)) - 1) < 1e-3
        if kind != "sgd":
            assert rel_frob(f64(S1[l]), ref["s1"]) < tol
        if kind == "adamw":
            assert rel_frob(f64(S2[l]), ref["s2"]) < tol
        assert rel_frob(f64(Wo[l]), ref["W"]) < max(tol, 4e-3 if dtype == "bf16" else 0)


def test_clip_is_active_in_the_step_cases(fpo):
    # guard: the parametrised cases above do exercise an active clip
    wl, gs, A, W = _case("bf16", seed=40 + 3 * 2 + 1)
    G = oracle.pseudograd(synth.to_numpy_exact(gs[0]), synth.to_numpy_exact(A[0]))
    s1, s2 = _states(wl, [G], "adamw", 3)
    r = oracle.optimizer_step(W[0].numpy(), G, kind=2, lr=2e-3, t=3, clip=1, s1=s1[0], s2=s2[0])
    assert r["scale"] < 1.0
    r = oracle.optimizer_step(W[0].numpy(), G, kind=0, lr=0.5, clip=2)
    assert r["scale"] < 1.0


@pytest.mark.parametrize("clip", ["none", "step"])
def test_optimizer_step_with_no_tokens(fpo, clip):
    """T = 0: G = 0, and AdamW still steps (decayed moments, weight decay), through the
    stand-alone passes whatever the clip (the fused pass needs a GEMM with tokens)."""
    wl, gs, A, W = _case("bf16", seed=77)
    g0 = [torch.zeros((0, wl.d), dtype=torch.bfloat16, device="cuda") for _ in range(wl.layers)]
    A0 = [torch.zeros((0, wl.d_ff), dtype=torch.bfloat16, device="cuda") for _ in range(wl.layers)]
    Gs = [np.zeros((wl.d, wl.d_ff)) for _ in range(wl.layers)]
    s1, s2 = _states(wl, [np.full((wl.d, wl.d_ff), 1e-3) for _ in range(wl.layers)], "adamw", 3)
    opt = fpo.optimizer_desc(2, lr=2e-3, clip=CLIPS[clip], step=3)
    Wm = [w.cuda() for w in W]
    S1 = [torch.from_numpy(x).cuda() for x in s1]
    S2 = [torch.from_numpy(x).cuda() for x in s2]
    ws = fpo.layer_optimize_grouped(g0, A0, opt, Wm, states1=S1, states2=S2)
    assert fpo.get_device_status(ws) == fpo.OK
    for l in range(wl.layers):
        ref = oracle.optimizer_step(W[l].numpy(), Gs[l], kind=2, lr=2e-3, t=3, clip=CLIPS[clip],
                                    s1=s1[l], s2=s2[l])
        W0 = W[l].double().numpy()
        assert rel_frob(f64(Wm[l]) - W0, ref["W"].astype(np.float64) - W0) < 1e-4
        assert rel_frob(f64(S1[l]), ref["s1"]) < 1e-6
        assert rel_frob(f64(S2[l]), ref["s2"]) < 1e-6


@pytest.mark.slow
def test_adamw_step_clip_full_size(fpo):
    """OLMo-2-7B-shaped layers (T = 16384, d = 4096, d_ff = 11008, 8 layers; bf16, so the
    step clip's first pass runs in the GEMM's epilogue), AdamW's first step with the clip
    active: every layer's ||dW|| is clip_frac ||W||, and 4 sampled rows of each dW are the
    oracle's AdamW step rows (from the oracle's G rows over all T tokens) times one common
    factor per layer.  AdamW's first step is lr (G / (|G| + eps) + wd W), a sign where
    |G| >> eps: elements whose G is within the GPU's fp32 accumulation error over 16384
    tokens of zero (|G| < 1e-4 rms(G), ~1e-4 of them; one at 9.5e-8 came out at -2.2e-8)
    may take either sign, and are left out of the row comparison."""
    wl = synth.WORKLOADS["olmo"]
    L = wl.layers
    g = synth.normal((wl.T, wl.d), std=1e-4, seed=9, tensor="h", layer=13, device="cuda").to(
        torch.bfloat16)
    A = [synth.make_A(wl, l, device="cuda") for l in range(L)]
    W0 = [synth.make_W_master(wl, l, device="cuda") for l in range(L)]
    Wm = [w.clone() for w in W0]
    S1 = [torch.zeros_like(w) for w in W0]
    S2 = [torch.zeros_like(w) for w in W0]
    lr, frac = 1e-3, 0.01
    opt = fpo.optimizer_desc(2, lr=lr, clip=1, clip_frac=frac, step=1)
    ws = fpo.layer_optimize_grouped([g] * L, A, opt, Wm, states1=S1, states2=S2)
    assert fpo.get_device_status(ws) == fpo.OK
    rows = [0, 1234, 2048, wl.d - 1]
    gcol = synth.to_numpy_exact(g[:, rows].contiguous())
    for l in range(L):
        dW = (Wm[l] - W0[l]).double()
        ratio = float(dW.norm() / W0[l].double().norm())
        assert abs(ratio - frac) < 1e-4 * frac
        G = oracle.pseudograd(gcol, synth.to_numpy_exact(A[l]))          # [4, d_ff]
        w_rows = W0[l][rows].double().cpu().numpy()
        step = -lr * (G / (np.abs(G) + 1e-8) + 0.01 * w_rows)              # AdamW, t = 1
        got = dW[rows].cpu().numpy()
        keep = np.abs(G) > 1e-4 * np.sqrt(np.mean(G * G))
        assert keep.mean() > 0.999
        got, step = got[keep], step[keep]
        s = np.sum(got * step) / np.sum(step * step)                       # common factor
        assert 0.0 < s < 1.0
        assert rel_frob(got, s * step) < 2e-3
