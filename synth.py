"""Seeded synthetic inputs for the FPO pseudogradient update.

This module only draws inputs; it contains none of the method's arithmetic,
and it is the one piece of code that both the CUDA path's tests and the oracle
tests use.  It sits outside the library package, so importing it loads no
native code: the oracle-only benchmark arm uses it without touching libfpo.  It stands in for the paper's forward-pass caches (Sec. 3.1 step 1:
the final pre-norm residual and each target layer's down-projection input)
and for its adaptation corpora (Sec. 4: packed 2048-token sequences), which
are not available here.

Recipe (every tensor has its own generator seeded from (seed, tensor, layer)):

* h      ~ N(0, 1)                      final pre-norm residual     [T, d]
* w      = 1 + 0.1 N(0, 1)              final RMSNorm weight        [d]
* W_U    ~ N(0, 0.02^2)                 unembedding (lm_head)       [V, d]
* A_l    = SiLU(N(0, 1)) * N(0, 1)      down-projection input       [T, d_ff] per layer
* W_l    ~ N(0, 0.02^2), fp32 master    down-projection weight      [d, d_ff] per layer
* y      uniform on [0, V), or Zipf(1.1) over token ranks (P(r) ~ r^-1.1,
         token id = r - 1, inverse-CDF on an fp64 CDF table)         [T] int32
* m_l    = N(0, 1) * exp(0.5 N(0, 1)) per token, every 64th token x 0.1
         (the per-layer MLP output feeding a post-FFN norm: per-token RMS
         varies widely and a few outlier tokens sit near 0.1)      [T, d] per layer
* gp_l   = 0.3 + 0.05 N(0, 1)         post-FFN RMSNorm weight      [d] per layer
* a_l, b_l  the two N(0, 1) draws behind A_l (gate and up pre-activations of
         the SwiGLU MLP, A_l = SiLU(a_l) b_l)                         [T, d_ff] per layer
* x_l    ~ N(0, 1)                      MLP input (after its norm)  [T, d] per layer
* W1_l, W2_l ~ N(0, 0.02^2), fp32 master  gate / up weights          [d_ff, d] per layer

Tensors are generated in fp32 and rounded to the storage dtype by torch.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch

_TENSOR_IDS = {"h": 1, "w": 2, "W_U": 3, "A": 4, "W": 5, "y": 6, "noise": 7, "m": 8, "gp": 9,
               "x": 10, "W1": 11, "W2": 12, "xpre": 13, "gq": 14}


@dataclass(frozen=True)
class Workload:
    """Shapes and hyperparameters of one synthetic FPO workload."""

    name: str
    T: int
    d: int
    d_ff: int
    V: int
    layers: int
    dtype: str = "bf16"          # "bf16" or "f32"
    targets: str = "uniform"     # "uniform" or "zipf"
    lr: float = 1e-4
    eps: float = 1e-6
    min_rms: float = 0.5
    seed: int = 0
    extra: dict = field(default_factory=dict, compare=False, hash=False)

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    @property
    def loss_scale(self) -> float:
        """Mean-reduced cross-entropy: s = 1/T."""
        return 1.0 / self.T if self.T > 0 else 1.0


# The five workloads of the benchmark set (shapes of models the paper trains and probes,
# packed 2048-token sequences, last 25% of layers as targets).
WORKLOADS = {
    "tiny": Workload("tiny-f32", T=128, d=64, d_ff=256, V=512, layers=2, dtype="f32",
                     targets="uniform", lr=1e-3),
    "olmo": Workload("olmo2-7b-shaped", T=8 * 2048, d=4096, d_ff=11008, V=100352, layers=8,
                     targets="zipf"),
    "qwen": Workload("qwen3-8b-shaped", T=8 * 2048, d=4096, d_ff=12288, V=151936, layers=9,
                     targets="zipf"),
    "falcon": Workload("falcon3-7b-shaped", T=16 * 2048, d=3072, d_ff=23040, V=131072, layers=7,
                       targets="uniform"),
    "diag": Workload("diag-qwen3-8b-shaped", T=4096, d=4096, d_ff=12288, V=151936, layers=36,
                     targets="zipf", lr=0.0),
}


def _gen(seed: int, tensor: str, layer: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed((seed * 1_000_003 + _TENSOR_IDS[tensor] * 10_007 + layer) & 0x7FFF_FFFF_FFFF)
    return g


def normal(shape, *, std=1.0, mean=0.0, seed=0, tensor="h", layer=0, device="cpu",
           dtype=torch.float32):
    x = torch.randn(shape, generator=_gen(seed, tensor, layer, device), device=device,
                    dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    if mean != 0.0:
        x.add_(mean)
    return x.to(dtype)


def make_h(wl: Workload, device="cpu"):
    return normal((wl.T, wl.d), seed=wl.seed, tensor="h", device=device, dtype=wl.torch_dtype)


def make_norm_w(wl: Workload, device="cpu"):
    return normal((wl.d,), std=0.1, mean=1.0, seed=wl.seed, tensor="w", device=device,
                  dtype=wl.torch_dtype)


def make_W_U(wl: Workload, device="cpu"):
    return normal((wl.V, wl.d), std=0.02, seed=wl.seed, tensor="W_U", device=device,
                  dtype=wl.torch_dtype)


def make_A(wl: Workload, layer: int, device="cpu"):
    g = _gen(wl.seed, "A", layer, device)
    a = torch.randn((wl.T, wl.d_ff), generator=g, device=device, dtype=torch.float32)
    b = torch.randn((wl.T, wl.d_ff), generator=g, device=device, dtype=torch.float32)
    a = torch.nn.functional.silu(a).mul_(b)
    return a.to(wl.torch_dtype)


def make_gate_up(wl: Workload, layer: int, device="cpu"):
    """(a_l, b_l): the gate and up pre-activations whose SwiGLU product is make_A's A_l."""
    g = _gen(wl.seed, "A", layer, device)
    a = torch.randn((wl.T, wl.d_ff), generator=g, device=device, dtype=torch.float32)
    b = torch.randn((wl.T, wl.d_ff), generator=g, device=device, dtype=torch.float32)
    return a.to(wl.torch_dtype), b.to(wl.torch_dtype)


def make_mlp_in(wl: Workload, layer: int, device="cpu"):
    return normal((wl.T, wl.d), seed=wl.seed, tensor="x", layer=layer, device=device,
                  dtype=wl.torch_dtype)


def make_gate_up_master(wl: Workload, layer: int, device="cpu"):
    return (normal((wl.d_ff, wl.d), std=0.02, seed=wl.seed, tensor="W1", layer=layer,
                   device=device),
            normal((wl.d_ff, wl.d), std=0.02, seed=wl.seed, tensor="W2", layer=layer,
                   device=device))


def make_W_master(wl: Workload, layer: int, device="cpu"):
    return normal((wl.d, wl.d_ff), std=0.02, seed=wl.seed, tensor="W", layer=layer,
                  device=device, dtype=torch.float32)


def make_targets(wl: Workload, device="cpu"):
    g = _gen(wl.seed, "y", 0, device)
    if wl.targets == "uniform":
        return torch.randint(0, wl.V, (wl.T,), generator=g, device=device, dtype=torch.int32)
    if wl.targets == "zipf":
        ranks = torch.arange(1, wl.V + 1, device=device, dtype=torch.float64)
        cdf = torch.cumsum(ranks.pow(-1.1), 0)
        cdf = cdf / cdf[-1]
        u = torch.rand((wl.T,), generator=g, device=device, dtype=torch.float64)
        idx = torch.searchsorted(cdf, u, right=True).clamp_(max=wl.V - 1)
        return idx.to(torch.int32)
    raise ValueError(f"unknown target distribution {wl.targets!r}")


def make_mlp_out(wl: Workload, layer: int, device="cpu"):
    g = _gen(wl.seed, "m", layer, device)
    m = torch.randn((wl.T, wl.d), generator=g, device=device, dtype=torch.float32)
    scale = torch.exp(0.5 * torch.randn((wl.T, 1), generator=g, device=device,
                                        dtype=torch.float32))
    scale[::64] = 0.1
    return (m * scale).to(wl.torch_dtype)


def make_post_norm_w(wl: Workload, layer: int, device="cpu"):
    return normal((wl.d,), std=0.05, mean=0.3, seed=wl.seed, tensor="gp", layer=layer,
                  device=device, dtype=wl.torch_dtype)


def make_pre_norm_in(wl: Workload, layer: int, device="cpu"):
    """Input of a layer's pre-MLP RMSNorm (the residual stream entering the MLP block):
    rows of log-normal scale around RMS 1, every 64th row (offset 32) at RMS ~0.2 so that
    the min-RMS clamp acts on some tokens."""
    g = _gen(wl.seed, "xpre", layer, device)
    x = torch.randn((wl.T, wl.d), generator=g, device=device, dtype=torch.float32)
    scale = torch.exp(0.3 * torch.randn((wl.T, 1), generator=g, device=device,
                                        dtype=torch.float32))
    scale[32::64] = 0.2
    return (x * scale).to(wl.torch_dtype)


def make_pre_norm_w(wl: Workload, layer: int, device="cpu"):
    return normal((wl.d,), std=0.1, mean=1.0, seed=wl.seed, tensor="gq", layer=layer,
                  device=device, dtype=wl.torch_dtype)


def make_noise(n: int, *, seed=0, layer=0, device="cpu"):
    """Standard normal noise used to synthesise 'true' gradients for the diagnostic."""
    return normal((n,), seed=seed, tensor="noise", layer=layer, device=device)


def make_all(wl: Workload, device="cpu", layers=None):
    """Every input of one FPO step as a dict of tensors on ``device``."""
    layers = range(wl.layers) if layers is None else layers
    return {
        "h": make_h(wl, device),
        "w": make_norm_w(wl, device),
        "W_U": make_W_U(wl, device),
        "y": make_targets(wl, device),
        "A": [make_A(wl, l, device) for l in layers],
        "W": [make_W_master(wl, l, device) for l in layers],
    }


def to_numpy_exact(t: torch.Tensor):
    """Host numpy view of a tensor with its exact stored values: fp32/fp64 as is,
    bf16 as uint16 bit patterns (the oracle upcasts them)."""
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view("uint16")
    return t.numpy()
