"""The library's kernel-launch counter (fpo_testing_kernel_launches), which bench.py
reads around its timed region: a step launches the same kernels every time, one per
kernel of the path."""
import pytest
import torch

import paper_2608_14563_gb300 as fpo

pytestmark = pytest.mark.gpu


def test_a_step_launches_the_same_kernels_each_time():
    g_ = torch.Generator(device="cuda").manual_seed(2)
    T, d, d_ff, V, L = 700, 256, 512, 2048, 2
    h = torch.randn(T, d, device="cuda", generator=g_).to(torch.bfloat16)
    w = torch.ones(d, device="cuda", dtype=torch.bfloat16)
    W_U = (0.02 * torch.randn(V, d, device="cuda", generator=g_)).to(torch.bfloat16)
    y = torch.randint(0, V, (T,), device="cuda", generator=g_, dtype=torch.int32)
    A = [torch.randn(T, d_ff, device="cuda", generator=g_).to(torch.bfloat16) for _ in range(L)]
    Wm = [torch.zeros(d, d_ff, device="cuda") for _ in range(L)]
    g = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    loss = torch.empty(1, device="cuda")

    def step():
        fpo.error_signal(h, w, W_U, y, g, loss_out=loss)
        fpo.layer_update_grouped(g, A, 1e-3, W_masters=Wm)

    counts = []
    for _ in range(3):
        n0 = fpo.kernel_launches()
        step()
        counts.append(fpo.kernel_launches() - n0)
    torch.cuda.synchronize()
    assert counts[0] == counts[1] == counts[2]
    # RMSNorm forward, logits pass, combine, gather, the two fixup GEMMs with the fixup lse
    # between them, fixup factors, loss mean, projection with the final-norm VJP in its
    # epilogue (+ its split-tail fixup when the last wave is split), grouped update
    assert counts[0] in (11, 12), counts
