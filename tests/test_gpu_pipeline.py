"""The input pipeline of a training loop: each step's inputs are copied from host memory
by fpo_h2d_copy on a copy stream running up to two steps ahead, into three rotating
device sets, while the steps run on the compute stream.  Every step has different inputs,
so a copy that overwrote a set still in use, or a step that read a set before its copy
landed, would give that step another step's results."""
import pytest
import torch

import paper_2608_14563_gb300 as fpo

pytestmark = pytest.mark.gpu


def test_pipelined_host_inputs_match_synchronous_steps():
    T, d, d_ff, V, L, steps, depth = 1000, 512, 1536, 4160, 2, 7, 3
    gen = torch.Generator().manual_seed(21)
    w = (1 + 0.1 * torch.randn(d, generator=gen)).to(torch.bfloat16).cuda()
    W_U = (0.02 * torch.randn(V, d, generator=gen)).to(torch.bfloat16).cuda()
    # per step: h, y and the layers' A_l, in page-locked host memory
    host = [[(torch.randn(T, d, generator=gen)).to(torch.bfloat16).pin_memory(),
             torch.randint(0, V, (T,), generator=gen, dtype=torch.int32).pin_memory()]
            + [torch.randn(T, d_ff, generator=gen).to(torch.bfloat16).pin_memory()
               for _ in range(L)] for _ in range(steps)]

    def run(h, y, A):
        g = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
        loss = torch.empty(1, device="cuda")
        G = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(L)]
        fpo.error_signal(h, w, W_U, y, g, loss_out=loss)
        fpo.layer_update_grouped(g, A, 0.0, G_outs=G)
        return [loss, g] + G

    # reference: each step's inputs copied synchronously, then the step
    ref = []
    for s in range(steps):
        h, y, *A = [t.cuda() for t in host[s]]
        ref.append([t.clone() for t in run(h, y, A)])
    torch.cuda.synchronize()

    sets = [[torch.empty_like(t, device="cuda") for t in host[0]] for _ in range(depth)]
    comp = torch.cuda.current_stream()
    copy = torch.cuda.Stream()
    ready = [torch.cuda.Event() for _ in range(depth)]
    freed = [torch.cuda.Event() for _ in range(depth)]
    for e in freed:
        e.record(comp)

    def prefetch(s):
        b = s % depth
        copy.wait_event(freed[b])
        fpo.h2d_copy(sets[b], host[s], stream=copy)
        ready[b].record(copy)

    out = []
    for s in range(depth - 1):
        prefetch(s)
    for s in range(steps):
        if s + depth - 1 < steps:
            prefetch(s + depth - 1)
        b = s % depth
        comp.wait_event(ready[b])
        h, y, *A = sets[b]
        res = run(h, y, A)
        freed[b].record(comp)
        out.append(res)
    torch.cuda.synchronize()
    for s in range(steps):
        for a, r in zip(out[s], ref[s]):
            assert torch.equal(a, r), f"step {s}"
