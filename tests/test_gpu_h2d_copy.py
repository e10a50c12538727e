"""fpo_h2d_copy: host-to-device copies by SM loads of mapped page-locked memory.

Byte copies are checked bit for bit against the source, with guard bytes after every
destination range, for ragged sizes (tails under 16 bytes), interior pointers, 64 buffers
in one launch, registered (not allocated) host memory, and a copy that runs while a
tensor-core GEMM occupies every SM on another stream.  Host-side errors: a pageable or
misaligned source, too many buffers."""
import ctypes

import numpy as np
import pytest
import torch

import paper_2608_14563_gb300 as fpo

pytestmark = pytest.mark.gpu

GUARD = 0xAB


def pinned_bytes(n, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(0, 256, (n,), dtype=torch.uint8, generator=g).pin_memory()


def guarded_dst(n, dev="cuda"):
    buf = torch.full((n + 64,), GUARD, dtype=torch.uint8, device=dev)
    return buf, buf[:n]


def check(buf, src):
    n = src.numel()
    out = buf.cpu()
    assert torch.equal(out[:n], src)
    assert bool((out[n:] == GUARD).all())


@pytest.mark.parametrize("n", [1, 15, 16, 17, 31, 4099, 1 << 20, 37_000_001])
def test_ragged_sizes(n):
    src = pinned_bytes(n, n)
    buf, dst = guarded_dst(n)
    fpo.h2d_copy([dst], [src])
    torch.cuda.synchronize()
    check(buf, src)


def test_empty_pairs_are_skipped():
    src = pinned_bytes(1000, 1)
    buf, dst = guarded_dst(1000)
    empty_h = torch.empty(0, dtype=torch.uint8).pin_memory()
    empty_d = torch.empty(0, dtype=torch.uint8, device="cuda")
    fpo.h2d_copy([empty_d, dst, empty_d], [empty_h, src, empty_h])
    fpo.h2d_copy([], [])
    torch.cuda.synchronize()
    check(buf, src)


def test_interior_pointers():
    base = pinned_bytes((1 << 20) + 4096, 7)
    src = base[48:48 + 300_007]           # 16-byte aligned offset inside the allocation
    buf, dst = guarded_dst(300_007)
    fpo.h2d_copy([dst], [src])
    torch.cuda.synchronize()
    check(buf, src)


def test_many_buffers_one_launch_and_beyond():
    rng = np.random.default_rng(3)
    sizes = [int(s) for s in rng.integers(1, 200_000, size=fpo.MAX_COPY_BUFFERS + 9)]
    srcs = [pinned_bytes(n, 100 + i) for i, n in enumerate(sizes)]
    pairs = [guarded_dst(n) for n in sizes]
    fpo.h2d_copy([d for _, d in pairs], srcs)   # two launches: 64 + 9
    torch.cuda.synchronize()
    for (buf, _), src in zip(pairs, srcs):
        check(buf, src)


def test_typed_tensors():
    g = torch.Generator().manual_seed(5)
    h = torch.randn(1000, 4096, generator=g).to(torch.bfloat16).pin_memory()
    y = torch.randint(0, 100352, (1000,), dtype=torch.int32, generator=g).pin_memory()
    dh = torch.empty(1000, 4096, dtype=torch.bfloat16, device="cuda")
    dy = torch.empty(1000, dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    fpo.h2d_copy([dh, dy], [h, y], stream=s)
    s.synchronize()
    assert torch.equal(dh.cpu(), h) and torch.equal(dy.cpu(), y)


def test_registered_host_memory():
    n = 5_000_003
    arr = np.random.default_rng(9).integers(0, 256, size=n + 64, dtype=np.uint8)
    off = (-arr.ctypes.data) % 16                   # a 16-byte aligned start inside arr
    view = arr[off:off + n]
    cr = torch.cuda.cudart()
    assert int(cr.cudaHostRegister(view.ctypes.data, n, 2)) == 0   # cudaHostRegisterMapped
    try:
        src = torch.from_numpy(view)
        buf, dst = guarded_dst(n)
        fpo.h2d_copy([dst], [src])
        torch.cuda.synchronize()
        check(buf, src)
    finally:
        cr.cudaHostUnregister(view.ctypes.data)


def test_copy_beside_a_gemm():
    """The copy and a persistent tensor-core GEMM run on two streams at once; both
    results match the same work done one after the other."""
    g = torch.Generator().manual_seed(11)
    T, d, d_ff, L = 4096, 1024, 2816, 4
    gt = torch.randn(T, d, generator=g).to(torch.bfloat16).cuda()
    As = [torch.randn(T, d_ff, generator=g).to(torch.bfloat16).cuda() for _ in range(L)]
    G_ref = [torch.empty(d, d_ff, dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    G = [torch.empty_like(x) for x in G_ref]
    fpo.layer_update_grouped(gt, As, 0.0, G_outs=G_ref)
    torch.cuda.synchronize()
    src = pinned_bytes(256 << 20, 12)
    buf, dst = guarded_dst(src.numel())
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    for _ in range(3):
        fpo.layer_update_grouped(gt, As, 0.0, G_outs=G, stream=sa)
    fpo.h2d_copy([dst], [src], stream=sb)
    torch.cuda.synchronize()
    check(buf, src)
    for a, b in zip(G, G_ref):
        assert torch.equal(a, b)


def test_host_errors():
    dst = torch.empty(4096, dtype=torch.uint8, device="cuda")
    pageable = torch.zeros(4096, dtype=torch.uint8)
    with pytest.raises(fpo.FpoError) as e:
        fpo.h2d_copy([dst], [pageable])
    assert e.value.code == 10   # FPO_ERR_ARG
    base = pinned_bytes(8192, 2)
    with pytest.raises(fpo.FpoError) as e:
        fpo.h2d_copy([dst], [base[8:8 + 4096]])
    assert e.value.code == 4    # FPO_ERR_ALIGN
    with pytest.raises(ValueError):
        fpo.h2d_copy([dst], [base[:100]])
    lib = fpo._lib
    vp, sz = ctypes.c_void_p, ctypes.c_size_t
    arr = (vp * 1)(dst.data_ptr())
    assert lib.fpo_h2d_copy(fpo.MAX_COPY_BUFFERS + 1, arr, arr, (sz * 1)(16), None) == 2
    # the context is still usable after the rejected calls
    src = pinned_bytes(4096, 4)
    fpo.h2d_copy([dst], [src])
    torch.cuda.synchronize()
    assert torch.equal(dst.cpu(), src)
