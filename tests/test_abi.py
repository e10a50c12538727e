"""The C-ABI library loads, exports every entry point include/fpo.h declares, and
rejects bad arguments on the host before touching a device (no GPU needed)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fpo.h")
TESTING_HEADER = os.path.join(ROOT, "include", "fpo_testing.h")
LIB = os.path.join(ROOT, "paper_2608_14563_gb300", "libfpo.so")


def declared_functions(header=HEADER):
    text = open(header).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fpo_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("fpo_error_signal", "fpo_layer_update", "fpo_layer_update_grouped",
                     "fpo_cosine", "fpo_get_device_status", "fpo_status_string",
                     "fpo_error_signal_workspace", "fpo_layer_update_workspace",
                     "fpo_cosine_workspace"):
        assert required in names


def test_library_exports_every_declared_symbol():
    out = subprocess.run(["nm", "-D", "--defined-only", LIB], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\sT\s+(fpo_\w+)$", out, flags=re.M))
    names = declared_functions() + declared_functions(TESTING_HEADER)
    assert "fpo_testing_direct_fixup_rows" in names
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    lib = ctypes.CDLL(LIB)
    for n in names:
        assert hasattr(lib, n)


def test_binding_loads_and_reports_version():
    import paper_2608_14563_gb300 as fpo
    assert fpo.abi_version() == 2
    assert fpo.status_string(0) == "FPO_OK"
    assert "TARGET_RANGE" in fpo.status_string(8)
    assert fpo.status_string(12345) == "unknown fpo status"


def test_binding_constants_match_the_header():
    """The binding's copies of the header's constants and enums equal the header's."""
    import paper_2608_14563_gb300 as fpo
    with open(os.path.join(ROOT, "include", "fpo.h")) as f:
        hdr = f.read()
    defines = dict(re.findall(r"#define (FPO_\w+) (\d+)", hdr))
    assert int(defines["FPO_ABI_VERSION"]) == fpo.ABI_VERSION == fpo.abi_version()
    assert int(defines["FPO_MAX_GROUPED_LAYERS"]) == fpo.MAX_GROUPED_LAYERS
    assert int(defines["FPO_MAX_COPY_BUFFERS"]) == fpo.MAX_COPY_BUFFERS
    assert int(defines["FPO_STAGE_EVENTS"]) == fpo.STAGE_EVENTS
    assert int(defines["FPO_AUTO_T_CHUNK"]) == fpo.AUTO_T_CHUNK
    enums = dict((k, int(v)) for k, v in re.findall(r"(FPO_\w+) = (\d+)", hdr))
    for name, value in [("FPO_F32", fpo.F32), ("FPO_BF16", fpo.BF16), ("FPO_OK", fpo.OK),
                        ("FPO_ES_AUTO", fpo.ES_AUTO), ("FPO_ES_RECOMPUTE", fpo.ES_RECOMPUTE),
                        ("FPO_ES_STORED_LOGITS", fpo.ES_STORED_LOGITS),
                        ("FPO_ES_DIRECT", fpo.ES_DIRECT), ("FPO_OPT_SGD", fpo.OPT_SGD),
                        ("FPO_OPT_SGD_MOMENTUM", fpo.OPT_SGD_MOMENTUM),
                        ("FPO_OPT_ADAMW", fpo.OPT_ADAMW), ("FPO_CLIP_NONE", fpo.CLIP_NONE),
                        ("FPO_CLIP_STEP", fpo.CLIP_STEP),
                        ("FPO_CLIP_GRADIENT", fpo.CLIP_GRADIENT)]:
        assert enums[name] == value, name


class _Lib:
    def __init__(self):
        import paper_2608_14563_gb300 as fpo
        self.fpo = fpo
        self.lib = fpo._lib


@pytest.fixture(scope="module")
def L():
    return _Lib()


def test_error_signal_workspace_query(L):
    fpo = L.fpo
    small = fpo.error_signal_desc(128, 64, 512, fpo.F32)
    assert fpo.error_signal_workspace(small) > 0
    # per token of the chunk: recompute holds a bf16 row of E; stored logits add an fp32
    # row of logits; direct (the bf16 default) holds a bf16 row of P, one fixup-list entry
    # and a bf16 row of d for the gathered rows of the fixup
    V, d = 151936, 4096
    for algo, per in ((fpo.ES_RECOMPUTE, 2 * V), (fpo.ES_STORED_LOGITS, 6 * V),
                      (fpo.ES_DIRECT, 2 * V + 4 + 2 * d), (fpo.ES_AUTO, 2 * V + 4 + 2 * d)):
        chunked = fpo.error_signal_desc(4096, 4096, V, fpo.BF16, t_chunk=1024, algo=algo)
        full = fpo.error_signal_desc(4096, 4096, V, fpo.BF16, algo=algo)
        diff = fpo.error_signal_workspace(full) - fpo.error_signal_workspace(chunked)
        assert abs(diff - 3072 * per) < 1024
    # fp32 has no direct form: AUTO and DIRECT take the stored-logits layout
    f32 = [fpo.error_signal_workspace(fpo.error_signal_desc(512, 64, 1000, fpo.F32, algo=a))
           for a in (fpo.ES_AUTO, fpo.ES_DIRECT, fpo.ES_STORED_LOGITS)]
    assert f32[0] == f32[1] == f32[2]
    assert fpo.error_signal_workspace(fpo.error_signal_desc(64, 64, 256, fpo.BF16, algo=7)) == 0
    bad = fpo.error_signal_desc(16, 12, 512, fpo.BF16)  # d not a multiple of 8
    assert fpo.error_signal_workspace(bad) == 0
    assert L.lib.fpo_error_signal_workspace(None) == 0


def test_error_signal_host_validation(L):
    fpo = L.fpo
    lib = L.lib
    desc = fpo.error_signal_desc(16, 64, 256, fpo.BF16)
    ws = fpo.error_signal_workspace(desc)
    fake = ctypes.c_void_p(1 << 20)   # never dereferenced: validation fails first
    mis = ctypes.c_void_p((1 << 20) + 8)
    call = lambda d, h=fake, ws_ptr=fake, ws_n=ws, g=fake: lib.fpo_error_signal(
        ctypes.byref(d) if d is not None else None, h, fake, fake, fake, g, None, None, ws_ptr, ws_n,
        None)
    assert call(None) == 1                                            # FPO_ERR_NULL
    assert call(fpo.error_signal_desc(16, 64, 256, 7)) == 3           # FPO_ERR_DTYPE
    assert call(fpo.error_signal_desc(-1, 64, 256, fpo.BF16)) == 2    # FPO_ERR_SHAPE
    assert call(fpo.error_signal_desc(16, 60, 256, fpo.BF16)) == 2    # d % 8
    assert call(fpo.error_signal_desc(16, 64, 250, fpo.BF16)) == 2    # V % 8
    assert call(desc, h=None) == 1
    assert call(desc, h=mis) == 4                                     # FPO_ERR_ALIGN
    assert call(desc, ws_ptr=None) == 5                               # FPO_ERR_WORKSPACE
    assert call(desc, ws_n=ws - 1) == 5
    assert call(desc, g=mis) == 4


def test_layer_update_and_cosine_host_validation(L):
    lib = L.lib
    fake = ctypes.c_void_p(1 << 20)
    mis = ctypes.c_void_p((1 << 20) + 4)
    ws = L.fpo.layer_update_workspace()
    assert lib.fpo_layer_update(16, 64, 128, 9, fake, fake, 0.1, fake, None, None, fake, ws, None) == 3
    assert lib.fpo_layer_update(16, 64, 100, 1, fake, fake, 0.1, fake, None, None, fake, ws, None) == 2
    assert lib.fpo_layer_update(16, 64, 128, 1, fake, fake, 0.1, None, None, None, fake, ws, None) == 1
    assert lib.fpo_layer_update(16, 64, 128, 1, fake, fake, 0.1, None, fake, fake, fake, ws, None) == 1
    assert lib.fpo_layer_update(16, 64, 128, 1, fake, mis, 0.1, fake, None, None, fake, ws, None) == 4
    assert lib.fpo_layer_update(16, 64, 128, 1, fake, fake, 0.1, fake, None, None, None, ws, None) == 5
    assert lib.fpo_layer_update(16, 64, 128, 1, fake, fake, 0.1, fake, None, None, fake, 8, None) == 5
    arr = (ctypes.c_void_p * 1)(fake.value)
    assert lib.fpo_layer_update_grouped(0, 16, 64, 128, 1, fake, arr, 0.1, arr, None, None, fake,
                                        ws, None) == 2
    assert lib.fpo_layer_update_grouped(65, 16, 64, 128, 1, fake, arr, 0.1, arr, None, None, fake,
                                        ws, None) == 2
    assert lib.fpo_cosine(-1, 1, fake, fake, fake, fake, 1 << 20, None) == 2
    assert lib.fpo_cosine(10, 5, fake, fake, fake, fake, 1 << 20, None) == 3
    assert lib.fpo_cosine(10, 1, None, fake, fake, fake, 1 << 20, None) == 1
    assert lib.fpo_cosine(10, 1, mis, fake, fake, fake, 1 << 20, None) == 4
    assert lib.fpo_get_device_status(None, None) == 5


def test_h2d_copy_host_validation(L):
    lib = L.lib
    vp, sz = ctypes.c_void_p, ctypes.c_size_t
    fake, mis = 1 << 20, (1 << 20) + 8
    one = lambda *x: (vp * len(x))(*x)   # noqa: E731
    assert lib.fpo_h2d_copy(-1, None, None, None, None) == 2
    assert lib.fpo_h2d_copy(65, None, None, None, None) == 2
    assert lib.fpo_h2d_copy(0, None, None, None, None) == 0
    assert lib.fpo_h2d_copy(1, None, one(fake), (sz * 1)(16), None) == 1
    assert lib.fpo_h2d_copy(1, one(fake), one(None), (sz * 1)(16), None) == 1
    assert lib.fpo_h2d_copy(1, one(fake), one(mis), (sz * 1)(16), None) == 4
    assert lib.fpo_h2d_copy(1, one(mis), one(fake), (sz * 1)(16), None) == 4


def test_rejected_calls_launch_no_kernel(L):
    """Host-side argument errors return before anything is enqueued: the library's
    launch counter does not move."""
    lib = L.lib
    n0 = L.fpo.kernel_launches()
    fake = ctypes.c_void_p(1 << 20)
    assert lib.fpo_cosine(10, 1, None, fake, fake, fake, 1 << 20, None) == 1
    assert lib.fpo_h2d_copy(-1, None, None, None, None) == 2
    assert L.fpo.kernel_launches() == n0
