import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TESTS = os.path.dirname(os.path.abspath(__file__))
for p in (ROOT, TESTS):
    if p not in sys.path:
        sys.path.insert(0, p)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA device (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running (full-size workloads)")


def _ensure_built():
    """Compile libfpo.so in-tree if it is missing (nvcc cross-compiles without a GPU)."""
    import importlib.util
    path = os.path.join(ROOT, "paper_2608_14563_gb300", "build.py")
    spec = importlib.util.spec_from_file_location("_fpo_build", path)
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    if not os.path.exists(b.LIB):
        b.build()


_ensure_built()


@pytest.fixture(scope="session")
def fpo():
    """The CUDA library through its Python binding; skips when no GPU is present.
    FPO_TEST_GEMM_VARIANT=0|1|2 runs the suite on the single-CTA GEMM, the CTA-pair
    GEMM with 256 x 256 tiles only, or the CTA pair with the 256 x 512 projection (the
    library default)."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_14563_gb300 as lib
    v = os.environ.get("FPO_TEST_GEMM_VARIANT")
    if v is not None:
        lib.set_gemm_variant(int(v))
    return lib
