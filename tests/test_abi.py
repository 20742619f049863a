"""The C-ABI library builds for sm_103a, loads without a GPU, exports every
symbol include/unif_moe.h declares, and rejects bad arguments before it
touches a device. No kernel runs here."""
import ctypes as C
import math
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "unif_moe.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2608_10392_gb300 import build
    build.build()
    import paper_2608_10392_gb300 as pkg
    return pkg.lib()


def declared_symbols():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"UNIF_MOE_API\s+[\w\s\*]+?\b(unif_moe_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_symbols()
    for n in ("unif_moe_create", "unif_moe_load_weights", "unif_moe_forward", "unif_moe_destroy"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    import paper_2608_10392_gb300 as pkg
    names = declared_symbols()
    assert sorted(pkg.EXPORTS) == names
    for n in names:
        assert hasattr(lib, n), n


def test_only_declared_symbols_are_exported(lib):
    import subprocess
    from paper_2608_10392_gb300 import LIB_PATH
    out = subprocess.run(["nm", "-D", "--defined-only", LIB_PATH], capture_output=True,
                         text=True).stdout
    ours = sorted(l.split()[-1] for l in out.splitlines() if " T unif_moe_" in l)
    assert ours == declared_symbols()


def test_argument_errors_without_gpu(lib):
    import paper_2608_10392_gb300 as pkg
    th = pkg.Thresholds()
    lib.unif_moe_default_thresholds(C.byref(th))
    assert math.isnan(th.tau) and math.isnan(th.alpha_fixed) and th.topk_fixed == 0
    h = C.c_void_p()
    assert lib.unif_moe_create(None, 64, 256, 4, 4, None, 1, 16) == -1
    assert lib.unif_moe_create(C.byref(h), 64, 256, 0, 4, None, 1, 16) == -1   # K = 0
    assert lib.unif_moe_create(C.byref(h), 64, 256, 4, 1, None, 1, 16) == -1   # B = 1
    assert lib.unif_moe_create(C.byref(h), 64, 256, 4, 65, None, 1, 16) == -1  # B > 64
    assert lib.unif_moe_create(C.byref(h), 64, 250, 4, 4, None, 1, 16) == -2   # H % B
    assert lib.unif_moe_create(C.byref(h), 96, 256, 4, 4, None, 1, 16) == -2   # bf16 d % 64
    assert b"d_model" in lib.unif_moe_last_error()
    bad = pkg.Thresholds(math.nan, math.nan, math.nan, 5, 0)
    assert lib.unif_moe_create(C.byref(h), 64, 256, 4, 4, C.byref(bad), 1, 16) == -1
    opts = pkg.Options()
    lib.unif_moe_default_options(C.byref(opts))
    assert opts.features == pkg.FEATURES_DEFAULT and opts.gemm_kernels == 0
    for o in (pkg.Options(16, 0), pkg.Options(3, 4), pkg.Options(3, -1)):  # unknown bit / kind
        assert lib.unif_moe_create_ex(C.byref(h), 64, 256, 4, 4, None, 1, 16, C.byref(o)) == -1
    assert b"options" in lib.unif_moe_last_error()
    assert lib.unif_moe_forward(None, None, None, 4, None, None, None, None) == -1
    assert lib.unif_moe_load_weights(None, None, None, None, None, None) == -1
    assert lib.unif_moe_load_upcycled(None, None, None, None, None, None) == -1
    assert lib.unif_moe_sublayer_forward(None, None, None, 4, None, None, None, None, None,
                                         1e-5, 1, None) == -1
    assert lib.unif_moe_backward(None, None, None, 4, None, None, None, None, None, None, 0.0,
                                 None, None) == -1
    assert lib.unif_moe_value_alignment(None, 0.98, None, None) == -1
    assert lib.unif_moe_functional_demand(None, None, 4, None, 0.98, 0.05, None, None, None,
                                          None) == -1
    assert lib.unif_moe_sync_status(None, None) == -1
    assert lib.unif_moe_forward_host(None, None, None, 4, None, None, None, None) == -1
    assert lib.unif_moe_forward_host_async(None, None, None, 4, None, None, None, None) == -1
    assert lib.unif_moe_forward_host_wait(None) == -1
    assert lib.unif_moe_max_rows(None) == -1
    assert lib.unif_moe_kernels_per_forward(None) == -1
    lib.unif_moe_destroy(None)


def test_missing_library_fails_loudly(tmp_path, monkeypatch):
    import paper_2608_10392_gb300 as pkg
    monkeypatch.setattr(pkg, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        pkg.lib(str(tmp_path / "absent.so"))


def test_product_code_never_touches_the_oracle():
    pkg_dir = os.path.join(ROOT, "paper_2608_10392_gb300")
    for dirpath, _, files in os.walk(pkg_dir):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "liboracle" not in text, f
                assert "from oracle" not in text, f


def test_library_reads_no_environment():
    """Behaviour is set through the ABI only: no getenv in the library."""
    csrc = os.path.join(ROOT, "paper_2608_10392_gb300", "csrc")
    for f in os.listdir(csrc):
        if f.endswith((".cu", ".cuh", ".h")):
            assert "getenv" not in open(os.path.join(csrc, f)).read(), f
