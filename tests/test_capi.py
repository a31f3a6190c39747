"""The C-ABI library loads without a GPU, exports every symbol include/sara.h declares, and
rejects invalid arguments before touching a device."""
import ctypes
import glob
import os
import re

import pytest

import __graft_entry__

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    __graft_entry__.build()
    import paper_2607_26253_gb300 as pkg
    return pkg.load()


def declared_symbols():
    names = []
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        names += re.findall(r"^SARA_API\s+[\w\s\*]*?\b(sara_\w+)\(", open(h).read(), re.M)
    return names


def test_exports_every_declared_symbol(lib):
    names = declared_symbols()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n


def test_binding_declares_every_symbol():
    import paper_2607_26253_gb300.sara as s
    assert set(declared_symbols()) == set(s.EXPORTED)


def test_invalid_arguments_rejected_without_gpu(lib):
    h = ctypes.c_void_p()
    assert lib.sara_create(None, None, None, ctypes.byref(h)) == -1
    assert b"cfg" in lib.sara_last_error(None)
    assert lib.sara_create(None, None, None, None) == -1
    # shape checks run before any CUDA call
    assert lib.sara_gemm_bf16(None, None, None, 1, 128, 64, None, 0, None) == -1
    assert lib.sara_collect_step(None, None, 0, 8, 2, None, 0, None) == -1
    assert lib.sara_teacher_force(None, 1, 2, None, 1, None, None, 0, None, None, 0) == -1
    assert lib.sara_sample(None, 1, 1, 0, None, None, None, None) == -1
    lib.sara_destroy(None)


def test_tau_is_an_exact_rational():
    from fractions import Fraction
    import paper_2607_26253_gb300 as pkg
    assert pkg.tau_fraction(0.45) == Fraction(9, 20)
    assert pkg.tau_fraction(0.4) == Fraction(2, 5)
    with pytest.raises(ValueError):
        pkg.tau_fraction(1.5)


def test_missing_library_fails_loudly(tmp_path):
    import paper_2607_26253_gb300.sara as s
    with pytest.raises(ImportError):
        s.load(str(tmp_path / "libsara.so"))
