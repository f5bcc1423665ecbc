"""The C-ABI library loads and exports every symbol the headers declare (CPU;
no compute call is made without a GPU)."""
import ctypes
import os

import pytest

from helpers import ROOT, header_symbols


def _lib_path():
    return os.path.join(ROOT, "paper_2608_10139_gb300", "libaiq.so")


@pytest.fixture(scope="module")
def built():
    from paper_2608_10139_gb300 import build
    return build.build()


def test_headers_declare_entry_points():
    syms = header_symbols()
    for s in ("aiq_init", "aiq_load_table", "aiq_load_model", "aiq_run_select", "aiq_run_join_select",
              "aiq_result", "aiq_op_gemm", "aiq_op_attention"):
        assert s in syms


def test_library_exports_every_declared_symbol(built):
    lib = ctypes.CDLL(built)
    missing = [s for s in header_symbols() if not hasattr(lib, s)]
    assert not missing, missing


def test_binding_signatures_cover_headers(built):
    from paper_2608_10139_gb300 import aiq
    assert set(header_symbols()) <= set(aiq._SIGS), set(header_symbols()) - set(aiq._SIGS)
    aiq.load_library()


def test_init_without_gpu_fails_cleanly(built):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2608_10139_gb300 import aiq
    with pytest.raises(aiq.AiqError):
        aiq.Context(0)
