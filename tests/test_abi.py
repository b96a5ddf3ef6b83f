"""The C-ABI library builds, loads and exports every entry point include/zoact.h declares.

CPU only: no compute call is made (there may be no GPU).
"""
import ctypes
import os
import re

from paper_2607_01125_gb300 import build as zbuild
from paper_2607_01125_gb300 import _lib

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "zoact.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(zoact_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_four_calls_of_the_method():
    names = _declared()
    for n in ["zoact_basis_init", "zoact_pair_forward", "zoact_loss_pair", "zoact_adam_step"]:
        assert n in names


def test_library_exports_every_declared_symbol():
    path = zbuild.build()
    lib = ctypes.CDLL(path)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing
    assert sorted(_lib.EXPORTS) == _declared()


def test_status_strings_without_gpu():
    zbuild.build()
    assert _lib.status_string(0) == "ok"
    assert "timed out" in _lib.status_string(_lib.ZOACT_ERR_TIMEOUT)
    assert _lib.status_string(12345) == "unknown status"


def test_layer_struct_matches_c_layout():
    # zoact_layer: 4 int32, then 4 pointers, then uint32 (+ padding) -> 56 bytes on LP64
    assert ctypes.sizeof(_lib.zoact_layer) == 56
    assert _lib.zoact_layer.W.offset == 16 and _lib.zoact_layer.layer_id.offset == 48
    assert ctypes.sizeof(_lib.zoact_coeff_block) == 24
