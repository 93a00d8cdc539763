"""The C-ABI library loads without a GPU and exports every function that
include/alq.h declares; host-only helpers and argument validation behave as
documented (no kernel is launched here)."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "alq.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*([a-z_0-9]+)\s*\(",
                       text, flags=re.M)
    return sorted(set(n for n in names if n not in ("if", "while")))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_22322_gb300 import build_lib
    path = build_lib.build()
    return C.CDLL(path)


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("al_encode", "al_decode", "uf8_encode", "uf8_decode", "al_adamw_step",
                 "al_adamw_step_multi", "al_adafactor_step", "al_came_step",
                 "al_apollo_step", "al_workspace_size"):
        assert must in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_host_helpers(lib):
    lib.al_num_blocks.restype = C.c_int64
    lib.al_num_blocks.argtypes = [C.c_int64, C.c_int]
    lib.al_state_bytes.restype = C.c_int64
    lib.al_state_bytes.argtypes = [C.c_int64, C.c_int, C.c_int]
    assert lib.al_num_blocks(1000, 256) == 4
    assert lib.al_num_blocks(0, 256) == 0
    assert lib.al_state_bytes(1 << 30, 2048, 8) == (1 << 30) + 8 * (1 << 19)
    assert lib.al_state_bytes(10, 256, 3) == -1


def test_validation_rejects_before_launch(lib):
    """Invalid calls return their status from the host checks; fake pointers
    are never dereferenced because nothing is launched."""
    vp = C.c_void_p
    f = lib.al_encode
    f.restype = C.c_int
    f.argtypes = [vp, C.c_int64, C.c_int, C.c_int, C.c_float, vp, vp, vp]
    A = 0x10000
    assert f(A, 1000, 100, 8, -53.0, A, A, None) == -2        # block not a power of two
    assert f(A, 1000, 256, 12, -53.0, A, A, None) == -2       # bit width
    assert f(A + 4, 1000, 256, 8, -53.0, A, A, None) == -3    # misaligned input
    assert f(None, 1000, 256, 8, -53.0, A, A, None) == -1     # null
    assert f(None, 0, 256, 8, -53.0, None, None, None) == 0   # n == 0: no-op
    assert f(A, -5, 256, 8, -53.0, A, A, None) == -1          # negative size
