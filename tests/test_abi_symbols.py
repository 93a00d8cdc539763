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
    lib.al_meta_count.restype = C.c_int64
    lib.al_meta_count.argtypes = [C.c_int64, C.c_int]
    assert lib.al_meta_count(1000, 256) == 8
    assert lib.al_meta_count(0, 256) == 0
    assert lib.al_meta_count(-1, 256) == -1
    lib.al_last_cuda_error.restype = C.c_char_p
    lib.alq_last_cuda_error.restype = C.c_char_p
    assert lib.al_last_cuda_error() == lib.alq_last_cuda_error() == b""


def test_status_aliases_match():
    """The AL_ status names are the ALQ_ codes."""
    text = open(HEADER).read()
    codes = dict(re.findall(r"#define (ALQ_\w+) \(?(-?\d+)\)?", text))
    aliases = dict(re.findall(r"#define (AL_\w+) (ALQ_\w+)", text))
    assert set(aliases) == {"AL_OK", "AL_ERR_INVALID_ARG", "AL_ERR_UNSUPPORTED", "AL_ERR_ALIGN",
                            "AL_ERR_WORKSPACE", "AL_ERR_CUDA"}
    for a, target in aliases.items():
        assert a[3:] == target[4:] and target in codes


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


def test_grouped_factored_plan_host_logic(lib):
    """al_factored_plan on the host: per-pass tile counts, workspace sizes
    and the argument checks (the plan only records fake pointers)."""
    from paper_2608_22322_gb300 import binding as Bn
    lib = Bn.lib  # the binding's handle carries the argument types
    A = 0x100000

    def mat(rows, cols, came, mom):
        ptrs = [A] * 8 if came else [A] * 4 + [None] * 4
        return Bn.FactoredMatrix(A, A, rows, cols, *ptrs, A if mom else None, A if mom else None)

    shapes = [(300, 772), (64, 512), (4096, 4096)]
    arr = (Bn.FactoredMatrix * 3)(*[mat(r, c, True, True) for r, c in shapes])
    ws = C.c_size_t(0)
    assert lib.al_factored_workspace_multi(arr, 3, C.byref(ws)) == 0
    per = []
    for r, c in shapes:
        b = C.c_size_t(0)
        assert lib.al_workspace_size(2, r, c, 0, C.byref(b)) == 0
        per.append(b.value)
    assert ws.value == sum(per)
    nb = C.c_size_t(0)
    assert lib.al_factored_plan_bytes(arr, 3, C.byref(nb)) == 0
    host = (C.c_uint8 * nb.value)()
    info = Bn.FactoredInfo()
    args = lambda op, a, w: (op, a, 3, 16, 128, 16, 128, 256, C.c_void_p(A), w, host,
                             nb.value, C.byref(info))
    assert lib.al_factored_plan(*args(2, arr, ws.value)) == 0
    tiles = lambda n, t: -(-n // t)
    assert info.nmat == 3 and info.op == 2 and info.has_momentum == 1
    assert info.total_params == sum(r * c for r, c in shapes)
    assert info.sumsq_tiles == sum(tiles(c, 256) * tiles(r, 64) for r, c in shapes)
    assert info.factor_tiles == sum(tiles(r, 128) + tiles(c, 128) for r, c in shapes)
    assert info.factor2_tiles == info.factor_tiles
    assert info.scale_tiles == sum(tiles(r + c, 256) for r, c in shapes)
    assert info.tiles == sum(tiles(r * c, 4096) for r, c in shapes)
    assert info.rms_chunks == sum(tiles(tiles(r * c, 4096), 8) for r, c in shapes)
    assert lib.al_factored_plan(*args(2, arr, ws.value - 1)) == -4   # workspace too small
    assert lib.al_factored_plan(*args(3, arr, ws.value)) == -1       # not a factored op
    # momentum in some matrices only; CAME without momentum; no confidence
    mixed = (Bn.FactoredMatrix * 3)(mat(300, 772, True, True), mat(64, 512, True, False),
                                   mat(8, 8, True, True))
    assert lib.al_factored_plan(*args(2, mixed, ws.value)) == -1
    nom = (Bn.FactoredMatrix * 3)(*[mat(r, c, True, False) for r, c in shapes])
    assert lib.al_factored_plan(*args(2, nom, ws.value)) == -1
    ada = (Bn.FactoredMatrix * 3)(*[mat(r, c, False, False) for r, c in shapes])
    assert lib.al_factored_plan(*args(1, ada, ws.value)) == 0
    assert info.has_momentum == 0 and info.factor2_tiles == 0
    assert lib.al_factored_plan(*args(2, ada, ws.value)) == -1       # CAME needs confidence
    bad = (Bn.FactoredMatrix * 3)(mat(300, 770, True, True), *[mat(r, c, True, True)
                                                               for r, c in shapes[1:]])
    assert lib.al_factored_plan(*args(2, bad, ws.value)) == -2       # cols % 4
