"""Python view of the C oracle (ctypes over oracle/_build/libalq_oracle.so).

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and the benchmark's
CPU-baseline leg may import this module. The product path (the package and
its CUDA library) never imports it, and it never imports the package.

Every function takes and returns numpy arrays. Functions ending in ``_step``
work on quantized states in place, exactly like the C-ABI entry points of the
CUDA library, so a test can run both on copies of the same inputs.
"""
from __future__ import annotations

import ctypes as C
import numpy as np

from . import build as _build

_lib = C.CDLL(_build.build())
_lib_plain = _lib
_lib_threaded = None

_f32p = np.ctypeslib.ndpointer(np.float32, flags="C_CONTIGUOUS")
_i8p = np.ctypeslib.ndpointer(np.int8, flags="C_CONTIGUOUS")
_u16p = np.ctypeslib.ndpointer(np.uint16, flags="C_CONTIGUOUS")
_vp = C.c_void_p
_i64 = C.c_int64
_int = C.c_int
_flt = C.c_float


class AdamWHP(C.Structure):
    _fields_ = [(k, C.c_float) for k in
                ("lr", "beta1", "beta2", "eps", "weight_decay", "log_floor")]


class AdafactorHP(C.Structure):
    _fields_ = [(k, C.c_float) for k in
                ("lr", "eps1", "clip_d", "decay_rate", "beta1", "weight_decay",
                 "log_floor")]


class CameHP(C.Structure):
    _fields_ = [(k, C.c_float) for k in
                ("lr", "beta1", "beta2", "beta3", "eps1", "eps2", "clip_d",
                 "weight_decay", "log_floor_v", "log_floor_c")]


class ApolloHP(C.Structure):
    _fields_ = ([(k, C.c_float) for k in
                 ("lr", "beta1", "beta2", "eps", "alpha", "weight_decay",
                  "norm_growth_gamma", "log_floor")] + [("rank", C.c_int32)])


_SIGS = []


def _sig(name, res, *args):
    _SIGS.append((name, res, list(args)))
    fn = getattr(_lib, name)
    fn.restype = res
    fn.argtypes = list(args)
    return fn


def use_threads(on: bool = True) -> int:
    """Switch every function of this module to the OpenMP build of the same
    source (all host cores; the same results bit for bit) or back to the
    plain single-threaded build. Returns the number of threads the next
    calls use (1 when the compiler has no OpenMP)."""
    global _lib, _lib_threaded
    if not on:
        _lib = _lib_plain
        return 1
    if _lib_threaded is None:
        path = _build.build_threaded()
        if path is None:
            return 1
        lib = C.CDLL(path)
        for name, res, args in _SIGS:
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib_threaded = lib
    _lib = _lib_threaded
    return threads()


def threads() -> int:
    """Threads the current build runs its parallel loops on (OpenMP's
    default: OMP_NUM_THREADS, else the cores this process may run on)."""
    import os
    if _lib is _lib_plain:
        return 1
    if os.environ.get("OMP_NUM_THREADS", "").isdigit():
        return int(os.environ["OMP_NUM_THREADS"])
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


_sig("ora_al_block_meta", _int, _f32p, _i64, _flt, C.POINTER(_flt), C.POINTER(_flt))
_sig("ora_al_quantize", C.c_uint32, _flt, _flt, _flt, _int)
_sig("ora_al_dequantize", _flt, C.c_uint32, _flt, _flt, _int)
_sig("ora_al_encode", None, _f32p, _i64, _int, _int, _flt, _vp, _f32p)
_sig("ora_al_decode", None, _vp, _f32p, _i64, _int, _int, _f32p)
_sig("ora_al_state_bytes", _i64, _i64, _int, _int)
_sig("ora_uf8_encode", None, _f32p, _i64, _int, _i8p, _f32p)
_sig("ora_uf8_decode", None, _i8p, _f32p, _i64, _int, _f32p)
_sig("ora_adamw_update_fp32", None, _f32p, _f32p, _f32p, _f32p, _i64,
     C.POINTER(AdamWHP), _i64)
_sig("ora_adamw_step", None, _f32p, _f32p, _vp, _vp, _vp, _vp, _i64,
     _int, _int, _int, C.POINTER(AdamWHP), _i64, _vp, _vp)
_sig("ora_adafactor_update_fp32", None, _f32p, _f32p, _i64, _i64, _f32p, _f32p,
     _vp, C.POINTER(AdafactorHP), _i64)
_sig("ora_adafactor_step", None, _f32p, _f32p, _i64, _i64, _vp, _f32p, _vp,
     _f32p, _int, _int, _vp, _vp, _int, C.POINTER(AdafactorHP), _i64, _vp, _vp,
     _vp)
_sig("ora_came_update_fp32", None, _f32p, _f32p, _i64, _i64, _f32p, _f32p,
     _f32p, _f32p, _f32p, C.POINTER(CameHP), _i64)
_sig("ora_came_step", None, _f32p, _f32p, _i64, _i64, _vp, _f32p, _vp, _f32p,
     _int, _int, _vp, _f32p, _vp, _f32p, _int, _int, _i8p, _f32p, _int,
     C.POINTER(CameHP), _i64, _vp)
_sig("ora_apollo_project", None, _f32p, _i64, _i64, _u16p, _int, _f32p)
_sig("ora_apollo_update_fp32", None, _f32p, _f32p, _i64, _i64, _u16p, _f32p,
     _f32p, C.POINTER(_flt), C.POINTER(ApolloHP), _i64, _vp)
_sig("ora_apollo_step", None, _f32p, _f32p, _i64, _i64, _u16p, _i8p, _f32p,
     _int, _vp, _f32p, _int, _int, C.POINTER(_flt), C.POINTER(ApolloHP), _i64,
     _vp, _vp, _vp)
_sig("ora_apollo_step_given_R", None, _f32p, _f32p, _i64, _i64, _f32p, _i8p, _f32p, _int,
     _vp, _f32p, _int, _int, C.POINTER(_flt), C.POINTER(ApolloHP), _i64, _vp)
_sig("ora_f32_to_bf16", C.c_uint16, _flt)
_sig("ora_bf16_to_f32", _flt, C.c_uint16)
_sig("ora_update_error", C.c_double, _f32p, _f32p, _i64, C.c_double)


# ------------------------------------------------------------------ helpers --
def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def code_dtype(bits: int):
    """Storage type of a state of this role precision (32: unquantized fp32)."""
    return np.uint8 if bits <= 8 else np.uint16 if bits <= 16 else np.float32


def num_blocks(n: int, block: int) -> int:
    return (n + block - 1) // block


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _hp(cls, d):
    return cls(**{k: d[k] for k, _ in cls._fields_})


# --------------------------------------------------------------------- AL ----
def al_block_meta(x, log_floor: float):
    """(l_min, Delta, any_positive) of one block (Eq. (3) + Sec. 4.1)."""
    x = _f32(x)
    lmin, delta = _flt(), _flt()
    anyp = _lib.ora_al_block_meta(x, x.size, log_floor, C.byref(lmin), C.byref(delta))
    return np.float32(lmin.value), np.float32(delta.value), bool(anyp)


def al_quantize(x: float, lmin: float, delta: float, bits: int) -> int:
    return int(_lib.ora_al_quantize(float(x), float(lmin), float(delta), bits))


def al_dequantize(q: int, lmin: float, delta: float, bits: int) -> np.float32:
    return np.float32(_lib.ora_al_dequantize(int(q), float(lmin), float(delta), bits))


def al_encode(x, block: int, bits: int, log_floor: float):
    """Return (codes, meta) for a flat fp32 array (Eq. (3)-(4))."""
    x = _f32(x).ravel()
    codes = np.zeros(x.size, dtype=code_dtype(bits))
    meta = np.zeros(2 * num_blocks(x.size, block), dtype=np.float32)
    _lib.ora_al_encode(x, x.size, block, bits, log_floor, _ptr(codes), meta)
    return codes, meta


def al_decode(codes, meta, block: int, bits: int):
    codes = np.ascontiguousarray(codes, dtype=code_dtype(bits))
    out = np.zeros(codes.size, dtype=np.float32)
    _lib.ora_al_decode(_ptr(codes), _f32(meta), codes.size, block, bits, out)
    return out


def al_state_bytes(n: int, block: int, bits: int) -> int:
    return int(_lib.ora_al_state_bytes(n, block, bits))


# -------------------------------------------------------------------- UF8 ----
def uf8_encode(m, block: int):
    m = _f32(m).ravel()
    codes = np.zeros(m.size, dtype=np.int8)
    absmax = np.zeros(num_blocks(m.size, block), dtype=np.float32)
    _lib.ora_uf8_encode(m, m.size, block, codes, absmax)
    return codes, absmax


def uf8_decode(codes, absmax, block: int):
    codes = np.ascontiguousarray(codes, dtype=np.int8)
    out = np.zeros(codes.size, dtype=np.float32)
    _lib.ora_uf8_decode(codes, _f32(absmax), codes.size, block, out)
    return out


# ------------------------------------------------------------------ AdamW ----
def adamw_update_fp32(p, g, m, v, hp: dict, t: int):
    """fp32-state AdamW; p, m, v are updated in place (float32 arrays)."""
    _lib.ora_adamw_update_fp32(p, _f32(g), m, v, p.size, C.byref(_hp(AdamWHP, hp)), t)


def adamw_step(p, g, m_codes, m_absmax, v_codes, v_meta, m_block, v_block,
               v_bits, hp: dict, t: int, want_fresh: bool = False):
    """Quantized AdamW step in place; optionally return the fresh (m, v).
    v_bits 32: the unquantized reference (m_codes and v_codes are fp32 m and
    v; m_absmax and v_meta are unused)."""
    mf = np.zeros(p.size, np.float32) if want_fresh else None
    vf = np.zeros(p.size, np.float32) if want_fresh else None
    _lib.ora_adamw_step(p, _f32(g), _ptr(m_codes), _ptr(m_absmax), _ptr(v_codes), _ptr(v_meta),
                        p.size, m_block, v_block, v_bits,
                        C.byref(_hp(AdamWHP, hp)), t, _ptr(mf), _ptr(vf))
    return (mf, vf) if want_fresh else None


# -------------------------------------------------------------- Adafactor ----
def adafactor_update_fp32(p, g, rows, cols, R, C_, M, hp: dict, t: int):
    _lib.ora_adafactor_update_fp32(p, _f32(g), rows, cols, R, C_, _ptr(M),
                                   C.byref(_hp(AdafactorHP, hp)), t)


def adafactor_step(p, g, rows, cols, r_codes, r_meta, c_codes, c_meta,
                   fac_bits, fac_block, m_codes, m_absmax, m_block, hp: dict,
                   t: int, want_fresh: bool = False):
    Rf = np.zeros(rows, np.float32) if want_fresh else None
    Cf = np.zeros(cols, np.float32) if want_fresh else None
    Mf = np.zeros(rows * cols, np.float32) if (want_fresh and m_codes is not None) else None
    _lib.ora_adafactor_step(p, _f32(g), rows, cols, _ptr(r_codes), r_meta,
                            _ptr(c_codes), c_meta, fac_bits, fac_block,
                            _ptr(m_codes), _ptr(m_absmax), m_block,
                            C.byref(_hp(AdafactorHP, hp)), t, _ptr(Rf), _ptr(Cf),
                            _ptr(Mf))
    return (Rf, Cf, Mf) if want_fresh else None


# ------------------------------------------------------------------- CAME ----
def came_update_fp32(p, g, rows, cols, Vr, Vc, Cr, Cc, M, hp: dict, t: int):
    _lib.ora_came_update_fp32(p, _f32(g), rows, cols, Vr, Vc, Cr, Cc, M,
                              C.byref(_hp(CameHP, hp)), t)


def came_step(p, g, rows, cols, vr_codes, vr_meta, vc_codes, vc_meta, v_bits,
              v_block, cr_codes, cr_meta, cc_codes, cc_meta, c_bits, c_block,
              m_codes, m_absmax, m_block, hp: dict, t: int,
              want_fresh: bool = False):
    fresh = np.zeros(2 * rows + 2 * cols + rows * cols, np.float32) if want_fresh else None
    _lib.ora_came_step(p, _f32(g), rows, cols, _ptr(vr_codes), vr_meta,
                       _ptr(vc_codes), vc_meta, v_bits, v_block, _ptr(cr_codes),
                       cr_meta, _ptr(cc_codes), cc_meta, c_bits, c_block,
                       m_codes, m_absmax, m_block, C.byref(_hp(CameHP, hp)), t,
                       _ptr(fresh))
    if not want_fresh:
        return None
    o = [0, rows, rows + cols, 2 * rows + cols, 2 * rows + 2 * cols]
    return (fresh[o[0]:o[1]], fresh[o[1]:o[2]], fresh[o[2]:o[3]],
            fresh[o[3]:o[4]], fresh[o[4]:])


# ----------------------------------------------------------------- APOLLO ----
def f32_to_bf16(x) -> np.ndarray:
    x = _f32(x)
    return np.array([_lib.ora_f32_to_bf16(float(v)) for v in x.ravel()],
                    dtype=np.uint16).reshape(x.shape)


def bf16_to_f32(b) -> np.ndarray:
    b = np.asarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def apollo_project(g, rows, cols, proj, rank):
    L = cols if rows <= cols else rows
    R = np.zeros(L * rank, np.float32)
    _lib.ora_apollo_project(_f32(g), rows, cols,
                            np.ascontiguousarray(proj, np.uint16), rank, R)
    return R


def apollo_update_fp32(p, g, rows, cols, proj, MP, VP, prev_norm, hp: dict,
                       t: int):
    """fp32-state APOLLO in place; returns (scales, new prev_norm)."""
    L = cols if rows <= cols else rows
    s = np.zeros(L, np.float32)
    pn = _flt(float(prev_norm))
    _lib.ora_apollo_update_fp32(p, _f32(g), rows, cols,
                                np.ascontiguousarray(proj, np.uint16), MP, VP,
                                C.byref(pn), C.byref(_hp(ApolloHP, hp)), t,
                                _ptr(s))
    return s, np.float32(pn.value)


def apollo_step(p, g, rows, cols, proj, m_codes, m_absmax, m_block, v_codes,
                v_meta, v_bits, v_block, prev_norm, hp: dict, t: int,
                want_fresh: bool = False):
    """Quantized APOLLO in place; returns (scales, prev_norm[, MP, VP])."""
    L = cols if rows <= cols else rows
    s = np.zeros(L, np.float32)
    pn = _flt(float(prev_norm))
    npj = L * hp["rank"]
    MPf = np.zeros(npj, np.float32) if want_fresh else None
    VPf = np.zeros(npj, np.float32) if want_fresh else None
    _lib.ora_apollo_step(p, _f32(g), rows, cols,
                         np.ascontiguousarray(proj, np.uint16), m_codes,
                         m_absmax, m_block, _ptr(v_codes), v_meta, v_bits,
                         v_block, C.byref(pn), C.byref(_hp(ApolloHP, hp)), t,
                         _ptr(s), _ptr(MPf), _ptr(VPf))
    if want_fresh:
        return s, np.float32(pn.value), MPf, VPf
    return s, np.float32(pn.value)


def apollo_step_given_R(p, g, rows, cols, R, m_codes, m_absmax, m_block, v_codes,
                        v_meta, v_bits, v_block, prev_norm, hp: dict, t: int):
    """Quantized APOLLO step in place for a given projection R (teacher-forced
    parity of everything after the projection); returns (scales, prev_norm)."""
    L = cols if rows <= cols else rows
    s = np.zeros(L, np.float32)
    pn = _flt(float(prev_norm))
    _lib.ora_apollo_step_given_R(p, _f32(g), rows, cols, _f32(R), m_codes, m_absmax,
                                 m_block, _ptr(v_codes), v_meta, v_bits, v_block,
                                 C.byref(pn), C.byref(_hp(ApolloHP, hp)), t, _ptr(s))
    return s, np.float32(pn.value)


def update_error(u_hat, u_ref, eps: float = 1e-12) -> float:
    """Relative update error of Eq. (2)."""
    a, b = _f32(u_hat).ravel(), _f32(u_ref).ravel()
    return float(_lib.ora_update_error(a, b, a.size, eps))
