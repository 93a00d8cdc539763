"""ctypes binding of libalq.so (the C ABI of include/alq.h).

Argument marshalling only: every function takes torch CUDA tensors, passes
their device pointers, sizes and the current CUDA stream to the library entry
point of the same name, and raises AlqError on a non-zero status. All the
arithmetic runs in the library's kernels; there is no fallback. If the
library has not been built (paper_2608_22322_gb300.build_lib.build()), loading
this module raises.
"""
from __future__ import annotations

import ctypes as C
import os

import torch

from . import build_lib

_LIB_PATH = build_lib.LIB
if not os.path.exists(_LIB_PATH):
    raise ImportError(
        f"CUDA library {_LIB_PATH} is missing: build it with "
        "paper_2608_22322_gb300.build_lib.build() (or __graft_entry__.build())")
lib = C.CDLL(_LIB_PATH)

ALQ_OK = 0
AL_OP_ADAFACTOR, AL_OP_CAME, AL_OP_APOLLO = 1, 2, 3


class AlqError(RuntimeError):
    def __init__(self, fn: str, status: int):
        name = lib.alq_status_string(status).decode()
        extra = lib.alq_last_cuda_error().decode()
        super().__init__(f"{fn} failed: {name}" + (f" ({extra})" if extra else ""))
        self.status = status


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


class AdamWTensor(C.Structure):
    _fields_ = [("p", C.c_void_p), ("g", C.c_void_p), ("m_codes", C.c_void_p),
                ("m_absmax", C.c_void_p), ("v_codes", C.c_void_p),
                ("v_meta", C.c_void_p), ("n", C.c_int64)]


class ApolloMatrix(C.Structure):
    _fields_ = [("p", C.c_void_p), ("g", C.c_void_p), ("rows", C.c_int64),
                ("cols", C.c_int64), ("proj", C.c_void_p), ("m_codes", C.c_void_p),
                ("m_absmax", C.c_void_p), ("v_codes", C.c_void_p), ("v_meta", C.c_void_p),
                ("prev_norm", C.c_void_p)]


class ApolloInfo(C.Structure):
    _fields_ = [("nmat", C.c_int32), ("rank", C.c_int32), ("v_bits", C.c_int32),
                ("limiter_ok", C.c_int32), ("total_params", C.c_int64),
                ("total_channels", C.c_int64), ("gemm_tiles", C.c_int64), ("mom_tiles", C.c_int64),
                ("upd_tiles", C.c_int64), ("workspace", C.c_void_p),
                ("norm_chunks", C.c_int64)]


class FactoredMatrix(C.Structure):
    _fields_ = [("p", C.c_void_p), ("g", C.c_void_p), ("rows", C.c_int64),
                ("cols", C.c_int64), ("vr_codes", C.c_void_p), ("vr_meta", C.c_void_p),
                ("vc_codes", C.c_void_p), ("vc_meta", C.c_void_p), ("cr_codes", C.c_void_p),
                ("cr_meta", C.c_void_p), ("cc_codes", C.c_void_p), ("cc_meta", C.c_void_p),
                ("m_codes", C.c_void_p), ("m_absmax", C.c_void_p)]


class FactoredInfo(C.Structure):
    _fields_ = [("nmat", C.c_int32), ("op", C.c_int32), ("v_bits", C.c_int32),
                ("v_block", C.c_int32), ("c_bits", C.c_int32), ("c_block", C.c_int32),
                ("m_block", C.c_int32), ("has_momentum", C.c_int32),
                ("total_params", C.c_int64), ("sumsq_tiles", C.c_int64),
                ("factor_tiles", C.c_int64), ("factor2_tiles", C.c_int64),
                ("scale_tiles", C.c_int64), ("tiles", C.c_int64), ("rms_chunks", C.c_int64),
                ("workspace", C.c_void_p)]


class MultiInfo(C.Structure):
    _fields_ = [("ntensors", C.c_int32), ("m_block", C.c_int32),
                ("v_block", C.c_int32), ("v_bits", C.c_int32),
                ("total_tiles", C.c_int64), ("total_elems", C.c_int64)]


_vp, _i64, _int, _flt = C.c_void_p, C.c_int64, C.c_int, C.c_float


def _sig(name, res, *args):
    f = getattr(lib, name)
    f.restype = res
    f.argtypes = list(args)


_sig("alq_status_string", C.c_char_p, _int)
_sig("alq_last_cuda_error", C.c_char_p)
_sig("alq_version", _int)
_sig("al_num_blocks", _i64, _i64, _int)
_sig("al_meta_count", _i64, _i64, _int)
_sig("al_state_bytes", _i64, _i64, _int, _int)
_sig("al_encode", _int, _vp, _i64, _int, _int, _flt, _vp, _vp, _vp)
_sig("al_decode", _int, _vp, _vp, _i64, _int, _int, _vp, _vp)
_sig("uf8_encode", _int, _vp, _i64, _int, _vp, _vp, _vp)
_sig("uf8_decode", _int, _vp, _vp, _i64, _int, _vp, _vp)
_sig("al_adamw_step", _int, _vp, _vp, _vp, _vp, _vp, _vp, _i64, _int, _int, _int,
     C.POINTER(AdamWHP), _i64, _vp)
_sig("al_adamw_plan_bytes", _int, _int, C.POINTER(C.c_size_t))
_sig("al_adamw_plan", _int, C.POINTER(AdamWTensor), _int, _int, _int, _int, _vp,
     C.c_size_t, C.POINTER(MultiInfo))
_sig("al_adamw_step_multi", _int, _vp, C.POINTER(MultiInfo), C.POINTER(AdamWHP), _i64, _vp)
_sig("al_workspace_size", _int, _int, _i64, _i64, _int, C.POINTER(C.c_size_t))
_sig("al_adafactor_step", _int, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _vp, _int, _int,
     _vp, _vp, _int, C.POINTER(AdafactorHP), _i64, _vp, C.c_size_t, _vp)
_sig("al_adafactor_step_noalloc", _int, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _vp, _int, _int,
     _vp, _vp, _int, C.POINTER(AdafactorHP), _i64, _vp)
_sig("al_adafactor_noalloc_capacity", C.c_size_t)
_sig("al_came_step", _int, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _vp, _int, _int,
     _vp, _vp, _vp, _vp, _int, _int, _vp, _vp, _int, C.POINTER(CameHP), _i64, _vp,
     C.c_size_t, _vp)
_sig("al_factored_plan_bytes", _int, C.POINTER(FactoredMatrix), _int, C.POINTER(C.c_size_t))
_sig("al_factored_workspace_multi", _int, C.POINTER(FactoredMatrix), _int,
     C.POINTER(C.c_size_t))
_sig("al_factored_plan", _int, _int, C.POINTER(FactoredMatrix), _int, _int, _int, _int, _int,
     _int, _vp, C.c_size_t, _vp, C.c_size_t, C.POINTER(FactoredInfo))
_sig("al_adafactor_step_multi", _int, _vp, C.POINTER(FactoredInfo), C.POINTER(AdafactorHP),
     _i64, _vp)
_sig("al_came_step_multi", _int, _vp, C.POINTER(FactoredInfo), C.POINTER(CameHP), _i64, _vp)
_sig("al_apollo_plan_bytes", _int, C.POINTER(ApolloMatrix), _int, C.POINTER(C.c_size_t))
_sig("al_apollo_workspace_multi", _int, C.POINTER(ApolloMatrix), _int, _int,
     C.POINTER(C.c_size_t))
_sig("al_apollo_plan", _int, C.POINTER(ApolloMatrix), _int, _int, _int, _vp, C.c_size_t, _vp,
     C.c_size_t, C.POINTER(ApolloInfo))
_sig("al_apollo_step_multi", _int, _vp, C.POINTER(ApolloInfo), C.POINTER(ApolloHP), _i64, _vp)
_sig("al_apollo_step", _int, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _int, _vp, _vp,
     _int, _int, _vp, C.POINTER(ApolloHP), _i64, _vp, C.c_size_t, _vp)


# ------------------------------------------------------------------ helpers --
def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream=None):
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _check(fn, st):
    if st != ALQ_OK:
        raise AlqError(fn, st)


def _hp(cls, d):
    return cls(**{k: d[k] for k, _ in cls._fields_})


# ------------------------------------------------------------------- sizes --
def version() -> int:
    return lib.alq_version()


def al_num_blocks(n: int, block: int) -> int:
    return lib.al_num_blocks(n, block)


def al_meta_count(n: int, block: int) -> int:
    return lib.al_meta_count(n, block)


def al_state_bytes(n: int, block: int, bits: int) -> int:
    return lib.al_state_bytes(n, block, bits)


def al_workspace_size(op: int, rows: int, cols: int, rank: int = 0) -> int:
    b = C.c_size_t(0)
    _check("al_workspace_size", lib.al_workspace_size(op, rows, cols, rank, C.byref(b)))
    return b.value


# ------------------------------------------------------------------- codec --
def al_encode(x, block, bits, log_floor, codes, meta, stream=None):
    _check("al_encode", lib.al_encode(_ptr(x), x.numel(), block, bits, log_floor,
                                      _ptr(codes), _ptr(meta), _stream(stream)))


def al_decode(codes, meta, block, bits, out, stream=None):
    _check("al_decode", lib.al_decode(_ptr(codes), _ptr(meta), out.numel(), block, bits,
                                      _ptr(out), _stream(stream)))


def uf8_encode(m, block, codes, absmax, stream=None):
    _check("uf8_encode", lib.uf8_encode(_ptr(m), m.numel(), block, _ptr(codes),
                                        _ptr(absmax), _stream(stream)))


def uf8_decode(codes, absmax, block, out, stream=None):
    _check("uf8_decode", lib.uf8_decode(_ptr(codes), _ptr(absmax), out.numel(), block,
                                        _ptr(out), _stream(stream)))


# ------------------------------------------------------------------- AdamW --
def al_adamw_step(p, g, m_codes, m_absmax, v_codes, v_meta, m_block, v_block, v_bits,
                  hp: dict, t: int, stream=None):
    h = _hp(AdamWHP, hp)
    _check("al_adamw_step", lib.al_adamw_step(
        _ptr(p), _ptr(g), _ptr(m_codes), _ptr(m_absmax), _ptr(v_codes), _ptr(v_meta),
        p.numel(), m_block, v_block, v_bits, C.byref(h), t, _stream(stream)))


class _BoundPlan:
    """Gradient rebinding shared by the plans. A plan binds device pointers;
    it keeps the optimizer's own arrays (parameters, states, workspace)
    alive but holds no gradient tensor: a training loop that frees its
    gradients every step (zero_grad(set_to_none=True)) passes the current
    ones to step(grads=...), and the host image is rebuilt with their
    addresses and copied to the plan's device buffer, in stream order, only
    when an address changed. A plan stepped without grads uses the
    gradients it was built with, which the caller must keep alive."""

    def _rebind(self, grads, stream):
        ptrs = [_ptr(g) for g in grads]
        if len(ptrs) != len(self._gptrs):
            raise ValueError(f"{type(self).__name__}.step: {len(ptrs)} gradients for "
                             f"{len(self._gptrs)} bound arrays")
        if ptrs == self._gptrs:
            return
        for i, p in enumerate(ptrs):
            self._arr[i].g = p
        self._build()
        self._gptrs = ptrs
        if stream is None:
            self.dev.copy_(self._host)
        else:
            with torch.cuda.stream(stream):
                self.dev.copy_(self._host)


class AdamWPlan(_BoundPlan):
    """Device copy of a multi-tensor AdamW plan (al_adamw_plan) and its host
    summary. `tensors` is a list of dicts with keys p, g, m_codes, m_absmax,
    v_codes, v_meta (torch CUDA tensors); see _BoundPlan for g."""

    def __init__(self, tensors, m_block, v_block, v_bits, device=None):
        nt = len(tensors)
        self._arr = (AdamWTensor * nt)()
        for i, t in enumerate(tensors):
            self._arr[i] = AdamWTensor(_ptr(t["p"]), _ptr(t["g"]), _ptr(t["m_codes"]),
                                       _ptr(t["m_absmax"]), _ptr(t["v_codes"]),
                                       _ptr(t["v_meta"]), t["p"].numel())
        self._gptrs = [_ptr(t["g"]) for t in tensors]
        self._cfg = (m_block, v_block, v_bits)
        nbytes = C.c_size_t(0)
        _check("al_adamw_plan_bytes", lib.al_adamw_plan_bytes(nt, C.byref(nbytes)))
        self._host = torch.zeros(nbytes.value, dtype=torch.uint8)
        self.info = MultiInfo()
        self._build()
        dev = device if device is not None else tensors[0]["p"].device
        self.dev = self._host.to(dev)
        # keep the optimizer's arrays alive while the plan is used (not g)
        self.tensors = [{k: v for k, v in t.items() if k != "g"} for t in tensors]

    def _build(self):
        _check("al_adamw_plan", lib.al_adamw_plan(self._arr, len(self._arr), *self._cfg,
                                                  self._host.data_ptr(), self._host.numel(),
                                                  C.byref(self.info)))

    def step(self, hp: dict, t: int, stream=None, grads=None):
        if grads is not None:
            self._rebind(grads, stream)
        h = _hp(AdamWHP, hp)
        _check("al_adamw_step_multi", lib.al_adamw_step_multi(
            _ptr(self.dev), C.byref(self.info), C.byref(h), t, _stream(stream)))


# --------------------------------------------------------------- factored --
def al_adafactor_step(p, g, rows, cols, r_codes, r_meta, c_codes, c_meta, fac_bits,
                      fac_block, m_codes, m_absmax, m_block, hp: dict, t: int,
                      workspace, stream=None):
    h = _hp(AdafactorHP, hp)
    _check("al_adafactor_step", lib.al_adafactor_step(
        _ptr(p), _ptr(g), rows, cols, _ptr(r_codes), _ptr(r_meta), _ptr(c_codes),
        _ptr(c_meta), fac_bits, fac_block, _ptr(m_codes), _ptr(m_absmax), m_block,
        C.byref(h), t, _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def al_adafactor_step_noalloc(p, g, rows, cols, r_codes, r_meta, c_codes, c_meta, fac_bits,
                              fac_block, m_codes, m_absmax, m_block, hp: dict, t: int,
                              stream=None):
    """al_adafactor_step without a workspace argument: the library supplies
    the scratch from a fixed array of al_adafactor_noalloc_capacity() bytes
    (for callers that cannot allocate device memory)."""
    h = _hp(AdafactorHP, hp)
    _check("al_adafactor_step_noalloc", lib.al_adafactor_step_noalloc(
        _ptr(p), _ptr(g), rows, cols, _ptr(r_codes), _ptr(r_meta), _ptr(c_codes),
        _ptr(c_meta), fac_bits, fac_block, _ptr(m_codes), _ptr(m_absmax), m_block,
        C.byref(h), t, _stream(stream)))


def al_adafactor_noalloc_capacity() -> int:
    return int(lib.al_adafactor_noalloc_capacity())


def al_came_step(p, g, rows, cols, vr_codes, vr_meta, vc_codes, vc_meta, v_bits,
                 v_block, cr_codes, cr_meta, cc_codes, cc_meta, c_bits, c_block,
                 m_codes, m_absmax, m_block, hp: dict, t: int, workspace, stream=None):
    h = _hp(CameHP, hp)
    _check("al_came_step", lib.al_came_step(
        _ptr(p), _ptr(g), rows, cols, _ptr(vr_codes), _ptr(vr_meta), _ptr(vc_codes),
        _ptr(vc_meta), v_bits, v_block, _ptr(cr_codes), _ptr(cr_meta), _ptr(cc_codes),
        _ptr(cc_meta), c_bits, c_block, _ptr(m_codes), _ptr(m_absmax), m_block,
        C.byref(h), t, _ptr(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream)))


def al_apollo_step(p, g, rows, cols, proj, m_codes, m_absmax, m_block, v_codes, v_meta,
                   v_bits, v_block, prev_norm, hp: dict, t: int, workspace, stream=None):
    h = _hp(ApolloHP, hp)
    _check("al_apollo_step", lib.al_apollo_step(
        _ptr(p), _ptr(g), rows, cols, _ptr(proj), _ptr(m_codes), _ptr(m_absmax), m_block,
        _ptr(v_codes), _ptr(v_meta), v_bits, v_block, _ptr(prev_norm), C.byref(h), t,
        _ptr(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


class FactoredPlan(_BoundPlan):
    """A grouped Adafactor or CAME step over many matrices (al_factored_plan
    / al_adafactor_step_multi / al_came_step_multi): owns the workspace and
    the device copy of the plan. `op` is AL_OP_ADAFACTOR or AL_OP_CAME;
    `mats` is a list of dicts with keys p, g, rows, cols, vr_codes, vr_meta,
    vc_codes, vc_meta, and for CAME cr_codes, cr_meta, cc_codes, cc_meta,
    and optionally (always for CAME) m_codes, m_absmax (torch CUDA
    tensors); see _BoundPlan for g."""

    _KEYS = ("vr_codes", "vr_meta", "vc_codes", "vc_meta", "cr_codes", "cr_meta", "cc_codes",
             "cc_meta", "m_codes", "m_absmax")

    def __init__(self, op, mats, v_bits, v_block, c_bits=16, c_block=128, m_block=256,
                 device=None):
        nm = len(mats)
        self._arr = (FactoredMatrix * nm)()
        for i, m in enumerate(mats):
            self._arr[i] = FactoredMatrix(_ptr(m["p"]), _ptr(m["g"]), m["rows"], m["cols"],
                                          *[_ptr(m.get(k)) for k in self._KEYS])
        self._gptrs = [_ptr(m["g"]) for m in mats]
        dev = device if device is not None else mats[0]["p"].device
        ws = C.c_size_t(0)
        _check("al_factored_workspace_multi",
               lib.al_factored_workspace_multi(self._arr, nm, C.byref(ws)))
        self.workspace = torch.zeros(ws.value, dtype=torch.uint8, device=dev)
        nbytes = C.c_size_t(0)
        _check("al_factored_plan_bytes",
               lib.al_factored_plan_bytes(self._arr, nm, C.byref(nbytes)))
        self._host = torch.zeros(nbytes.value, dtype=torch.uint8)
        self.info = FactoredInfo()
        self.op = op
        self._cfg = (v_bits, v_block, c_bits, c_block, m_block)
        self._build()
        self.dev = self._host.to(dev)
        # keep the optimizer's arrays alive while the plan is used (not g)
        self.mats = [{k: v for k, v in m.items() if k != "g"} for m in mats]

    def _build(self):
        _check("al_factored_plan", lib.al_factored_plan(
            self.op, self._arr, len(self._arr), *self._cfg, _ptr(self.workspace),
            self.workspace.numel(), self._host.data_ptr(), self._host.numel(),
            C.byref(self.info)))

    def step(self, hp: dict, t: int, stream=None, grads=None):
        if grads is not None:
            self._rebind(grads, stream)
        if self.op == AL_OP_ADAFACTOR:
            h = _hp(AdafactorHP, hp)
            _check("al_adafactor_step_multi", lib.al_adafactor_step_multi(
                _ptr(self.dev), C.byref(self.info), C.byref(h), t, _stream(stream)))
        else:
            h = _hp(CameHP, hp)
            _check("al_came_step_multi", lib.al_came_step_multi(
                _ptr(self.dev), C.byref(self.info), C.byref(h), t, _stream(stream)))


class ApolloPlan(_BoundPlan):
    """A grouped APOLLO step over many matrices (al_apollo_plan /
    al_apollo_step_multi): owns the workspace and the device copy of the
    plan. `mats` is a list of dicts with keys p, g, rows, cols, proj, m_codes,
    m_absmax, v_codes, v_meta (torch CUDA tensors; proj holds bf16 bits) and
    optionally prev_norm (a one-element fp32 tensor: the norm-growth
    limiter's state, needed on every matrix when hp's norm_growth_gamma >
    0); see _BoundPlan for g."""

    def __init__(self, mats, rank, v_bits, device=None):
        nm = len(mats)
        self._arr = (ApolloMatrix * nm)()
        for i, m in enumerate(mats):
            self._arr[i] = ApolloMatrix(_ptr(m["p"]), _ptr(m["g"]), m["rows"], m["cols"],
                                        _ptr(m["proj"]), _ptr(m["m_codes"]),
                                        _ptr(m["m_absmax"]), _ptr(m["v_codes"]),
                                        _ptr(m["v_meta"]), _ptr(m.get("prev_norm")))
        self._gptrs = [_ptr(m["g"]) for m in mats]
        dev = device if device is not None else mats[0]["p"].device
        ws = C.c_size_t(0)
        _check("al_apollo_workspace_multi",
               lib.al_apollo_workspace_multi(self._arr, nm, rank, C.byref(ws)))
        self.workspace = torch.zeros(ws.value, dtype=torch.uint8, device=dev)
        nbytes = C.c_size_t(0)
        _check("al_apollo_plan_bytes", lib.al_apollo_plan_bytes(self._arr, nm, C.byref(nbytes)))
        self._host = torch.zeros(nbytes.value, dtype=torch.uint8)
        self.info = ApolloInfo()
        self._cfg = (rank, v_bits)
        self._build()
        self.dev = self._host.to(dev)
        # keep the optimizer's arrays alive while the plan is used (not g)
        self.mats = [{k: v for k, v in m.items() if k != "g"} for m in mats]

    def _build(self):
        _check("al_apollo_plan", lib.al_apollo_plan(
            self._arr, len(self._arr), *self._cfg, _ptr(self.workspace),
            self.workspace.numel(), self._host.data_ptr(), self._host.numel(),
            C.byref(self.info)))

    def step(self, hp: dict, t: int, stream=None, grads=None):
        if grads is not None:
            self._rebind(grads, stream)
        h = _hp(ApolloHP, hp)
        _check("al_apollo_step_multi", lib.al_apollo_step_multi(
            _ptr(self.dev), C.byref(self.info), C.byref(h), t, _stream(stream)))
