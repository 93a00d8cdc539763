"""torch.optim optimizers over the library's quantized steps.

Drop-in optimizers whose states are stored as the paper stores them: the
second moment (AdamW), the factored second moment (Adafactor), the factored
second moment and confidence (CAME) and the projected second moment (APOLLO)
AL-coded (Sec. 4.1, AL8 or AL16 per role, Sec. 6.2), momentum UF8-coded
(Sec. 4.3). Every step runs in the CUDA library through the C ABI (there is
no CPU path); this module only keeps the per-parameter state tensors, groups
the parameters into launches and follows torch.optim's conventions
(param_groups, state_dict / load_state_dict, closures, learning-rate
schedulers changing group["lr"]).

Per-role precision (Sec. 4.5; Sec. 6.2, "AL8 second moments with UF8
momentum", "AL16 for both V and C"): each param group chooses the bit width
of its states (v_bits, c_bits, fac_bits: 8 or 16 for AL codes, 32 for the
unquantized FP32 role; AdamW's v_bits 32 keeps m in fp32 too) and block
sizes; migrate_bits() re-codes a trained AL state from AL8 to AL16 or back
through the codec. Parameter grouping (Sec. 6.1): G0 gives every parameter
the selected configuration; g1_param_groups() builds G1, which keeps the
states of one-dimensional tensors, biases, normalization parameters, token
embeddings and the language-model head unquantized. Parameters that a method
cannot take (APOLLO needs matrices) are routed to the quantized AdamW step.
The factored optimizers step each param group's matrices in grouped
launches (al_adafactor_step_multi / al_came_step_multi).
"""
from __future__ import annotations

import math

import torch

from . import binding as B

__all__ = ["AdamW", "Adafactor", "CAME", "Apollo", "g1_param_groups"]


def _log2_floor(x: float) -> float:
    """l_floor = log2(x) rounded to fp32 (Sec. 4.1: the log of the squared
    numerical floor)."""
    import numpy as np
    return float(np.float32(math.log2(x)))


def _code_dtype(bits: int):
    """Storage dtype of a state of this width (AL16 codes travel as int16
    bits; 32 is the unquantized fp32 state)."""
    return torch.uint8 if bits == 8 else torch.int16 if bits == 16 else torch.float32


def _check_bits(bits: int, what: str):
    if bits not in (8, 16, 32):
        raise ValueError(f"{what} must be 8, 16 or 32")


def g1_param_groups(named_parameters, protected: dict, others: dict = None,
                    patterns=("bias", "norm", "embed", "lm_head", "wte", "wpe")):
    """Sec. 6.1's G1 grouping: one-dimensional tensors, biases, normalization
    parameters, token embeddings and the language-model head (by name: any of
    `patterns` in the parameter's name) form a protected group whose options
    are `protected` (e.g. dict(v_bits=32) for AdamW, dict(fac_bits=32) for
    Adafactor: states unquantized); the remaining tensors keep `others` (the
    selected low-precision path). Returns param groups for the optimizers of
    this module. G0 is simply all parameters in one group."""
    prot, rest = [], []
    for name, p in named_parameters:
        low = name.lower()
        (prot if p.dim() <= 1 or any(k in low for k in patterns) else rest).append(p)
    groups = []
    if rest:
        groups.append(dict(params=rest, **(others or {})))
    if prot:
        groups.append(dict(params=prot, **protected))
    return groups


def _check_param(p: torch.Tensor, what: str):
    if not p.is_cuda or p.dtype != torch.float32 or not p.is_contiguous():
        raise ValueError(f"{what}: parameters must be contiguous float32 CUDA tensors")
    if p.grad is not None and (p.grad.dtype != torch.float32 or not p.grad.is_contiguous()):
        raise ValueError(f"{what}: gradients must be contiguous float32")


def _blocks(n: int, block: int) -> int:
    return (n + block - 1) // block


class _Base(torch.optim.Optimizer):
    """Shared conventions: integer code tensors survive load_state_dict (torch
    casts every non-step state tensor to the parameter's dtype), and
    migrate_bits re-codes AL states."""

    # state key -> group key holding its bit width (None: UF8 int8 codes)
    _CODES: dict = {}
    # group key whose value 32 keeps the momentum in fp32 too (AdamW)
    _M_FOLLOWS = None
    # AL state key -> (metadata key, group key of its block size)
    _AL: dict = {}

    def load_state_dict(self, state_dict):
        super().load_state_dict(state_dict)
        for group in self.param_groups:
            for p in group["params"]:
                st = self.state.get(p)
                if not st:
                    continue
                for key, bits_key in self._CODES.items():
                    if key in st:
                        if bits_key is None:
                            raw = self._M_FOLLOWS and group[self._M_FOLLOWS] == 32
                            dt = torch.float32 if raw else torch.int8
                        else:
                            dt = _code_dtype(group[bits_key])
                        st[key] = st[key].to(dtype=dt)

    @torch.no_grad()
    def migrate_bits(self, bits_key: str, new_bits: int):
        """Re-code every AL state whose width is group[bits_key] to new_bits
        (8 or 16): decode with the current width, encode with the new one
        (Eq. (4)-(5)); block sizes and l_floor are unchanged."""
        if new_bits not in (8, 16):
            raise ValueError("new_bits must be 8 or 16")
        for group in self.param_groups:
            old = group[bits_key]
            if old == new_bits:
                continue
            if old == 32:
                raise ValueError("migrate_bits re-codes AL8/AL16 states; an FP32 group stays FP32")
            for p in group["params"]:
                st = self.state.get(p)
                if not st:
                    continue
                for key, (meta_key, block_key) in self._AL.items():
                    if key not in st or self._CODES.get(key) != bits_key:
                        continue
                    codes, meta = st[key], st[meta_key]
                    block = group[block_key]
                    vals = torch.empty(codes.numel(), dtype=torch.float32, device=codes.device)
                    B.al_decode(codes, meta, block, old, vals)
                    new_codes = torch.empty(codes.numel(), dtype=_code_dtype(new_bits),
                                            device=codes.device)
                    B.al_encode(vals, block, new_bits, group[self._floor_key(key)], new_codes, meta)
                    st[key] = new_codes
            group[bits_key] = new_bits

    def _floor_key(self, state_key: str) -> str:
        return "log_floor"


class AdamW(_Base):
    """AdamW (Sec. 3.1, Eq. (1)) with UF8 momentum and AL-coded second moment;
    one fused launch per group and step over every parameter with a gradient
    (al_adamw_step_multi). v_bits 8 or 16 (AL8/AL16 V, UF8 M) or 32 (m and
    v unquantized fp32), blocks powers of two in [128, 4096]; log_floor
    defaults to log2(eps^2)."""

    _CODES = {"m_codes": None, "v_codes": "v_bits"}
    _AL = {"v_codes": ("v_meta", "v_block")}
    _M_FOLLOWS = "v_bits"

    def __init__(self, params, lr=1e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=1e-2,
                 v_bits=8, v_block=256, m_block=256, log_floor=None):
        _check_bits(v_bits, "v_bits")
        defaults = dict(lr=lr, betas=betas, eps=eps, weight_decay=weight_decay, v_bits=v_bits,
                        v_block=v_block, m_block=m_block,
                        log_floor=log_floor if log_floor is not None else _log2_floor(eps * eps))
        super().__init__(params, defaults)
        self._plans: dict = {}

    def _init_state(self, p, group):
        n = p.numel()
        st = self.state[p]
        st["step"] = 0
        raw = group["v_bits"] == 32
        st["m_codes"] = torch.zeros(n, dtype=torch.float32 if raw else torch.int8, device=p.device)
        st["m_absmax"] = torch.zeros(0 if raw else _blocks(n, group["m_block"]),
                                     dtype=torch.float32, device=p.device)
        st["v_codes"] = torch.zeros(n, dtype=_code_dtype(group["v_bits"]), device=p.device)
        st["v_meta"] = torch.zeros(0 if raw else 2 * _blocks(n, group["v_block"]),
                                   dtype=torch.float32, device=p.device)

    def _plan(self, tensors, group):
        """A cached plan over these tensors, keyed on the addresses of the
        parameters and states only: gradients are rebound at every step
        (the plan holds none, so freed gradients are not kept alive)."""
        key = (_state_key(tensors, ("p", "m_codes", "m_absmax", "v_codes", "v_meta")),
               group["m_block"], group["v_block"], group["v_bits"])
        plan = self._plans.get(key)
        if plan is None:
            if len(self._plans) > 64:
                self._plans.clear()
            plan = B.AdamWPlan(tensors, group["m_block"], group["v_block"], group["v_bits"])
            self._plans[key] = plan
        return plan

    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        for group in self.param_groups:
            buckets: dict = {}
            for p in group["params"]:
                if p.grad is None:
                    continue
                _check_param(p, "AdamW")
                if not self.state[p]:
                    self._init_state(p, group)
                st = self.state[p]
                st["step"] += 1
                buckets.setdefault(st["step"], []).append(
                    dict(p=p, g=p.grad, m_codes=st["m_codes"], m_absmax=st["m_absmax"],
                         v_codes=st["v_codes"], v_meta=st["v_meta"]))
            b1, b2 = group["betas"]
            hp = dict(lr=group["lr"], beta1=b1, beta2=b2, eps=group["eps"],
                      weight_decay=group["weight_decay"], log_floor=group["log_floor"])
            for t, tensors in buckets.items():
                self._plan(tensors, group).step(hp, t, grads=[x["g"] for x in tensors])
        return loss

    def migrate_bits(self, bits_key: str = "v_bits", new_bits: int = 16):
        self._plans.clear()
        super().migrate_bits(bits_key, new_bits)


def _state_key(items, keys):
    """Plan cache key: the addresses of the parameters and states a plan
    binds (never the gradients')."""
    return tuple(tuple(0 if it.get(k) is None else it[k].data_ptr() for k in keys)
                 for it in items)


def _as_matrix(p: torch.Tensor):
    """(rows, cols) of a parameter for the factored steps: a matrix as is,
    higher ranks flattened to [shape[0], rest], vectors as [1, n]."""
    if p.dim() >= 2:
        return p.shape[0], p.numel() // p.shape[0]
    return 1, p.numel()


class Adafactor(_Base):
    """Adafactor (Sec. 3.1: factored second moment) with AL-coded row/column
    factors (fac_bits 8 or 16, fac_block; 32: unquantized fp32 factors) and
    optional UF8 momentum (beta1 > 0); rho_t = 1 - t^decay_rate, RMS clip d.
    Vectors are treated as 1 x n matrices. Each group's matrices step in one
    grouped launch per pass."""

    _CODES = {"r_codes": "fac_bits", "c_codes": "fac_bits", "m_codes": None}
    _AL = {"r_codes": ("r_meta", "fac_block"), "c_codes": ("c_meta", "fac_block")}

    def __init__(self, params, lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9,
                 weight_decay=0.0, fac_bits=16, fac_block=128, m_block=256, log_floor=None):
        _check_bits(fac_bits, "fac_bits")
        defaults = dict(lr=lr, eps1=eps1, clip_d=clip_d, decay_rate=decay_rate, beta1=beta1,
                        weight_decay=weight_decay, fac_bits=fac_bits, fac_block=fac_block,
                        m_block=m_block,
                        log_floor=log_floor if log_floor is not None else _log2_floor(eps1))
        super().__init__(params, defaults)
        self._plans: dict = {}

    def _init_state(self, p, group):
        rows, cols = _as_matrix(p)
        dev, fb = p.device, group["fac_block"]
        st = self.state[p]
        st["step"] = 0
        raw = group["fac_bits"] == 32
        st["r_codes"] = torch.zeros(rows, dtype=_code_dtype(group["fac_bits"]), device=dev)
        st["r_meta"] = torch.zeros(0 if raw else 2 * _blocks(rows, fb), dtype=torch.float32,
                                   device=dev)
        st["c_codes"] = torch.zeros(cols, dtype=_code_dtype(group["fac_bits"]), device=dev)
        st["c_meta"] = torch.zeros(0 if raw else 2 * _blocks(cols, fb), dtype=torch.float32,
                                   device=dev)
        if group["beta1"] > 0:
            st["m_codes"] = torch.zeros(p.numel(), dtype=torch.int8, device=dev)
            st["m_absmax"] = torch.zeros(_blocks(p.numel(), group["m_block"]),
                                         dtype=torch.float32, device=dev)

    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        for group in self.param_groups:
            hp = {k: group[k] for k in ("lr", "eps1", "clip_d", "decay_rate", "beta1",
                                        "weight_decay", "log_floor")}
            buckets: dict = {}
            for p in group["params"]:
                if p.grad is None:
                    continue
                _check_param(p, "Adafactor")
                if not self.state[p]:
                    self._init_state(p, group)
                st = self.state[p]
                st["step"] += 1
                rows, cols = _as_matrix(p)
                buckets.setdefault(st["step"], []).append(
                    dict(p=p, g=p.grad, rows=rows, cols=cols, vr_codes=st["r_codes"],
                         vr_meta=st["r_meta"], vc_codes=st["c_codes"], vc_meta=st["c_meta"],
                         m_codes=st.get("m_codes"), m_absmax=st.get("m_absmax")))
            for t, mats in buckets.items():
                _grouped_plan(self._plans, B.AL_OP_ADAFACTOR, mats, group["fac_bits"],
                              group["fac_block"], 16, 128, group["m_block"]).step(
                                  hp, t, grads=[m["g"] for m in mats])
        return loss


def _grouped_plan(cache: dict, op, mats, v_bits, v_block, c_bits, c_block, m_block):
    """A cached FactoredPlan over these matrices (plans bind pointers; the
    key holds parameter and state addresses, gradients are rebound at each
    step)."""
    key = (op, v_bits, v_block, c_bits, c_block, m_block,
           _state_key(mats, ("p", "vr_codes", "vr_meta", "vc_codes", "vc_meta", "cr_codes",
                             "cr_meta", "cc_codes", "cc_meta", "m_codes", "m_absmax")))
    plan = cache.get(key)
    if plan is None:
        if len(cache) > 64:
            cache.clear()
        plan = B.FactoredPlan(op, mats, v_bits, v_block, c_bits, c_block, m_block)
        cache[key] = plan
    return plan


class CAME(_Base):
    """CAME (Sec. 3.1: dense momentum, factored second moment and factored
    confidence; beta3 0.9999 in Sec. 6.1) with AL-coded factors (v_bits and
    c_bits, 8 or 16; 32: unquantized fp32 factors, e.g. the paper's FP32-C
    variant c_bits=32) and UF8 momentum. Each group's matrices step in one
    grouped launch per pass."""

    _CODES = {"vr_codes": "v_bits", "vc_codes": "v_bits", "cr_codes": "c_bits",
              "cc_codes": "c_bits", "m_codes": None}
    _AL = {"vr_codes": ("vr_meta", "v_block"), "vc_codes": ("vc_meta", "v_block"),
           "cr_codes": ("cr_meta", "c_block"), "cc_codes": ("cc_meta", "c_block")}

    def __init__(self, params, lr=1e-4, betas=(0.9, 0.999, 0.9999), eps=(1e-30, 1e-16),
                 clip_d=1.0, weight_decay=0.0, v_bits=16, v_block=128, c_bits=16, c_block=128,
                 m_block=256):
        _check_bits(v_bits, "v_bits")
        _check_bits(c_bits, "c_bits")
        defaults = dict(lr=lr, betas=betas, eps=eps, clip_d=clip_d, weight_decay=weight_decay,
                        v_bits=v_bits, v_block=v_block, c_bits=c_bits, c_block=c_block,
                        m_block=m_block, log_floor_v=_log2_floor(eps[0]),
                        log_floor_c=_log2_floor(eps[1]))
        super().__init__(params, defaults)
        self._plans: dict = {}

    def _floor_key(self, state_key: str) -> str:
        return "log_floor_c" if state_key.startswith("c") else "log_floor_v"

    def _init_state(self, p, group):
        rows, cols = _as_matrix(p)
        dev = p.device
        st = self.state[p]
        st["step"] = 0
        for pre, bits, blk in (("v", group["v_bits"], group["v_block"]),
                               ("c", group["c_bits"], group["c_block"])):
            for side, m in (("r", rows), ("c", cols)):
                st[f"{pre}{side}_codes"] = torch.zeros(m, dtype=_code_dtype(bits), device=dev)
                st[f"{pre}{side}_meta"] = torch.zeros(0 if bits == 32 else 2 * _blocks(m, blk),
                                                      dtype=torch.float32, device=dev)
        st["m_codes"] = torch.zeros(p.numel(), dtype=torch.int8, device=dev)
        st["m_absmax"] = torch.zeros(_blocks(p.numel(), group["m_block"]), dtype=torch.float32,
                                     device=dev)

    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        for group in self.param_groups:
            b1, b2, b3 = group["betas"]
            e1, e2 = group["eps"]
            hp = dict(lr=group["lr"], beta1=b1, beta2=b2, beta3=b3, eps1=e1, eps2=e2,
                      clip_d=group["clip_d"], weight_decay=group["weight_decay"],
                      log_floor_v=group["log_floor_v"], log_floor_c=group["log_floor_c"])
            buckets: dict = {}
            for p in group["params"]:
                if p.grad is None:
                    continue
                _check_param(p, "CAME")
                if not self.state[p]:
                    self._init_state(p, group)
                st = self.state[p]
                st["step"] += 1
                rows, cols = _as_matrix(p)
                m = dict(p=p, g=p.grad, rows=rows, cols=cols, m_codes=st["m_codes"],
                         m_absmax=st["m_absmax"])
                for k in ("vr", "vc", "cr", "cc"):
                    m[k + "_codes"], m[k + "_meta"] = st[k + "_codes"], st[k + "_meta"]
                buckets.setdefault(st["step"], []).append(m)
            for t, mats in buckets.items():
                _grouped_plan(self._plans, B.AL_OP_CAME, mats, group["v_bits"], group["v_block"],
                              group["c_bits"], group["c_block"], group["m_block"]).step(
                                  hp, t, grads=[m["g"] for m in mats])
        return loss


def _apollo_ok(p: torch.Tensor, rank: int) -> bool:
    if p.dim() != 2:
        return False
    rows, cols = p.shape
    s = min(rows, cols)
    return cols % 4 == 0 and s % 8 == 0 and rows * cols < (1 << 31)


class Apollo(_Base):
    """APOLLO (Sec. 3.1: moments of a random low-rank projection of the
    gradient give a channel-wise scale of the original gradient; rank 256 and
    projection refresh every 200 steps in Sec. 6.1) with UF8 M^P and AL-coded
    V^P (v_bits), stepped for all matrices of a group in one grouped launch
    sequence (al_apollo_step_multi). The projection of each matrix is drawn
    from N(0, 1/rank) (seeded by `seed` and the parameter's index, redrawn
    every proj_gap steps) and rounded to bf16. norm_growth_gamma > 0 turns on
    the norm-growth limiter (each matrix's scaled-gradient norm may grow by at
    most that factor per step; per-matrix state "prev_norm"). Parameters that
    are not eligible matrices (vectors, shapes the kernels do not take) are
    stepped by the quantized AdamW with the same lr, betas, eps and weight
    decay."""

    _CODES = {"m_codes": None, "v_codes": "v_bits"}
    _AL = {"v_codes": ("v_meta", "rank")}

    def __init__(self, params, lr=1e-4, betas=(0.9, 0.999), eps=1e-8, alpha=1.0,
                 weight_decay=0.0, rank=256, v_bits=8, proj_gap=200, seed=0, log_floor=None,
                 norm_growth_gamma=0.0):
        if rank not in (128, 256):
            raise ValueError("rank must be 128 or 256")
        defaults = dict(lr=lr, betas=betas, eps=eps, alpha=alpha, weight_decay=weight_decay,
                        rank=rank, v_bits=v_bits, proj_gap=proj_gap, seed=seed,
                        norm_growth_gamma=norm_growth_gamma,
                        log_floor=log_floor if log_floor is not None else _log2_floor(eps * eps))
        super().__init__(params, defaults)
        others = [p for g in self.param_groups for p in g["params"] if not _apollo_ok(p, rank)]
        self._adamw = (AdamW(others, lr=lr, betas=betas, eps=eps, weight_decay=weight_decay,
                             v_bits=v_bits) if others else None)
        self._other = {id(p) for p in others}
        self._plans: dict = {}

    def _init_state(self, p, group, index):
        rows, cols = p.shape
        r, dev = group["rank"], p.device
        npj = max(rows, cols) * r
        st = self.state[p]
        st["step"] = 0
        st["index"] = index
        st["proj"] = torch.empty(r * min(rows, cols), dtype=torch.int16, device=dev)
        st["m_codes"] = torch.zeros(npj, dtype=torch.int8, device=dev)
        st["m_absmax"] = torch.zeros(npj // r, dtype=torch.float32, device=dev)
        st["v_codes"] = torch.zeros(npj, dtype=_code_dtype(group["v_bits"]), device=dev)
        st["v_meta"] = torch.zeros(2 * (npj // r), dtype=torch.float32, device=dev)
        st["prev_norm"] = torch.zeros(1, dtype=torch.float32, device=dev)

    def _draw_projection(self, p, group, st):
        gen = torch.Generator(device=p.device)
        epoch = (st["step"] - 1) // group["proj_gap"]
        gen.manual_seed(int(group["seed"]) * 1_000_003 + 7919 * st["index"] + epoch)
        P = torch.empty(st["proj"].numel(), dtype=torch.float32, device=p.device)
        P.normal_(0.0, math.sqrt(1.0 / group["rank"]), generator=gen)
        st["proj"].copy_(P.to(torch.bfloat16).view(torch.int16))

    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        if self._adamw is not None:
            self._adamw.param_groups[0]["lr"] = self.param_groups[0]["lr"]
            self._adamw.step()
        index = 0
        for group in self.param_groups:
            buckets: dict = {}
            for p in group["params"]:
                index += 1
                if id(p) in self._other or p.grad is None:
                    continue
                _check_param(p, "Apollo")
                if not self.state[p]:
                    self._init_state(p, group, index)
                st = self.state[p]
                st["step"] += 1
                if (st["step"] - 1) % group["proj_gap"] == 0:
                    self._draw_projection(p, group, st)
                rows, cols = p.shape
                if "prev_norm" not in st:  # a state saved before the limiter existed
                    st["prev_norm"] = torch.zeros(1, dtype=torch.float32, device=p.device)
                buckets.setdefault(st["step"], []).append(
                    dict(p=p, g=p.grad, rows=rows, cols=cols, proj=st["proj"],
                         m_codes=st["m_codes"], m_absmax=st["m_absmax"],
                         v_codes=st["v_codes"], v_meta=st["v_meta"],
                         prev_norm=st["prev_norm"]))
            b1, b2 = group["betas"]
            hp = dict(lr=group["lr"], beta1=b1, beta2=b2, eps=group["eps"],
                      alpha=group["alpha"], weight_decay=group["weight_decay"],
                      norm_growth_gamma=group.get("norm_growth_gamma", 0.0),
                      log_floor=group["log_floor"], rank=group["rank"])
            for t, mats in buckets.items():
                key = (_state_key(mats, ("p", "proj", "m_codes", "m_absmax", "v_codes",
                                         "v_meta", "prev_norm")), group["rank"],
                       group["v_bits"])
                plan = self._plans.get(key)
                if plan is None:
                    if len(self._plans) > 8:
                        self._plans.clear()
                    plan = B.ApolloPlan(mats, group["rank"], group["v_bits"])
                    self._plans[key] = plan
                plan.step(hp, t, grads=[m["g"] for m in mats])
        return loss

    def state_dict(self):
        sd = super().state_dict()
        if self._adamw is not None:
            sd["adamw"] = self._adamw.state_dict()
        return sd

    def load_state_dict(self, state_dict):
        sd = dict(state_dict)
        inner = sd.pop("adamw", None)
        super().load_state_dict(sd)
        for group in self.param_groups:
            for p in group["params"]:
                st = self.state.get(p)
                if st and "proj" in st:
                    st["proj"] = st["proj"].to(dtype=torch.int16)
                if st and "index" in st:
                    st["index"] = int(st["index"])
        if inner is not None and self._adamw is not None:
            self._adamw.load_state_dict(inner)
        self._plans.clear()

    def migrate_bits(self, bits_key: str = "v_bits", new_bits: int = 16):
        self._plans.clear()
        super().migrate_bits(bits_key, new_bits)
        if self._adamw is not None:
            self._adamw.migrate_bits("v_bits", new_bits)
