"""Helpers shared by the GPU parity tests (seeded inputs, comparisons)."""
import math

import numpy as np

from paper_2608_22322_gb300 import workloads as wl

FLOOR = float(np.float32(math.log2(1e-16)))
ADAMW_HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01,
                log_floor=FLOOR)


def gpu_available() -> bool:
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


def state_mix(n, block, seed):
    """Non-negative fp32 state covering the codec's regimes block by block:
    narrow/medium/wide log-uniform spreads, 10% exact zeros, an all-zero
    block, a constant block, a block below the floor, -0.0 entries and a
    ragged tail."""
    r = wl.rng(seed)
    x = np.empty(n, np.float32)
    nb = (n + block - 1) // block
    for b in range(nb):
        lo, hi = b * block, min(n, (b + 1) * block)
        kind = b % 6
        if kind == 0:
            v = np.exp2(r.uniform(-30, -28, hi - lo))
        elif kind == 1:
            v = np.exp2(r.uniform(-40, -20, hi - lo))
        elif kind == 2:
            v = np.exp2(r.uniform(-90, 40, hi - lo))
        elif kind == 3:
            v = np.full(hi - lo, 3.3e-7)
        elif kind == 4:
            v = np.exp2(r.uniform(-80, -60, hi - lo))  # below the -53 floor
        else:
            v = (r.standard_normal(hi - lo) * 1e-3) ** 2
        x[lo:hi] = v.astype(np.float32)
    x[r.random(n) < 0.1] = 0.0
    if nb > 2:
        x[block:2 * block] = 0.0
    x[::97] = -0.0
    return x


def bytes_equal(a: np.ndarray, b: np.ndarray) -> int:
    """Number of differing bytes between two arrays of the same layout."""
    a = np.ascontiguousarray(a).view(np.uint8)
    b = np.ascontiguousarray(b).view(np.uint8)
    assert a.shape == b.shape
    return int(np.sum(a != b))


def step_size(p_new: np.ndarray, p_old: np.ndarray, hp: dict) -> np.ndarray:
    """|lr * u| of an AdamW step, recovered from the oracle's parameters
    before and after it: p_new - (1 - lr wd) p_old."""
    decay = 1.0 - hp["lr"] * hp["weight_decay"]
    return np.abs(p_new.astype(np.float64) - decay * p_old.astype(np.float64))


def params_off(ref: np.ndarray, got: np.ndarray, steps: np.ndarray, rtol: float = 1e-5) -> int:
    """Number of parameters outside |got - ref| <= rtol (|ref| + steps).

    The fused AdamW kernel forms the update direction u = m / (sqrt(v) c2 +
    eps) with the hardware's approximate square root and reciprocal (a few
    ulp; every state, code and block constant stays exact). Over t steps a
    parameter then drifts from the oracle's by at most about 2^-21 of the
    summed step sizes |lr u| (steps) plus one fp32 rounding of p per step:
    within rtol = 1e-5 of |p| + steps, the parameter tolerance of the
    method's parity bar, for t up to a few hundred."""
    ref = ref.astype(np.float64)
    d = np.abs(got.astype(np.float64) - ref)
    return int(np.sum(~(d <= rtol * (np.abs(ref) + steps))))
