"""The OpenMP build of the oracle (the benchmark's all-core CPU baseline)
gives the plain build's results bit for bit: its parallel loops have
independent iterations and every reduction keeps its sequential order."""
import math

import numpy as np
import pytest

import oracle as ora
from paper_2608_22322_gb300 import workloads as wl

FLOOR = float(np.float32(math.log2(1e-16)))


def _run(threaded):
    if threaded and ora.use_threads(True) == 1 and ora._lib is ora._lib_plain:
        pytest.skip("no OpenMP in this compiler")
    try:
        out = {}
        # AdamW over an odd-sized tensor
        n = 256 * 777 + 13
        p = (wl.rng(1).standard_normal(n) * 0.02).astype(np.float32)
        mc, ma = np.zeros(n, np.int8), np.zeros(-(-n // 256), np.float32)
        vc, vm = np.zeros(n, np.uint8), np.zeros(2 * -(-n // 256), np.float32)
        hp = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01, log_floor=FLOOR)
        for t in (1, 2, 3):
            ora.adamw_step(p, wl.gaussian_grad((n,), 1e-3, 10 + t), mc, ma, vc, vm, 256, 256, 8,
                           hp, t)
        out["adamw"] = (p, mc, ma, vc, vm)
        # CAME (factored sums over rows and columns, residual sums)
        rows, cols = 96, 200
        st = [np.zeros(rows, np.uint16), np.zeros(2, np.float32), np.zeros(cols, np.uint16),
              np.zeros(4, np.float32)]
        cst = [x.copy() for x in st]
        pc = wl.param_init((rows, cols), 3).ravel()
        cmc, cma = np.zeros(rows * cols, np.int8), np.zeros(rows * cols // 256 + 1, np.float32)
        chp = dict(lr=1e-4, beta1=0.9, beta2=0.999, beta3=0.9999, eps1=1e-30, eps2=1e-16,
                   clip_d=1.0, weight_decay=0.0, log_floor_v=-99.66, log_floor_c=FLOOR)
        for t in (1, 2):
            ora.came_step(pc, wl.student_t_grad((rows, cols), 1e-3, 3.0, 0.05, 50 + t).ravel(),
                          rows, cols, *st, 16, 128, *cst, 16, 128, cmc, cma, 256, chp, t)
        out["came"] = (pc, cmc, cma, *st, *cst)
        # APOLLO with the projection and the limiter, channels over rows
        r_, c_, rank = 160, 48, 16
        P = wl.bf16_bits(wl.gaussian_projection(rank, c_, 4))
        pa = wl.param_init((r_, c_), 5).ravel()
        amc, ama = np.zeros(r_ * rank, np.int8), np.zeros(r_, np.float32)
        avc, avm = np.zeros(r_ * rank, np.uint8), np.zeros(2 * r_, np.float32)
        ahp = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0, weight_decay=0.0,
                   norm_growth_gamma=1.01, log_floor=FLOOR, rank=rank)
        prev = 0.0
        for t in (1, 2):
            s, prev = ora.apollo_step(pa, wl.gaussian_grad((r_, c_), 1e-3, 70 + t).ravel(), r_,
                                      c_, P, amc, ama, rank, avc, avm, 8, rank, prev, ahp, t)
        out["apollo"] = (pa, amc, ama, avc, avm, s, np.array([prev], np.float32))
        return out
    finally:
        ora.use_threads(False)


def test_threaded_oracle_equals_plain():
    a = _run(False)
    b = _run(True)
    for k in a:
        for x, y in zip(a[k], b[k]):
            assert np.array_equal(np.asarray(x).view(np.uint8), np.asarray(y).view(np.uint8)), k
