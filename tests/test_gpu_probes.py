"""The controlled probes of Sec. 5 on the GPU (paper_2608_22322_gb300/probes.py).

The paper does not state its generators, so the probe values are checked
against its qualitative claims and orderings on synthetic log-normal
regimes: adaptive AL8 keeps the single-step update error of Eq. (2) below
1% in the narrow, medium and wide regimes at block size 2048 (Sec. 5.2);
AL16 is far below AL8; over a 5K-step second-moment EMA (beta2 = 0.999,
FP32 momentum in the update error) the drift stays below 1% and rises with
the block size across 256, 512, 1024 and 2048 (Sec. 5.5's sweep: 0.577% ->
0.814%; Sec. 5.6: 0.562% / 0.280% at 256, 0.736% / 0.357% at 2048).

The quantized EMA itself is checked against the oracle: with lr = 0 the
fused step leaves p at zero and only the states evolve, so 5000 steps of
the same gradients through the oracle's AdamW step must end in the same
codes and block constants bit for bit, and the drift measured from them
must be the same number.
"""
import math

import numpy as np
import pytest

from gpu_util import gpu_available
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]


@pytest.fixture(scope="module")
def probes():
    from paper_2608_22322_gb300 import probes
    return probes


@pytest.mark.parametrize("regime", ["narrow", "medium", "wide"])
def test_single_step_update_error_below_one_percent(probes, regime):
    e8 = probes.single_step_update_error(regime, 2048, 8, n=1 << 20)
    e16 = probes.single_step_update_error(regime, 2048, 16, n=1 << 20)
    assert e8 < 0.01, e8
    assert e16 < e8 / 50, (e16, e8)


def test_ema_drift_5k_steps_rises_with_block_size(probes):
    res = {b: probes.ema_drift(5000, b, 8, n=1 << 18) for b in (256, 512, 1024, 2048)}
    d = [res[b][0] for b in (256, 512, 1024, 2048)]
    u = [res[b][1] for b in (256, 512, 1024, 2048)]
    print("5K-step EMA drift by block size:", ", ".join(f"{x:.3%}" for x in d),
          "update error:", ", ".join(f"{x:.3%}" for x in u))
    assert all(a < b for a, b in zip(d, d[1:])), d
    assert d[-1] < 0.01 and u[-1] < 0.01, (d, u)
    assert u[0] < u[-1] and all(x < y for x, y in zip(u, d)), (u, d)


@pytest.mark.parametrize("block", [256, 2048])
def test_ema_drift_matches_oracle(probes, block):
    """5000 steps of one gradient sequence (per-block lognormal scales, 2%
    exact zeros) through the GPU probe and through the oracle's AdamW step
    with lr = 0: identical final codes and block constants, and the same V
    drift (both against a float64 EMA of the same gradients)."""
    import torch
    import oracle as ora
    n, steps, beta1, beta2, eps = 2 * 2048, 5000, 0.9, 0.999, 1e-8
    r = wl.rng(4242 + block)
    scale = np.exp2(r.normal(-12.0, 1.25, n // block)).repeat(block).astype(np.float32)
    draws = {}

    def grad_host(t):
        if t not in draws:
            draws.clear()
            g = (wl.rng(10_000 * block + t).standard_normal(n) * scale).astype(np.float32)
            g[wl.rng(20_000 * block + t).random(n) < 0.02] = 0.0
            draws[t] = g
        return draws[t]

    drift_gpu, upd_gpu, (mc, ma, vc, vm) = probes.ema_drift(
        steps, block, 8, n=n, beta1=beta1, beta2=beta2, eps=eps,
        grad_fn=lambda t: torch.from_numpy(grad_host(t)).cuda(), return_state=True)
    hp = dict(lr=0.0, beta1=beta1, beta2=beta2, eps=eps, weight_decay=0.0,
              log_floor=float(np.float32(math.log2(eps * eps))))
    p = np.zeros(n, np.float32)
    hmc, hma = np.zeros(n, np.int8), np.zeros(n // 256, np.float32)
    hvc, hvm = np.zeros(n, np.uint8), np.zeros(2 * (n // block), np.float32)
    v64 = np.zeros(n)
    for t in range(1, steps + 1):
        g = grad_host(t)
        ora.adamw_step(p, g, hmc, hma, hvc, hvm, 256, block, 8, hp, t)
        v64 = beta2 * v64 + (1.0 - beta2) * g.astype(np.float64) ** 2
    assert np.all(p == 0.0)
    for want, got in ((hmc, mc), (hma, ma), (hvc, vc), (hvm, vm)):
        assert np.array_equal(want.view(np.uint8), got.cpu().numpy().view(np.uint8))
    v_hat = ora.al_decode(hvc, hvm, block, 8).astype(np.float64)
    drift_ora = np.linalg.norm(v_hat - v64) / np.linalg.norm(v64)
    print(f"block {block}: V drift GPU probe {drift_gpu:.4%}, oracle {drift_ora:.4%}")
    assert abs(drift_gpu - drift_ora) <= 1e-6 * drift_ora
