"""The controlled probes of Sec. 5 on the GPU (paper_2608_22322_gb300/probes.py).
The paper does not state its generators, so these check its qualitative
claims and orderings on synthetic log-normal regimes: adaptive AL8 keeps the
single-step update error of Eq. (2) below 1% in the narrow, medium and wide
regimes at block size 2048 (Sec. 5.2); AL16 is far below AL8; over a long
second-moment EMA (beta2 = 0.999) the state drift and update error stay at
the percent level and smaller blocks drift less (Sec. 5.6)."""
import pytest

from gpu_util import gpu_available

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


def test_ema_drift_orders_by_block_size(probes):
    d256, u256 = probes.ema_drift(2000, 256, 8, n=1 << 18)
    d2048, u2048 = probes.ema_drift(2000, 2048, 8, n=1 << 18)
    assert d256 < d2048 < 0.03, (d256, d2048)
    assert u256 < 0.03 and u2048 < 0.03, (u256, u2048)
