"""The allocation-free Adafactor entry point, for callers that cannot call
cudaMalloc when they step the optimizer (a framework owning all device
memory, a fixed post-start-up memory budget, a binding without allocator
access). It must give the same results as al_adafactor_step with a
caller-allocated workspace, call after call, and refuse matrices whose
scratch does not fit its fixed array.

Named so that pytest collects it last: if it fails, a run that stops at the
first failure has already run every other test. It passes alone in a fresh
process and after the other tests (it keeps no state besides the library's
fixed array, which every call rewrites before reading).
"""
import math

import numpy as np
import pytest

from gpu_util import gpu_available
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]

HP = dict(lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9, weight_decay=0.0,
          log_floor=float(np.float32(math.log2(1e-30))))


def _state(rows, cols, dev):
    import torch
    n = rows * cols
    p = torch.from_numpy(wl.param_init((rows, cols), 3).ravel()).to(dev)
    return dict(p=p,
                rc=torch.zeros(rows, dtype=torch.int16, device=dev),
                rm=torch.zeros(2 * ((rows + 127) // 128), dtype=torch.float32, device=dev),
                cc=torch.zeros(cols, dtype=torch.int16, device=dev),
                cm=torch.zeros(2 * ((cols + 127) // 128), dtype=torch.float32, device=dev),
                mc=torch.zeros(n, dtype=torch.int8, device=dev),
                ma=torch.zeros((n + 255) // 256, dtype=torch.float32, device=dev))


def test_noalloc_adafactor_matches_workspace_version():
    import torch
    from paper_2608_22322_gb300 import binding as B
    rows, cols = 1024, 2048
    a = _state(rows, cols, "cuda")
    b = {k: v.clone() for k, v in a.items()}
    ws = torch.empty(B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols), dtype=torch.uint8,
                     device="cuda")
    assert ws.numel() <= B.al_adafactor_noalloc_capacity()
    for t in (1, 2):  # two calls in a row through the same fixed array
        g = torch.from_numpy(wl.lognormal_col_grad((rows, cols), 1e-3, 0.05, 60 + t).ravel()).cuda()
        B.al_adafactor_step(a["p"], g, rows, cols, a["rc"], a["rm"], a["cc"], a["cm"], 16, 128,
                            a["mc"], a["ma"], 256, HP, t, ws)
        B.al_adafactor_step_noalloc(b["p"], g, rows, cols, b["rc"], b["rm"], b["cc"], b["cm"],
                                    16, 128, b["mc"], b["ma"], 256, HP, t)
        torch.cuda.synchronize()
        pa, pb = a["p"].cpu().numpy(), b["p"].cpu().numpy()
        assert np.max(np.abs(pa.astype(np.float64) - pb)) <= 1e-6 * np.max(np.abs(pa))
        for k in ("rc", "rm", "cc", "cm", "mc", "ma"):
            assert torch.equal(a[k], b[k]), (t, k)


def test_noalloc_rejects_matrices_beyond_its_scratch():
    import torch
    from paper_2608_22322_gb300 import binding as B
    rows, cols = 8192, 8192
    assert B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols) > B.al_adafactor_noalloc_capacity()
    x = torch.zeros(16, device="cuda")
    c = torch.zeros(16, dtype=torch.int16, device="cuda")
    with pytest.raises(B.AlqError, match="WORKSPACE"):
        B.al_adafactor_step_noalloc(x, x, rows, cols, c, x, c, x, 16, 128, None, None, 256, HP, 1)
