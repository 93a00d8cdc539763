"""The allocation-free Adafactor entry point, for callers that cannot call
cudaMalloc when they step the optimizer (a framework owning all device
memory, a fixed post-start-up memory budget, a binding without allocator
access). It must give the same results as al_adafactor_step with a
caller-allocated workspace, bit for bit, call after call, and refuse
matrices whose scratch does not fit its fixed array.

Both sides start from dirty scratch, so a read of a scratch word that the
call has not written first would show: the caller's workspace is filled
with 0xFF bytes (NaN as floats) before every call, and before the compared
calls the library's fixed array is left dirty by a call on another shape.

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


def _state(rows, cols, dev, seed=3):
    import torch
    n = rows * cols
    p = torch.from_numpy(wl.param_init((rows, cols), seed).ravel()).to(dev)
    return dict(p=p,
                rc=torch.zeros(rows, dtype=torch.int16, device=dev),
                rm=torch.zeros(2 * ((rows + 127) // 128), dtype=torch.float32, device=dev),
                cc=torch.zeros(cols, dtype=torch.int16, device=dev),
                cm=torch.zeros(2 * ((cols + 127) // 128), dtype=torch.float32, device=dev),
                mc=torch.zeros(n, dtype=torch.int8, device=dev),
                ma=torch.zeros((n + 255) // 256, dtype=torch.float32, device=dev))


def _noalloc(B, s, g, rows, cols, t):
    B.al_adafactor_step_noalloc(s["p"], g, rows, cols, s["rc"], s["rm"], s["cc"], s["cm"],
                                16, 128, s["mc"], s["ma"], 256, HP, t)


def test_noalloc_adafactor_matches_workspace_version():
    import torch
    from paper_2608_22322_gb300 import binding as B
    rows, cols = 1024, 2048
    a = _state(rows, cols, "cuda")
    b = {k: v.clone() for k, v in a.items()}
    ws = torch.empty(B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols), dtype=torch.uint8,
                     device="cuda")
    assert ws.numel() <= B.al_adafactor_noalloc_capacity()
    # another shape whose scratch covers this one's and more: its partials,
    # scales and clip factor are left in the fixed array
    drows, dcols = 4096, 4096
    assert B.al_workspace_size(B.AL_OP_ADAFACTOR, drows, dcols) >= ws.numel()
    d = _state(drows, dcols, "cuda", seed=5)
    dg = torch.from_numpy(wl.lognormal_col_grad((drows, dcols), 1e-1, 0.05, 99).ravel()).cuda()
    # t = 1, 2: the entry point called twice in a row; t = 3 after another
    # dirtying call
    for t in (1, 2, 3):
        g = torch.from_numpy(wl.lognormal_col_grad((rows, cols), 1e-3, 0.05, 60 + t).ravel()).cuda()
        if t != 2:
            _noalloc(B, d, dg, drows, dcols, t)
        ws.fill_(0xFF)
        B.al_adafactor_step(a["p"], g, rows, cols, a["rc"], a["rm"], a["cc"], a["cm"], 16, 128,
                            a["mc"], a["ma"], 256, HP, t, ws)
        _noalloc(B, b, g, rows, cols, t)
        torch.cuda.synchronize()
        for k in ("p", "rc", "rm", "cc", "cm", "mc", "ma"):
            assert torch.equal(a[k].view(torch.uint8), b[k].view(torch.uint8)), (t, k)
        assert torch.isfinite(a["p"]).all()


def test_noalloc_rejects_matrices_beyond_its_scratch():
    import torch
    from paper_2608_22322_gb300 import binding as B
    rows, cols = 8192, 8192
    assert B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols) > B.al_adafactor_noalloc_capacity()
    x = torch.zeros(16, device="cuda")
    c = torch.zeros(16, dtype=torch.int16, device="cuda")
    with pytest.raises(B.AlqError, match="WORKSPACE"):
        B.al_adafactor_step_noalloc(x, x, rows, cols, c, x, c, x, 16, 128, None, None, 256, HP, 1)
