"""GPU parity of the Adafactor and CAME steps (AL-coded factors, UF8
momentum) with the oracle.

Sec. 3.1 (factored second moment; CAME's factored confidence), Sec. 6.1
hyperparameters, Eq. (3)-(5) for the factor codes. Same seeded states and
gradients on both sides, at the workloads' own sizes and step counts
(Adafactor 4096 x 4096 for 20 steps, CAME 2048 x 5632 for 10) and smaller
and ragged shapes. The fp32 state arithmetic is identical on both sides;
the row/column means and the RMS are sums computed to beyond double
accuracy and rounded once on both sides (two-float partials merged in fp64
on the GPU, fp64 in the oracle), so every fresh factor is the same fp32
value unless a sum lies within ~1e-16 of an fp32 rounding boundary (about
one value in 2^29). Bar, after every step: every factor code and every
block constant (l_min, Delta) of R, C (and CAME's C^(r), C^(c)), every
momentum code and block absmax bit for bit, and the parameters bit for bit
(the update is the oracle's IEEE arithmetic in the same order; measured on
every shape and step), which implies the parity bar of 1e-5 relative.
"""
import math

import numpy as np
import pytest

import oracle as ora
from gpu_util import bytes_equal, gpu_available
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]

F1 = float(np.float32(math.log2(1e-30)))
F2 = float(np.float32(math.log2(1e-16)))
ADA_HP = dict(lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9,
              weight_decay=0.0, log_floor=F1)
CAME_HP = dict(lr=1e-4, beta1=0.9, beta2=0.999, beta3=0.9999, eps1=1e-30, eps2=1e-16,
               clip_d=1.0, weight_decay=0.0, log_floor_v=F1, log_floor_c=F2)


@pytest.fixture(scope="module")
def B():
    from paper_2608_22322_gb300 import binding
    return binding


def _t(a):
    import torch
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a.copy()).cuda()


def _exact(name, want, got):
    """Bytes of a GPU array that differ from the oracle's (asserted zero)."""
    got = got.cpu().numpy()
    bad = bytes_equal(want, got)
    assert bad == 0, f"{name}: {bad} bytes differ from the oracle"
    return bad


def _cmp_p(want, got, what):
    got = got.cpu().numpy()
    err = np.max(np.abs(got.astype(np.float64) - want))
    assert err <= 1e-6 * np.max(np.abs(want)), f"{what}: max |dp| = {err}"
    return int(np.sum(want.view(np.uint32) != got.view(np.uint32)))


def _state(n, bits, block):
    nb = (n + block - 1) // block
    return np.zeros(n, ora.code_dtype(bits)), np.zeros(2 * nb, np.float32)


@pytest.mark.parametrize("rows,cols,bits,fblock,mom,steps", [
    (4096, 4096, 16, 128, True, 20),    # the Adafactor workload, its 20 steps
    (512, 1024, 16, 128, True, 20),     # the same setting, smaller matrix
    (300, 772, 16, 128, True, 6),       # ragged tiles
    (257, 2048, 8, 256, False, 6),      # AL8 factors, no momentum
])
def test_adafactor_matches_oracle(B, rows, cols, bits, fblock, mom, steps):
    import torch
    n = rows * cols
    p = wl.param_init((rows, cols), 5).ravel()
    rc, rm = _state(rows, bits, fblock)
    cc, cm = _state(cols, bits, fblock)
    mc = np.zeros(n, np.int8) if mom else None
    ma = np.zeros((n + 255) // 256, np.float32) if mom else None
    d = dict(p=_t(p), rc=_t(rc), rm=_t(rm), cc=_t(cc), cm=_t(cm),
             mc=_t(mc) if mom else None, ma=_t(ma) if mom else None)
    ws = torch.empty(B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols), dtype=torch.uint8,
                     device="cuda")
    p_inexact = 0
    for t in range(1, steps + 1):
        g = wl.lognormal_col_grad((rows, cols), 1e-3, 0.05, 7000 + t).ravel()
        ora.adafactor_step(p, g, rows, cols, rc, rm, cc, cm, bits, fblock, mc, ma, 256,
                           ADA_HP, t)
        B.al_adafactor_step(d["p"], _t(g), rows, cols, d["rc"], d["rm"], d["cc"], d["cm"],
                            bits, fblock, d["mc"], d["ma"], 256, ADA_HP, t, ws)
        torch.cuda.synchronize()
        p_inexact = _cmp_p(p, d["p"], f"step {t}")
        for name, want, key in (("R codes", rc, "rc"), ("R l_min/Delta", rm, "rm"),
                                ("C codes", cc, "cc"), ("C l_min/Delta", cm, "cm")) + (
                (("M codes", mc, "mc"), ("M absmax", ma, "ma")) if mom else ()):
            _exact(f"step {t} {name}", want, d[key])
    print(f"adafactor {rows}x{cols}, {steps} steps: codes, block constants and parameters "
          f"exact ({p_inexact} of {n} parameters differ)")
    assert p_inexact == 0


@pytest.mark.parametrize("rows,cols,steps,bits,fblock", [
    (2048, 5632, 10, 16, 128),  # one matrix of the CAME workload, its 10 steps
    (256, 1408, 10, 16, 128), (130, 516, 5, 16, 128),
    (512, 4096, 6, 8, 2048),  # the paper's all-AL8 CAME variant (Sec. 6.2 table, B = 2048)
])
def test_came_matches_oracle(B, rows, cols, steps, bits, fblock):
    import torch
    n = rows * cols
    p = wl.param_init((rows, cols), 8).ravel()
    st = [_state(rows, bits, fblock), _state(cols, bits, fblock), _state(rows, bits, fblock),
          _state(cols, bits, fblock)]
    mc = np.zeros(n, np.int8)
    ma = np.zeros((n + 255) // 256, np.float32)
    dp = _t(p)
    dst = [(_t(c), _t(m)) for c, m in st]
    dmc, dma = _t(mc), _t(ma)
    ws = torch.empty(B.al_workspace_size(B.AL_OP_CAME, rows, cols), dtype=torch.uint8,
                     device="cuda")
    p_inexact = 0
    for t in range(1, steps + 1):
        g = wl.student_t_grad((rows, cols), 1e-3, 3.0, 0.05, 8000 + t).ravel()
        ora.came_step(p, g, rows, cols, st[0][0], st[0][1], st[1][0], st[1][1], bits, fblock,
                      st[2][0], st[2][1], st[3][0], st[3][1], bits, fblock, mc, ma, 256, CAME_HP, t)
        B.al_came_step(dp, _t(g), rows, cols, dst[0][0], dst[0][1], dst[1][0], dst[1][1], bits,
                       fblock, dst[2][0], dst[2][1], dst[3][0], dst[3][1], bits, fblock, dmc, dma,
                       256, CAME_HP, t, ws)
        torch.cuda.synchronize()
        p_inexact = _cmp_p(p, dp, f"step {t}")
        for name, (c, m), (dc, dm) in zip(("V^(r)", "V^(c)", "C^(r)", "C^(c)"), st, dst):
            _exact(f"step {t} {name} codes", c, dc)
            _exact(f"step {t} {name} l_min/Delta", m, dm)
        _exact(f"step {t} M codes", mc, dmc)
        _exact(f"step {t} M absmax", ma, dma)
    print(f"came {rows}x{cols}, {steps} steps: codes, block constants and parameters "
          f"exact ({p_inexact} of {n} parameters differ)")
    assert p_inexact == 0


def test_factored_rejects_bad_arguments(B):
    import torch
    x = torch.zeros(64 * 64, device="cuda")
    c = torch.zeros(64, dtype=torch.int16, device="cuda")
    m = torch.zeros(2, device="cuda")
    ws = torch.empty(B.al_workspace_size(B.AL_OP_ADAFACTOR, 64, 64), dtype=torch.uint8,
                     device="cuda")
    with pytest.raises(B.AlqError, match="UNSUPPORTED"):   # cols not a multiple of 4
        B.al_adafactor_step(x, x, 64, 62, c, m, c, m, 16, 128, None, None, 256, ADA_HP, 1, ws)
    with pytest.raises(B.AlqError, match="WORKSPACE"):
        B.al_adafactor_step(x, x, 64, 64, c, m, c, m, 16, 128, None, None, 256, ADA_HP, 1,
                            ws[:16])


def _fac_states(rows, cols, bits, block, came, seed):
    """Zero factored states of one matrix (numpy), with its parameters."""
    n = rows * cols
    st = dict(p=wl.param_init((rows, cols), seed).ravel())
    for k, ln in (("vr", rows), ("vc", cols)) + ((("cr", rows), ("cc", cols)) if came else ()):
        c, m = _state(ln, bits, block)
        st[k + "_codes"], st[k + "_meta"] = c, m
    st["m_codes"] = np.zeros(n, np.int8)
    st["m_absmax"] = np.zeros((n + 255) // 256, np.float32)
    return st


@pytest.mark.parametrize("op,mom,bits,block", [("adafactor", True, 16, 128),
                                               ("adafactor", False, 8, 256),
                                               ("came", True, 16, 128),
                                               ("came", True, 8, 2048)])
def test_grouped_factored_step_matches_single(B, op, mom, bits, block):
    """The grouped step (one launch per pass over all matrices) gives every
    matrix exactly the per-matrix step's parameters, codes and metadata."""
    import torch
    came = op == "came"
    shapes = [(300, 772), (64, 512), (512, 1024), (130, 516), (257, 2048)]
    single = [_fac_states(r, c, bits, block, came, 40 + i) for i, (r, c) in enumerate(shapes)]
    dg = [{k: _t(v) for k, v in s_.items()} for s_ in single]
    ds = [{k: _t(v) for k, v in s_.items()} for s_ in single]
    grads = [torch.zeros(r * c, dtype=torch.float32, device="cuda") for r, c in shapes]
    mats = []
    for (r, c), d, g in zip(shapes, dg, grads):
        m = dict(p=d["p"], g=g, rows=r, cols=c, vr_codes=d["vr_codes"], vr_meta=d["vr_meta"],
                 vc_codes=d["vc_codes"], vc_meta=d["vc_meta"])
        if came:
            m.update(cr_codes=d["cr_codes"], cr_meta=d["cr_meta"], cc_codes=d["cc_codes"],
                     cc_meta=d["cc_meta"])
        if mom:
            m.update(m_codes=d["m_codes"], m_absmax=d["m_absmax"])
        mats.append(m)
    plan = B.FactoredPlan(B.AL_OP_CAME if came else B.AL_OP_ADAFACTOR, mats, bits, block, bits,
                          block, 256)
    assert plan.info.nmat == len(shapes) and plan.info.has_momentum == int(mom)
    wss = [torch.empty(B.al_workspace_size(B.AL_OP_CAME if came else B.AL_OP_ADAFACTOR, r, c),
                       dtype=torch.uint8, device="cuda") for r, c in shapes]
    for t in range(1, 4):
        for i, (r, c) in enumerate(shapes):
            grads[i].copy_(torch.from_numpy(
                wl.student_t_grad((r, c), 1e-3, 3.0, 0.05, 900 + 10 * t + i).ravel()))
        if came:
            plan.step(CAME_HP, t)
        else:
            plan.step(ADA_HP, t)
        for i, (r, c) in enumerate(shapes):
            d = ds[i]
            if came:
                B.al_came_step(d["p"], grads[i], r, c, d["vr_codes"], d["vr_meta"], d["vc_codes"],
                               d["vc_meta"], bits, block, d["cr_codes"], d["cr_meta"],
                               d["cc_codes"], d["cc_meta"], bits, block, d["m_codes"],
                               d["m_absmax"], 256, CAME_HP, t, wss[i])
            else:
                B.al_adafactor_step(d["p"], grads[i], r, c, d["vr_codes"], d["vr_meta"],
                                    d["vc_codes"], d["vc_meta"], bits, block,
                                    d["m_codes"] if mom else None,
                                    d["m_absmax"] if mom else None, 256, ADA_HP, t, wss[i])
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            for k in dg[i]:
                if not mom and k.startswith("m_"):
                    continue
                a = dg[i][k].cpu().numpy()
                b = ds[i][k].cpu().numpy()
                assert bytes_equal(a, b) == 0, (op, t, i, k)


def test_came_per_matrix_steps_on_streams_match_sequence(B):
    """Per-matrix CAME steps dealt over several streams (the benchmark's
    schedule: each matrix with its own workspace, the passes of different
    matrices running concurrently) give every matrix exactly the
    parameters, codes and metadata of the same steps run one after another
    on one stream."""
    import torch
    shapes = [(300, 772), (64, 512), (512, 1024), (130, 516), (257, 2048)]
    seq = [_fac_states(r, c, 16, 128, True, 60 + i) for i, (r, c) in enumerate(shapes)]
    da = [{k: _t(v) for k, v in s_.items()} for s_ in seq]
    db = [{k: _t(v) for k, v in s_.items()} for s_ in seq]
    grads = [torch.zeros(r * c, dtype=torch.float32, device="cuda") for r, c in shapes]

    def ws():
        return [torch.empty(B.al_workspace_size(B.AL_OP_CAME, r, c), dtype=torch.uint8,
                            device="cuda") for r, c in shapes]

    wa, wb = ws(), ws()
    streams = [torch.cuda.Stream() for _ in range(3)]

    def step(d, i, t, w, stream):
        r, c = shapes[i]
        B.al_came_step(d["p"], grads[i], r, c, d["vr_codes"], d["vr_meta"], d["vc_codes"],
                       d["vc_meta"], 16, 128, d["cr_codes"], d["cr_meta"], d["cc_codes"],
                       d["cc_meta"], 16, 128, d["m_codes"], d["m_absmax"], 256, CAME_HP, t,
                       w, stream=stream)

    for t in range(1, 4):
        for i, (r, c) in enumerate(shapes):
            grads[i].copy_(torch.from_numpy(
                wl.student_t_grad((r, c), 1e-3, 3.0, 0.05, 700 + 10 * t + i).ravel()))
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            step(da[i], i, t, wa[i], torch.cuda.current_stream())
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            step(db[i], i, t, wb[i], streams[i % len(streams)])
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            for k in da[i]:
                assert bytes_equal(da[i][k].cpu().numpy(), db[i][k].cpu().numpy()) == 0, (t, i, k)


@pytest.mark.parametrize("op,vb,cb", [("adafactor", 32, 0), ("came", 16, 32), ("came", 32, 32)])
def test_fp32_factor_roles_match_oracle(B, op, vb, cb):
    """Factors kept unquantized (bits 32, Sec. 4.5): Adafactor with fp32
    factors, the paper's FP32-C CAME (AL16 V, fp32 C) and CAME with fp32 V
    and C, against the oracle; and the grouped step equals the per-matrix
    step bit for bit."""
    import torch
    rows, cols = 300, 772
    came = op == "came"

    def fac(ln, bits):
        if bits == 32:
            return np.zeros(ln, np.float32), None
        return _state(ln, bits, 128)

    p = wl.param_init((rows, cols), 17).ravel()
    st = [fac(rows, vb), fac(cols, vb)] + ([fac(rows, cb), fac(cols, cb)] if came else [])
    n = rows * cols
    mc = np.zeros(n, np.int8)
    ma = np.zeros((n + 255) // 256, np.float32)
    dt = lambda a: None if a is None else _t(a)
    d1 = dict(p=_t(p), st=[(dt(c), dt(m)) for c, m in st], mc=_t(mc), ma=_t(ma))
    d2 = dict(p=_t(p), st=[(dt(c), dt(m)) for c, m in st], mc=_t(mc), ma=_t(ma))
    g_dev = torch.zeros(n, dtype=torch.float32, device="cuda")
    keys = ["vr", "vc", "cr", "cc"]
    m = dict(p=d2["p"], g=g_dev, rows=rows, cols=cols, m_codes=d2["mc"], m_absmax=d2["ma"])
    for k, (c, me) in zip(keys, d2["st"]):
        m[k + "_codes"], m[k + "_meta"] = c, me
    plan = B.FactoredPlan(B.AL_OP_CAME if came else B.AL_OP_ADAFACTOR, [m], vb, 128,
                          cb if came else 16, 128, 256)
    ws = torch.empty(B.al_workspace_size(B.AL_OP_CAME if came else B.AL_OP_ADAFACTOR, rows, cols),
                     dtype=torch.uint8, device="cuda")
    flips = 0
    for t in range(1, 5):
        g = wl.student_t_grad((rows, cols), 1e-3, 3.0, 0.05, 4400 + t).ravel()
        g_dev.copy_(torch.from_numpy(g))
        dummy = np.zeros(2, np.float32)
        hm = lambda x: dummy if x is None else x
        if came:
            ora.came_step(p, g, rows, cols, st[0][0], hm(st[0][1]), st[1][0], hm(st[1][1]), vb,
                          128, st[2][0], hm(st[2][1]), st[3][0], hm(st[3][1]), cb, 128, mc, ma,
                          256, CAME_HP, t)
            s_ = d1["st"]
            B.al_came_step(d1["p"], g_dev, rows, cols, s_[0][0], s_[0][1], s_[1][0], s_[1][1], vb,
                           128, s_[2][0], s_[2][1], s_[3][0], s_[3][1], cb, 128, d1["mc"],
                           d1["ma"], 256, CAME_HP, t, ws)
            plan.step(CAME_HP, t)
        else:
            ora.adafactor_step(p, g, rows, cols, st[0][0], hm(st[0][1]), st[1][0], hm(st[1][1]),
                               32, 128, mc, ma, 256, ADA_HP, t)
            s_ = d1["st"]
            B.al_adafactor_step(d1["p"], g_dev, rows, cols, s_[0][0], s_[0][1], s_[1][0],
                                s_[1][1], 32, 128, d1["mc"], d1["ma"], 256, ADA_HP, t, ws)
            plan.step(ADA_HP, t)
        torch.cuda.synchronize()
        _cmp_p(p, d1["p"], f"step {t}")
        for (c, _), (dc, _), bits in zip(st, d1["st"], [vb, vb, cb, cb]):
            if bits == 32:
                got = dc.cpu().numpy()
                assert np.max(np.abs(got - c) / np.maximum(np.abs(c), 1e-38)) < 1e-5
            else:
                flips += _exact("factor codes", c, dc)
        flips += _exact("M codes", mc, d1["mc"])
        for a, b in zip([d1["p"], d1["mc"], d1["ma"]] + [x for x, _ in d1["st"]],
                        [d2["p"], d2["mc"], d2["ma"]] + [x for x, _ in d2["st"]]):
            assert bytes_equal(a.cpu().numpy(), b.cpu().numpy()) == 0, t
    print(f"{op} v{vb} c{cb}: codes exact ({flips} bytes differ)")
