"""Pins of the oracle's optimizer steps (fp32-state forms and quantized forms).

Each fp32-state optimizer is compared with an independent implementation or a
closed form the mathematics fixes:
  AdamW      torch.optim.AdamW in float64 over 10 steps; the t = 1 closed form
             p1 = p0 (1 - lr wd) - lr g / (|g| + eps).
  Adafactor  torch.optim.Adafactor's update direction (it scales by its own
             relative step size alpha_t, which the test divides out); the
             rank-1 closed form u = sign(g).
  CAME       rank-1 closed forms at t = 1 and t = 2; with beta1 = 0 the
             clipped update equals torch Adafactor's at t = 1 (non-square G,
             which pins the row/column orientation).
  APOLLO     with an identity projection the projected moments are Adam's:
             torch.optim.Adam gives Rt; with an orthogonal Hadamard projection
             the channel norms are preserved; rows > cols equals the
             transposed problem.
The quantized forms are checked for the exact-zero/dormant behaviour and for
tracking their fp32 forms within the quantization error (Eq. (2)).
"""
import math

import numpy as np
import pytest
import torch

import oracle as ora
from paper_2608_22322_gb300 import workloads as wl

FLOOR = float(np.float32(math.log2(1e-16)))
ADAMW_HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01,
                log_floor=FLOOR)


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


# =================================================================== AdamW ==
def test_fp32_adamw_matches_torch_adamw():
    w = wl.AdamWSingle(shape=(64, 512))
    p = w.p0.ravel().copy()
    m = np.zeros_like(p)
    v = np.zeros_like(p)
    tp = torch.tensor(w.p0.ravel(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([tp], lr=1e-3, betas=(0.9, 0.999), eps=1e-8,
                            weight_decay=0.01, foreach=False)
    p0 = p.copy()
    for t in range(1, 11):
        g = w.grad(t).ravel()
        ora.adamw_update_fp32(p, g, m, v, ADAMW_HP, t)
        tp.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
    ref = tp.detach().numpy()
    assert _rel(p - p0, ref - p0) < 1e-5


def test_fp32_adamw_first_step_closed_form():
    w = wl.AdamWSingle(shape=(32, 256))
    p = w.p0.ravel().copy()
    g = w.grad(1).ravel()
    m = np.zeros_like(p)
    v = np.zeros_like(p)
    ora.adamw_update_fp32(p, g, m, v, ADAMW_HP, 1)
    g64 = g.astype(np.float64)
    want = (w.p0.ravel().astype(np.float64) * (1 - 1e-3 * 0.01)
            - 1e-3 * g64 / (np.abs(g64) + 1e-8))
    d = p.astype(np.float64) - w.p0.ravel()
    assert _rel(d, want - w.p0.ravel()) < 1e-6


@pytest.mark.parametrize("v_bits", [8, 16])
def test_quantized_adamw_dormant_and_tracking(v_bits):
    """Dormant rows keep zero codes and only decay; the quantized step tracks
    the fp32-state step within the quantization error."""
    w = wl.AdamWSingle(shape=(64, 1024))
    n = w.p0.size
    p = w.p0.ravel().copy()
    mc = np.zeros(n, np.int8)
    ma = np.zeros(n // 256, np.float32)
    vc = np.zeros(n, ora.code_dtype(v_bits))
    vm = np.zeros(2 * (n // 256), np.float32)
    pf = w.p0.ravel().copy()
    mf = np.zeros(n, np.float32)
    vf = np.zeros(n, np.float32)
    decay = np.float32(1.0 - 1e-3 * 0.01)
    pd = w.p0.copy()
    for t in range(1, 11):
        g = w.grad(t).ravel()
        ora.adamw_step(p, g, mc, ma, vc, vm, 256, 256, v_bits, ADAMW_HP, t)
        ora.adamw_update_fp32(pf, g, mf, vf, ADAMW_HP, t)
        pd = (pd * decay).astype(np.float32)
    rows = w.dormant
    np.testing.assert_array_equal(mc.reshape(w.shape)[rows], 0)
    np.testing.assert_array_equal(vc.reshape(w.shape)[rows], 0)
    np.testing.assert_array_equal(p.reshape(w.shape)[rows], pd[rows])
    np.testing.assert_array_equal(vc == 0, vf == 0)
    # displacement error (Eq. (2) on the accumulated update)
    assert ora.update_error(p - w.p0.ravel(), pf - w.p0.ravel()) < 0.03


# =============================================================== Adafactor ==
def _torch_adafactor_steps(G_list, p0, lr, decay_rate, d, eps2=1e-3):
    """Run torch.optim.Adafactor (float64) and return the per-step update
    direction u_hat_t = -(p_t - p_{t-1}) / alpha_t."""
    tp = torch.tensor(p0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.Adafactor([tp], lr=lr, beta2_decay=decay_rate,
                                eps=(1e-30, eps2), d=d, weight_decay=0.0,
                                foreach=False)
    dirs = []
    for t, G in enumerate(G_list, start=1):
        before = tp.detach().clone()
        rms_p = float(before.norm()) / math.sqrt(before.numel())
        alpha = max(eps2, rms_p) * min(lr, 1.0 / math.sqrt(t))
        tp.grad = torch.tensor(G, dtype=torch.float64)
        opt.step()
        dirs.append(-(tp.detach() - before).numpy() / alpha)
    return dirs


def test_fp32_adafactor_direction_matches_torch():
    rows, cols = 48, 80
    hp = dict(lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9,
              weight_decay=0.0, log_floor=float(np.float32(math.log2(1e-30))))
    Gs = [wl.lognormal_col_grad((rows, cols), 1e-3, 0.05, 300 + t) for t in range(6)]
    p0 = wl.param_init((rows, cols), 9)
    ref = _torch_adafactor_steps(Gs, p0, 1e-3, -0.8, 1.0)
    p = p0.ravel().copy()
    R = np.zeros(rows, np.float32)
    Cc = np.zeros(cols, np.float32)
    for t, G in enumerate(Gs, start=1):
        before = p.copy()
        ora.adafactor_update_fp32(p, G.ravel(), rows, cols, R, Cc, None, hp, t)
        mine = -(p.astype(np.float64) - before) / hp["lr"]
        assert _rel(mine, ref[t - 1].ravel()) < 2e-5, t


def test_fp32_adafactor_rank1_closed_form():
    """G = a b^T: the factored V_hat is exact, u = sign(g), RMS(u) = 1."""
    rows, cols = 24, 40
    r = wl.rng(17)
    a = np.exp(r.standard_normal(rows)) * 1e-3
    b = np.exp(r.standard_normal(cols)) * np.sign(r.standard_normal(cols))
    G = np.outer(a, b).astype(np.float32)
    hp = dict(lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9,
              weight_decay=0.0, log_floor=-99.0)
    p = np.zeros(rows * cols, np.float32)
    R = np.zeros(rows, np.float32)
    Cc = np.zeros(cols, np.float32)
    M = np.zeros(rows * cols, np.float32)
    for t in (1, 2):
        before = p.copy()
        ora.adafactor_update_fp32(p, G.ravel(), rows, cols, R, Cc, M, hp, t)
        step = -(p.astype(np.float64) - before) / hp["lr"]
        m_want = (1 - 0.9 ** t) * np.sign(G.ravel())  # momentum of sign(g)
        assert np.max(np.abs(step - m_want)) < 1e-5, t


# ==================================================================== CAME ==
CAME_HP = dict(lr=1e-4, beta1=0.9, beta2=0.999, beta3=0.9999, eps1=1e-30,
               eps2=1e-16, clip_d=1.0, weight_decay=0.0, log_floor_v=-99.0,
               log_floor_c=-53.0)


def _came_fp32_run(G_list, hp, rows, cols):
    p = np.zeros(rows * cols, np.float32)
    st = [np.zeros(rows, np.float32), np.zeros(cols, np.float32),
          np.zeros(rows, np.float32), np.zeros(cols, np.float32),
          np.zeros(rows * cols, np.float32)]
    steps = []
    for t, G in enumerate(G_list, start=1):
        before = p.copy()
        ora.came_update_fp32(p, G.ravel(), rows, cols, *st, hp, t)
        steps.append(-(p.astype(np.float64) - before) / hp["lr"])
    return steps, st


def test_fp32_came_rank1_closed_forms():
    rows, cols = 20, 36
    r = wl.rng(23)
    a = np.exp(r.standard_normal(rows)) * 1e-3
    b = np.exp(r.standard_normal(cols)) * np.sign(r.standard_normal(cols))
    G = np.outer(a, b).astype(np.float32)
    steps, _ = _came_fp32_run([G, G], CAME_HP, rows, cols)
    sg = np.sign(G.ravel())
    b1, b3, e2 = 0.9, 0.9999, 1e-16
    # t = 1: u_hat = sign(g) after clipping; m = (1-b1) u_hat;
    # residual (u_hat - m)^2 + eps2 = b1^2 + eps2 everywhere; S = (1-b3) b1^2
    m1 = (1 - b1)
    c1 = (1 - b3) * (b1 ** 2 + e2)
    assert np.max(np.abs(steps[0] - sg * m1 / math.sqrt(c1))) < 1e-3 * m1 / math.sqrt(c1)
    # t = 2 with the same G: m = b1 m1 + (1-b1); C = b3 c1 + (1-b3)(1-m)^2
    m2 = b1 * m1 + (1 - b1)
    c2 = b3 * c1 + (1 - b3) * ((1 - m2) ** 2 + e2)
    assert np.max(np.abs(steps[1] - sg * m2 / math.sqrt(c2))) < 1e-3 * m2 / math.sqrt(c2)


def test_fp32_came_beta1_zero_equals_clipped_adafactor():
    """beta1 = 0: m = u_hat, the residual is eps2 everywhere, S = (1-b3) eps2
    and the step is u_hat / sqrt(S), with u_hat the RMS-normalised factored
    update that torch Adafactor computes at t = 1."""
    rows, cols = 30, 52
    G = wl.student_t_grad((rows, cols), 1e-3, 3.0, 0.05, 41)
    hp = dict(CAME_HP, beta1=0.0, eps2=1e-2)
    steps, _ = _came_fp32_run([G], hp, rows, cols)
    # the hyperparameters are fp32 (1 - 0.9999f = 1.00017e-4)
    S = (1 - float(np.float32(hp["beta3"]))) * float(np.float32(hp["eps2"]))
    uhat = steps[0] * math.sqrt(S)
    # CAME's u is Adafactor's u / sqrt(1 - beta2) (RMS >> 1), so its clipped
    # update is the RMS-normalised direction of torch Adafactor's update
    ref = _torch_adafactor_steps([G], wl.param_init((rows, cols), 3), 1e-3,
                                 -0.8, 1.0)[0].ravel()
    ref = ref / np.sqrt(np.mean(ref ** 2))
    assert _rel(uhat, ref) < 2e-5


# ================================================================== APOLLO ==
APOLLO_HP = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0,
                 weight_decay=0.0, norm_growth_gamma=0.0, log_floor=FLOOR)


def _bf16_exact(x):
    return wl.bf16_bits(x).astype(np.uint32).__lshift__(16).view(np.float32)


def test_fp32_apollo_identity_projection_is_adam():
    """rank = rows (short side), P = I: Rt is torch Adam's direction on R."""
    rows, cols, T = 16, 40, 5
    hp = dict(APOLLO_HP, rank=rows)
    P = wl.bf16_bits(np.eye(rows, dtype=np.float32))
    p = np.zeros(rows * cols, np.float32)
    MP = np.zeros(cols * rows, np.float32)
    VP = np.zeros(cols * rows, np.float32)
    x = torch.zeros(cols, rows, dtype=torch.float64, requires_grad=True)
    adam = torch.optim.Adam([x], lr=1.0, betas=(0.9, 0.999), eps=1e-8,
                            foreach=False)
    for t in range(1, T + 1):
        G = _bf16_exact(wl.gaussian_grad((rows, cols), 1e-3, 500 + t))
        Rm = G.T.astype(np.float64)  # channel-major [cols][rows]
        before = p.copy()
        s, _ = ora.apollo_update_fp32(p, G.ravel(), rows, cols, P, MP, VP, 0.0, hp, t)
        xb = x.detach().clone()
        x.grad = torch.tensor(Rm)
        adam.step()
        Rt = -(x.detach() - xb).numpy()
        s_ref = np.linalg.norm(Rt, axis=1) / (np.linalg.norm(Rm, axis=1) + 1e-8)
        assert _rel(s, s_ref) < 1e-5, t
        step = -(p.astype(np.float64) - before) / hp["lr"]
        assert _rel(step, (G * s_ref[None, :]).ravel()) < 1e-5, t


def _hadamard(k):
    H = np.array([[1.0]])
    while H.shape[0] < k:
        H = np.block([[H, H], [H, -H]])
    return H


def test_fp32_apollo_orthogonal_projection_first_step():
    """Orthogonal P = H/4 (16x16, exact in bf16): R = P G keeps every channel
    norm; at t = 1, Rt = R / (|R| + eps) after bias correction."""
    rows, cols = 16, 24
    hp = dict(APOLLO_HP, rank=rows)
    Pf = (_hadamard(rows) / 4.0).astype(np.float32)
    P = wl.bf16_bits(Pf)
    G = (wl.rng(8).integers(-64, 64, (rows, cols)) * 2.0 ** -14).astype(np.float32)
    R = (Pf.astype(np.float64) @ G.astype(np.float64)).T  # exact
    G64 = G.astype(np.float64)
    np.testing.assert_allclose(np.linalg.norm(R, axis=1),
                               np.linalg.norm(G64, axis=0), rtol=1e-12)
    p = np.zeros(rows * cols, np.float32)
    s, _ = ora.apollo_update_fp32(p, G.ravel(), rows, cols, P,
                                  np.zeros(rows * cols, np.float32),
                                  np.zeros(rows * cols, np.float32), 0.0, hp, 1)
    Rt = R / (np.abs(R) + 1e-8)
    s_ref = np.linalg.norm(Rt, axis=1) / (np.linalg.norm(G64, axis=0) + 1e-8)
    assert _rel(s, s_ref) < 1e-5


def test_fp32_apollo_transpose_symmetry():
    """rows > cols projects the columns; it equals the transposed problem."""
    short, long_, rank = 24, 56, 8
    hp = dict(APOLLO_HP, rank=rank)
    P = wl.bf16_bits(wl.gaussian_projection(rank, short, 6))
    G = wl.gaussian_grad((long_, short), 1e-3, 60)
    res = []
    for Gm, (r_, c_) in ((G, (long_, short)), (np.ascontiguousarray(G.T), (short, long_))):
        p = np.zeros(Gm.size, np.float32)
        MP = np.zeros(long_ * rank, np.float32)
        VP = np.zeros(long_ * rank, np.float32)
        for t in (1, 2):
            s, _ = ora.apollo_update_fp32(p, Gm.ravel(), r_, c_, P, MP, VP, 0.0, hp, t)
        res.append((p.reshape(r_, c_), s))
    np.testing.assert_array_equal(res[0][0], res[1][0].T)
    np.testing.assert_array_equal(res[0][1], res[1][1])


def test_fp32_apollo_norm_growth_limiter():
    """With gamma > 0 the scaled-gradient norm grows at most by gamma."""
    rows, cols, rank = 16, 32, 8
    hp = dict(APOLLO_HP, rank=rank, norm_growth_gamma=1.01)
    P = wl.bf16_bits(wl.gaussian_projection(rank, rows, 2))
    p = np.zeros(rows * cols, np.float32)
    MP = np.zeros(cols * rank, np.float32)
    VP = np.zeros(cols * rank, np.float32)
    prev = np.float32(0.0)
    norms = []
    for t in range(1, 6):
        G = wl.gaussian_grad((rows, cols), 1e-3 * (10.0 if t == 3 else 1.0), 70 + t)
        before = p.copy()
        _, prev = ora.apollo_update_fp32(p, G.ravel(), rows, cols, P, MP, VP, prev, hp, t)
        norms.append(np.linalg.norm((p.astype(np.float64) - before) / hp["lr"]))
        assert abs(norms[-1] - float(prev)) <= 1e-5 * norms[-1]
    for a, b in zip(norms, norms[1:]):
        assert b <= 1.01 * a * (1 + 1e-5)


def test_projection_exact_small_integers():
    """With small-integer bf16-exact inputs the projection is exact, so it
    equals an integer matrix product."""
    rows, cols, rank = 12, 20, 6
    Pi = wl.rng(1).integers(-8, 8, (rank, rows)).astype(np.float32)
    Gi = wl.rng(2).integers(-8, 8, (rows, cols)).astype(np.float32)
    R = ora.apollo_project(Gi.ravel(), rows, cols, wl.bf16_bits(Pi), rank)
    want = (Pi.astype(np.int64) @ Gi.astype(np.int64)).T.ravel()
    np.testing.assert_array_equal(R.astype(np.int64), want)


# ==================================================== quantized factored ==
def test_quantized_adafactor_and_came_track_fp32():
    rows, cols = 64, 96
    Gs = [wl.lognormal_col_grad((rows, cols), 1e-3, 0.05, 900 + t) for t in range(5)]
    hp = dict(lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9,
              weight_decay=0.0, log_floor=float(np.float32(math.log2(1e-30))))
    p = np.zeros(rows * cols, np.float32)
    pf = p.copy()
    rc = np.zeros(rows, np.uint16); rm = np.zeros(2, np.float32)
    cc = np.zeros(cols, np.uint16); cm = np.zeros(2, np.float32)
    mc = np.zeros(rows * cols, np.int8); ma = np.zeros(rows * cols // 256, np.float32)
    R = np.zeros(rows, np.float32); Cc = np.zeros(cols, np.float32)
    M = np.zeros(rows * cols, np.float32)
    for t, G in enumerate(Gs, start=1):
        ora.adafactor_step(p, G.ravel(), rows, cols, rc, rm, cc, cm, 16, 128,
                           mc, ma, 256, hp, t)
        ora.adafactor_update_fp32(pf, G.ravel(), rows, cols, R, Cc, M, hp, t)
    assert ora.update_error(p, pf) < 0.02

    hpc = dict(CAME_HP, lr=1e-3)
    p = np.zeros(rows * cols, np.float32)
    codes = [np.zeros(rows, np.uint16), np.zeros(2, np.float32),
             np.zeros(cols, np.uint16), np.zeros(2, np.float32)]
    ccodes = [np.zeros(rows, np.uint16), np.zeros(2, np.float32),
              np.zeros(cols, np.uint16), np.zeros(2, np.float32)]
    mc = np.zeros(rows * cols, np.int8); ma = np.zeros(rows * cols // 256, np.float32)
    for t, G in enumerate(Gs, start=1):
        ora.came_step(p, G.ravel(), rows, cols, *codes, 16, 128, *ccodes, 16, 128,
                      mc, ma, 256, hpc, t)
    steps, _ = _came_fp32_run(Gs, hpc, rows, cols)
    pf = -hpc["lr"] * np.sum(steps, axis=0)
    assert ora.update_error(p, pf) < 0.02


# ======================================================== FP32 state role ==
# Sec. 4.5 (state policy): a state may stay unquantized (FP32) instead of
# AL8 / AL16; with bits = 32 the steps keep it as plain fp32 values.
def test_fp32_role_adamw_step_is_torch_adamw():
    """v_bits = 32 (m and v dense fp32) through the step: torch.optim.AdamW
    (float64) over 10 steps, as the fp32 update itself."""
    w = wl.AdamWSingle(shape=(64, 512))
    p = w.p0.ravel().copy()
    m = np.zeros_like(p)
    v = np.zeros_like(p)
    tp = torch.tensor(w.p0.ravel(), dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([tp], lr=1e-3, betas=(0.9, 0.999), eps=1e-8,
                            weight_decay=0.01, foreach=False)
    p0 = p.copy()
    for t in range(1, 11):
        g = w.grad(t).ravel()
        ora.adamw_step(p, g, m, None, v, None, 256, 256, 32, ADAMW_HP, t)
        tp.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
    assert _rel(p - p0, tp.detach().numpy() - p0) < 1e-5
    assert np.any(m != 0) and np.all(v >= 0)


def test_fp32_role_adafactor_step_matches_torch():
    """fac_bits = 32 through the step (no momentum): torch.optim.Adafactor's
    update direction."""
    rows, cols = 48, 80
    hp = dict(lr=1e-3, eps1=1e-30, clip_d=1.0, decay_rate=-0.8, beta1=0.9,
              weight_decay=0.0, log_floor=float(np.float32(math.log2(1e-30))))
    Gs = [wl.lognormal_col_grad((rows, cols), 1e-3, 0.05, 300 + t) for t in range(6)]
    p0 = wl.param_init((rows, cols), 9)
    ref = _torch_adafactor_steps(Gs, p0, 1e-3, -0.8, 1.0)
    p = p0.ravel().copy()
    R = np.zeros(rows, np.float32)
    Cc = np.zeros(cols, np.float32)
    dummy = np.zeros(2, np.float32)
    for t, G in enumerate(Gs, start=1):
        before = p.copy()
        ora.adafactor_step(p, G.ravel(), rows, cols, R, dummy, Cc, dummy, 32, 128, None, None,
                           256, hp, t)
        mine = -(p.astype(np.float64) - before) / hp["lr"]
        assert _rel(mine, ref[t - 1].ravel()) < 2e-5, t
    assert np.all(R > 0) and np.all(Cc > 0)


def test_fp32_role_came_step_is_fp32_update():
    """CAME with V and C in FP32 through the step equals the fp32 update on
    plain arrays bit for bit; the paper's FP32-C variant (AL16 V, FP32 C)
    tracks it."""
    rows, cols = 40, 96
    hp = dict(lr=1e-4, beta1=0.9, beta2=0.999, beta3=0.9999, eps1=1e-30, eps2=1e-16,
              clip_d=1.0, weight_decay=0.0, log_floor_v=float(np.float32(math.log2(1e-30))),
              log_floor_c=float(np.float32(math.log2(1e-16))))
    p0 = wl.param_init((rows, cols), 13).ravel()
    pa, pb, pc = p0.copy(), p0.copy(), p0.copy()
    n = rows * cols
    fa = [np.zeros(rows, np.float32), np.zeros(cols, np.float32), np.zeros(rows, np.float32),
          np.zeros(cols, np.float32)]
    fb = [x.copy() for x in fa]
    Ma = np.zeros(n, np.float32)
    mc = np.zeros(n, np.int8)
    ma = np.zeros(n // 256 + 1, np.float32)
    mc2, ma2 = mc.copy(), ma.copy()
    dummy = np.zeros(2, np.float32)
    vr16 = np.zeros(rows, np.uint16)
    vr16m = np.zeros(2 * (rows // 128 + 1), np.float32)
    vc16 = np.zeros(cols, np.uint16)
    vc16m = np.zeros(2 * (cols // 128 + 1), np.float32)
    cr, cc = np.zeros(rows, np.float32), np.zeros(cols, np.float32)
    mc3, ma3 = mc.copy(), ma.copy()
    for t in range(1, 6):
        g = wl.student_t_grad((rows, cols), 1e-3, 3.0, 0.05, 70 + t).ravel()
        # reference: fp32 update on plain states, momentum through UF8 as in the step
        M = ora.uf8_decode(mc2, ma2, 256)
        ora.came_update_fp32(pa, g, rows, cols, *fa, M, hp, t)
        mc2, ma2 = ora.uf8_encode(M, 256)
        ora.came_step(pb, g, rows, cols, fb[0], dummy, fb[1], dummy, 32, 128, fb[2], dummy,
                      fb[3], dummy, 32, 128, mc, ma, 256, hp, t)
        ora.came_step(pc, g, rows, cols, vr16, vr16m, vc16, vc16m, 16, 128, cr, dummy, cc,
                      dummy, 32, 128, mc3, ma3, 256, hp, t)
        assert np.array_equal(pa.view(np.uint32), pb.view(np.uint32)), t
        for x, y in zip(fa, fb):
            assert np.array_equal(x.view(np.uint32), y.view(np.uint32)), t
    assert ora.update_error(pc - p0, pa - p0) < 0.03

