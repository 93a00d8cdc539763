"""GPU parity of the APOLLO step (tcgen05 projection, UF8 M^P, AL8 V^P,
channel-wise scale) with the oracle.

Sec. 3.1 (projected moments give a channel-wise scale of the original
gradient), Sec. 6.1 (rank 256, channel-wise), at the TinyLlama matrix
shapes (2048 x 2048, 5632 x 2048, 2048 x 5632, 256 x 2048) and smaller,
ragged ones. The projection R = P bf16(G) runs on the tensor cores with
fp32 accumulation, so it is not bit-exact: the test bounds it against the
double-precision product of the same bf16 operands (the oracle's
projection) at 1e-5 of each channel's norm. Everything after the
projection follows the oracle's arithmetic exactly, except the
bias-corrected ratio M/(sqrt(V) + eps) behind the channel scales, which
takes the approximate square root and reciprocal (it moves p only): fed the
GPU's own R (teacher-forced), the oracle must reproduce the projected-moment
codes and their block constants bit for bit, and the parameters within 1e-5
of |p| plus the step size.
Free-running, the two trajectories see different R (fp32 against double
accumulation), and each channel's AL block starts at its smallest R^2,
whose relative error is the largest: block constants shift, codes move by
a level, and the difference in the parameters' displacement is bounded by
the codec's own error. Bar: the displacement (p_t - p_0) within 1e-4
relative of the oracle's after 10 steps (the AL8 codec's displacement
error against fp32 states is ~6e-4 at these ranks), parameters within 1e-5
relative; code and constant differences are reported.
"""
import math

import numpy as np
import pytest

import oracle as ora
from gpu_util import gpu_available, params_off, step_size
from paper_2608_22322_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not gpu_available(), reason="needs a CUDA GPU")]

FLOOR = float(np.float32(math.log2(1e-16)))
HP = dict(lr=1e-4, beta1=0.9, beta2=0.999, eps=1e-8, alpha=1.0, weight_decay=0.0,
          norm_growth_gamma=0.0, log_floor=FLOOR, rank=256)


@pytest.fixture(scope="module")
def B():
    from paper_2608_22322_gb300 import binding
    return binding


def _t(a):
    import torch
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(np.ascontiguousarray(a).copy()).cuda()


def _r256(x):
    return (x + 255) & ~255


class Apollo:
    def __init__(self, B, rows, cols, hp, seed):
        import torch
        self.B, self.rows, self.cols, self.hp = B, rows, cols, hp
        r = hp["rank"]
        self.s, self.L = min(rows, cols), (cols if rows <= cols else rows)
        self.P = wl.bf16_bits(wl.gaussian_projection(r, self.s, seed))
        n_p = self.L * r
        self.h = dict(p=wl.param_init((rows, cols), seed + 1).ravel(),
                      mc=np.zeros(n_p, np.int8), ma=np.zeros(n_p // r, np.float32),
                      vc=np.zeros(n_p, np.uint8), vm=np.zeros(2 * (n_p // r), np.float32))
        self.prev = np.float32(0.0)
        self.d = {k: _t(v) for k, v in self.h.items()}
        self.dP = _t(self.P)
        self.dprev = torch.zeros(1, dtype=torch.float32, device="cuda")
        self.ws = torch.zeros(B.al_workspace_size(B.AL_OP_APOLLO, rows, cols, r),
                              dtype=torch.uint8, device="cuda")

    def step(self, g, t):
        h, d, r = self.h, self.d, self.hp["rank"]
        _, self.prev = ora.apollo_step(h["p"], g, self.rows, self.cols, self.P, h["mc"], h["ma"],
                                       r, h["vc"], h["vm"], 8, r, self.prev, self.hp, t)
        self.B.al_apollo_step(d["p"], _t(g), self.rows, self.cols, self.dP, d["mc"], d["ma"], r,
                              d["vc"], d["vm"], 8, r, self.dprev, self.hp, t, self.ws)

    def device_R(self):
        import torch
        r = self.hp["rank"]
        raw = self.ws[:4 * self.L * r].clone()  # R leads the workspace
        torch.cuda.synchronize()
        return raw.view(torch.float32).cpu().numpy()


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("rows,cols", [(256, 512), (512, 256), (384, 640), (200, 332),
                                       (332, 200), (8, 8), (16, 8), (8, 36)])
def test_projection_matches_double_product(B, rows, cols):
    """The tcgen05 GEMM (G converted to bf16 inside the projection, both
    channel layouts, ragged K and channel tiles) against the double product
    of the same bf16 inputs."""
    import torch
    a = Apollo(B, rows, cols, HP, seed=11)
    g = wl.gaussian_grad((rows, cols), 1e-3, 12).ravel()
    a.step(g, 1)
    torch.cuda.synchronize()
    Rg = a.device_R().reshape(a.L, 256)
    Ro = ora.apollo_project(g, rows, cols, a.P, 256).reshape(a.L, 256)
    assert np.all(np.isfinite(Rg)), "projection pipeline reported a failure (NaN)"
    per_ch = np.linalg.norm(Ro.astype(np.float64), axis=1, keepdims=True)
    assert np.max(np.abs(Rg - Ro) / per_ch) < 1e-5
    assert _rel(Rg, Ro) < 1e-5


CONFIG5 = [(2048, 2048), (5632, 2048), (2048, 5632), (256, 2048)]


@pytest.mark.parametrize("rows,cols,steps", [(256, 1024, 6), (1024, 512, 6), (1024, 2816, 2)]
                         + [(r, c, 3) for r, c in CONFIG5])
def test_apollo_teacher_forced_exact_states(B, rows, cols, steps):
    """Each step from the GPU's own pre-step state and its own R: codes and
    metadata agree with the oracle bit for bit, parameters within 1e-5 of
    |p| plus the step size."""
    import torch
    a = Apollo(B, rows, cols, HP, seed=21)
    for t in range(1, steps + 1):
        g = wl.gaussian_grad((rows, cols), 1e-3, 300 + t).ravel()
        snap = {k: v.cpu().numpy().copy() for k, v in a.d.items()}
        p_before = snap["p"].copy()
        a.B.al_apollo_step(a.d["p"], _t(g), rows, cols, a.dP, a.d["mc"], a.d["ma"], 256,
                           a.d["vc"], a.d["vm"], 8, 256, a.dprev, a.hp, t, a.ws)
        torch.cuda.synchronize()
        R = a.device_R()
        assert np.all(np.isfinite(R)), "projection pipeline reported a failure (NaN)"
        ora.apollo_step_given_R(snap["p"], g, rows, cols, R, snap["mc"], snap["ma"], 256,
                                snap["vc"], snap["vm"], 8, 256, 0.0, a.hp, t)
        p_dev = a.d["p"].cpu().numpy()
        for k in ("mc", "ma", "vc", "vm"):
            got = a.d[k].cpu().numpy()
            bad = int(np.sum(got.view(np.uint8) != snap[k].view(np.uint8)))
            assert bad == 0, f"step {t}: {k} differs in {bad} bytes"
        bad = params_off(snap["p"], p_dev, step_size(snap["p"], p_before, a.hp))
        assert bad == 0, f"step {t}: {bad} parameters outside the tolerance"


@pytest.mark.parametrize("rows,cols,steps", [(256, 1024, 10), (1024, 512, 10)]
                         + [(r, c, 10) for r, c in CONFIG5])
def test_apollo_free_running(B, rows, cols, steps):
    import torch
    a = Apollo(B, rows, cols, HP, seed=21)
    p0 = a.h["p"].copy()
    R_err = 0.0
    for t in range(1, steps + 1):
        g = wl.gaussian_grad((rows, cols), 1e-3, 300 + t).ravel()
        a.step(g, t)
        if t == 1:
            torch.cuda.synchronize()
            Rg = a.device_R().reshape(a.L, 256)
            Ro = ora.apollo_project(g, rows, cols, a.P, 256).reshape(a.L, 256)
            per_ch = np.linalg.norm(Ro.astype(np.float64), axis=1, keepdims=True)
            R_err = float(np.max(np.abs(Rg - Ro) / per_ch))
            assert R_err < 1e-5
    torch.cuda.synchronize()
    pd = a.d["p"].cpu().numpy()
    assert _rel(pd, a.h["p"]) < 1e-5
    disp = _rel(pd - p0, a.h["p"] - p0)
    n_codes = a.L * 256
    diff = {k: int(np.sum(a.d[k].cpu().numpy().view(np.uint8) != a.h[k].view(np.uint8)))
            for k in ("mc", "vc", "vm")}
    print(f"apollo {rows}x{cols}, {steps} steps: R error {R_err:.1e} of the channel norm; "
          f"relative displacement error {disp:.2e}; differing M^P codes {diff['mc']}, "
          f"V^P codes {diff['vc']} of {n_codes}, V^P constant bytes {diff['vm']} of "
          f"{8 * a.L}")
    assert disp < 1e-4


def test_apollo_norm_growth_limiter(B):
    import torch
    hp = dict(HP, norm_growth_gamma=1.01)
    a = Apollo(B, 256, 512, hp, seed=31)
    for t in range(1, 5):
        g = wl.gaussian_grad((256, 512), 1e-3 * (10.0 if t == 3 else 1.0), 400 + t).ravel()
        a.step(g, t)
        torch.cuda.synchronize()
        assert abs(float(a.dprev.item()) - float(a.prev)) <= 1e-5 * float(a.prev)
        assert _rel(a.d["p"].cpu().numpy(), a.h["p"]) < 1e-5


# ------------------------------------------------------------ grouped step --
def _mat_state(rows, cols, rank, v_bits, seed):
    s_, L = min(rows, cols), max(rows, cols)
    P = wl.bf16_bits(wl.gaussian_projection(rank, s_, seed))
    n_p = L * rank
    vdt = np.uint8 if v_bits == 8 else np.uint16
    return dict(p=wl.param_init((rows, cols), seed + 1).ravel(), proj=P,
                m_codes=np.zeros(n_p, np.int8), m_absmax=np.zeros(n_p // rank, np.float32),
                v_codes=np.zeros(n_p, vdt), v_meta=np.zeros(2 * (n_p // rank), np.float32))


@pytest.mark.parametrize("rank,v_bits", [(128, 8), (256, 8), (256, 16)])
def test_apollo_grouped_step_matches_single(B, rank, v_bits):
    """One grouped launch sequence over matrices of mixed shape (channels
    along columns and along rows, short side below, equal to and above the
    rank, ragged 128-channel tiles) gives, matrix by matrix, bit-for-bit the
    results of al_apollo_step: parameters, projected-moment codes and block
    metadata, over three steps."""
    import torch
    shapes = [(64, 256), (384, 128), (256, 256), (136, 1000), (1000, 136), (512, 2048)]
    hp = dict(HP, rank=rank)
    single, grouped = [], []
    for i, (rows, cols) in enumerate(shapes):
        st = _mat_state(rows, cols, rank, v_bits, 300 + 7 * i)
        single.append({k: _t(v) for k, v in st.items()})
        grouped.append({k: _t(v) for k, v in st.items()})
        single[-1]["prev"] = torch.zeros(1, dtype=torch.float32, device="cuda")
    grads = {}
    for t in range(1, 4):
        for i, (rows, cols) in enumerate(shapes):
            grads[(i, t)] = _t(wl.gaussian_grad((rows, cols), 1e-3, 9000 + 13 * i + t).ravel())
    plans = {}
    for t in range(1, 4):
        for i, (rows, cols) in enumerate(shapes):
            d = single[i]
            ws = torch.zeros(B.al_workspace_size(B.AL_OP_APOLLO, rows, cols, rank),
                             dtype=torch.uint8, device="cuda")
            B.al_apollo_step(d["p"], grads[(i, t)], rows, cols, d["proj"], d["m_codes"],
                             d["m_absmax"], rank, d["v_codes"], d["v_meta"], v_bits, rank,
                             d["prev"], hp, t, ws)
        # the plan binds the gradient buffers, so step t gets its own plan
        mats = [dict(grouped[i], g=grads[(i, t)], rows=rows, cols=cols)
                for i, (rows, cols) in enumerate(shapes)]
        plans[t] = B.ApolloPlan(mats, rank, v_bits)
        plans[t].step(hp, t)
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            for k in ("p", "m_codes", "m_absmax", "v_codes", "v_meta"):
                a = single[i][k].cpu().numpy().view(np.uint8)
                b = grouped[i][k].cpu().numpy().view(np.uint8)
                assert np.array_equal(a, b), (shapes[i], k, t)
    info = plans[3].info
    assert info.nmat == len(shapes)
    assert info.gemm_tiles == sum((max(r, c) + 127) // 128 for r, c in shapes)


@pytest.mark.parametrize("rank", [128, 256])
def test_apollo_grouped_limiter_matches_single(B, rank):
    """The norm-growth limiter in the grouped step (per-matrix chunk
    partials of ||G s||^2, one limiter thread per matrix) gives every matrix
    bit for bit the single-matrix step's parameters, states and previous
    norm over four steps; the previous norms follow the oracle's within
    1e-5. The scaled update G s does not grow with the gradient's scale
    (s_j normalises each channel), so the cap is engaged by channels that
    wake up: every other channel has a zero gradient at steps 1 and 2 (s_j =
    0) and all are active from step 3, when ||G s|| grows by about sqrt(2)."""
    import torch
    shapes = [(64, 256), (384, 128), (136, 1000), (1000, 136), (512, 2048)]
    hp = dict(HP, rank=rank, norm_growth_gamma=1.01)
    single, grouped, host = [], [], []
    for i, (rows, cols) in enumerate(shapes):
        st = _mat_state(rows, cols, rank, 8, 500 + 11 * i)
        host.append(dict({k: v.copy() for k, v in st.items()}, prev=np.float32(0.0)))
        single.append({k: _t(v) for k, v in st.items()})
        grouped.append({k: _t(v) for k, v in st.items()})
        single[-1]["prev"] = torch.zeros(1, dtype=torch.float32, device="cuda")
        grouped[-1]["prev_norm"] = torch.zeros(1, dtype=torch.float32, device="cuda")
    grads = [torch.zeros(r * c, dtype=torch.float32, device="cuda") for r, c in shapes]
    plan = B.ApolloPlan([dict(grouped[i], g=grads[i], rows=r, cols=c)
                         for i, (r, c) in enumerate(shapes)], rank, 8)
    assert plan.info.limiter_ok == 1
    capped = 0
    for t in range(1, 5):
        for i, (rows, cols) in enumerate(shapes):
            g = wl.gaussian_grad((rows, cols), 1e-3, 9500 + 13 * i + t)
            if t < 3:  # every other channel dormant
                if rows <= cols:
                    g[:, ::2] = 0.0
                else:
                    g[::2, :] = 0.0
            g = g.ravel()
            grads[i].copy_(torch.from_numpy(g))
            d = single[i]
            ws = torch.zeros(B.al_workspace_size(B.AL_OP_APOLLO, rows, cols, rank),
                             dtype=torch.uint8, device="cuda")
            B.al_apollo_step(d["p"], grads[i], rows, cols, d["proj"], d["m_codes"],
                             d["m_absmax"], rank, d["v_codes"], d["v_meta"], 8, rank, d["prev"],
                             hp, t, ws)
            h = host[i]
            before = h["prev"]
            _, h["prev"] = ora.apollo_step(h["p"], g, rows, cols, h["proj"], h["m_codes"],
                                           h["m_absmax"], rank, h["v_codes"], h["v_meta"], 8,
                                           rank, h["prev"], hp, t)
            if t == 3:  # the woken channels: the norm is capped at 1.01 x the last
                capped += int(abs(float(h["prev"]) - 1.01 * float(before))
                              <= 1e-6 * float(h["prev"]))
        plan.step(hp, t)
        torch.cuda.synchronize()
        for i in range(len(shapes)):
            for k in ("p", "m_codes", "m_absmax", "v_codes", "v_meta"):
                a = single[i][k].cpu().numpy().view(np.uint8)
                b = grouped[i][k].cpu().numpy().view(np.uint8)
                assert np.array_equal(a, b), (shapes[i], k, t)
            assert single[i]["prev"].item() == grouped[i]["prev_norm"].item(), (shapes[i], t)
            assert abs(grouped[i]["prev_norm"].item() - float(host[i]["prev"])) <= \
                1e-5 * float(host[i]["prev"]), (shapes[i], t)
    assert capped == len(shapes)  # the spike at t = 3 engaged every matrix's cap


def test_apollo_grouped_rejects_limiter_without_state_and_bad_arguments(B):
    import torch
    st = {k: _t(v) for k, v in _mat_state(64, 256, 128, 8, 5).items()}
    g = torch.zeros(64 * 256, dtype=torch.float32, device="cuda")
    plan = B.ApolloPlan([dict(st, g=g, rows=64, cols=256)], 128, 8)
    assert plan.info.limiter_ok == 0
    with pytest.raises(B.AlqError, match="INVALID_ARG"):  # no prev_norm for the limiter
        plan.step(dict(HP, rank=128, norm_growth_gamma=1.01), 1)
    with pytest.raises(B.AlqError):
        plan.step(dict(HP, rank=256), 1)  # rank differs from the plan's
    with pytest.raises(B.AlqError):
        B.ApolloPlan([dict(st, g=g, rows=64, cols=254)], 128, 8)  # cols % 4 != 0
